"""GPU parity: the CUDA path through the C ABI against the CPU oracle.

Decode attention must satisfy |gpu - oracle| <= 1e-2 * max(1, |oracle|)
elementwise; migrated bytes and block tables must be bit-exact; a session's
decode output must be bit-identical before and after a pause/resume round
trip, across batch compositions and across physical placements.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

TOL = 1e-2


@pytest.fixture(scope="module")
def pkg(cuda_dev):
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_25782_gb300 as P
    return P


def scaled_err(got, ref):
    return np.max(np.abs(got - ref) / np.maximum(1.0, np.abs(ref))) if ref.size else 0.0


def direct_case(P, lens, L=2, Hq=32, Hkv=4, bt=16, seed=0, spare=7, k_scale=1.0, max_batch=None):
    """Pool whose hot blocks are filled directly by the input generator at a
    seeded random placement (decode tested on its own)."""
    dev = torch.device("cuda:0")
    nb = int(sum(-(-t // bt) for t in lens)) + spare
    max_ctx = max(max(lens), bt)
    pool = P.Pool(num_layers=L, num_hot_blocks=nb, cold_bytes=256, num_q_heads=Hq,
                  num_kv_heads=Hkv, block_tokens=bt, max_sessions=4,
                  max_batch=max_batch or L * len(lens), max_context=max_ctx)
    tables = synth.random_block_tables(seed, lens, bt, nb)
    sess = list(range(len(lens)))
    synth.fill_hot_pool_torch(pool.hot, seed, sess, lens, tables, L, Hkv, 128, bt, k_scale)
    q = synth.queries_torch(seed, sess, range(L), Hq, 128, dev)
    return pool, sess, tables, q


def gpu_decode(pool, layer, q, tables, lens):
    dev = torch.device("cuda:0")
    t = torch.as_tensor(tables, device=dev)
    s = torch.as_tensor(np.asarray(lens, dtype=np.int32), device=dev)
    B = len(lens)
    shape = (pool.L if layer < 0 else 1, B, pool.Hq, 128)
    out = torch.full(shape, float("nan"), dtype=torch.float32, device=dev)
    qq = q if layer < 0 else q[layer:layer + 1]
    pool.decode_attention(layer, qq.contiguous(), t, s, B, t.shape[1],
                          getattr(pool, "_scale", 1 / math.sqrt(128)), out)
    torch.cuda.synchronize()
    return out.cpu().double().numpy()


def host_hot(pool, seed, sess, lens, tables, k_scale=1.0):
    return synth.hot_pool_np(seed, sess, lens, tables, pool.num_hot_blocks, pool.L, pool.Hkv,
                             128, pool.bt, k_scale)


LENGTHS = [1, 2, 15, 16, 17, 31, 33, 63, 64, 65, 127, 128, 129, 255, 511, 512, 513, 1000,
           1023, 1024, 1025, 1793, 2047, 2048, 2049, 4096, 4097, 6143, 8191, 8193, 17000]


def test_decode_many_lengths_all_and_per_layer(pkg):
    lens = LENGTHS
    pool, sess, tables, q = direct_case(pkg, lens, L=2, seed=1)
    ref = oracle.paged_decode(host_hot(pool, 1, sess, lens, tables), q.cpu().view(torch.int16)
                              .numpy().view(np.uint16), tables, lens, 1 / math.sqrt(128), 32)
    got_all = gpu_decode(pool, -1, q, tables, lens)
    assert scaled_err(got_all, ref) <= TOL
    for l in range(2):
        got = gpu_decode(pool, l, q, tables, lens)
        assert np.array_equal(got[0], got_all[l])   # one launch per layer == all layers
    assert pool.check_device() == 0


@pytest.mark.parametrize("Hq,Hkv", [(32, 4), (16, 4), (8, 4), (4, 4), (8, 8), (8, 1)])
def test_decode_group_sizes(pkg, Hq, Hkv):
    lens = [5, 77, 300, 1500]
    pool, sess, tables, q = direct_case(pkg, lens, L=1, Hq=Hq, Hkv=Hkv, seed=2)
    hot = synth.hot_pool_np(2, sess, lens, tables, pool.num_hot_blocks, 1, Hkv, 128, 16)
    ref = oracle.paged_decode(hot, q.cpu().view(torch.int16).numpy().view(np.uint16), tables,
                              lens, 1 / math.sqrt(128), Hq)
    assert scaled_err(gpu_decode(pool, -1, q, tables, lens), ref) <= TOL


def test_decode_block_64(pkg):
    lens = [1, 63, 64, 65, 700, 3001]
    pool, sess, tables, q = direct_case(pkg, lens, L=2, bt=64, seed=3)
    ref = oracle.paged_decode(host_hot(pool, 3, sess, lens, tables),
                              q.cpu().view(torch.int16).numpy().view(np.uint16), tables, lens,
                              1 / math.sqrt(128), 32)
    assert scaled_err(gpu_decode(pool, -1, q, tables, lens), ref) <= TOL


@pytest.mark.parametrize("k_scale,scale", [(1 / math.sqrt(128), 1.0), (1.0, 1 / math.sqrt(128)),
                                           (1.0, 0.5)])
def test_decode_scale_readings(pkg, k_scale, scale):
    lens = [700, 1234]
    pool, sess, tables, q = direct_case(pkg, lens, L=1, seed=4, k_scale=k_scale)
    pool._scale = scale
    hot = host_hot(pool, 4, sess, lens, tables, k_scale)
    ref = oracle.paged_decode(hot, q.cpu().view(torch.int16).numpy().view(np.uint16), tables,
                              lens, scale, 32)
    assert scaled_err(gpu_decode(pool, -1, q, tables, lens), ref) <= TOL


def test_decode_independent_of_batch_and_placement(pkg):
    lens = [900, 33, 4100]
    pool, sess, tables, q = direct_case(pkg, lens, L=1, seed=5, spare=300)
    full = gpu_decode(pool, 0, q, tables, lens)
    # alone, and in another batch order
    alone = gpu_decode(pool, 0, q[:, 2:3], tables[2:3], lens[2:3])
    assert np.array_equal(alone[0, 0], full[0, 2])
    order = [2, 0, 1]
    perm = gpu_decode(pool, 0, q[:, order], tables[order], [lens[i] for i in order])
    for i, o in enumerate(order):
        assert np.array_equal(perm[0, i], full[0, o])
    # move every block of session 0 to fresh physical blocks
    hv = pool.hot_view()
    used = set(tables[tables >= 0].tolist())
    free = [b for b in range(pool.num_hot_blocks) if b not in used]
    n0 = -(-lens[0] // 16)
    t2 = tables.copy()
    t2[0, :n0] = free[:n0]
    src = torch.as_tensor(tables[0, :n0].astype(np.int64), device=hv.device)
    dst = torch.as_tensor(np.asarray(free[:n0], dtype=np.int64), device=hv.device)
    hv[dst] = hv[src]
    moved = gpu_decode(pool, 0, q, t2, lens)
    assert np.array_equal(moved, full)


def test_ring_depths_bit_identical(pkg):
    """The split kernel's launch variant follows the size of the grid: one
    CTA per SM with 8 warps (one of a split's eight accumulators each), or 2
    or 3 CTAs per SM with 4 warps (two accumulators each) and 3- or 2-deep
    tile rings. The variants change where the accumulators run and how far
    ahead tiles are fetched, never which tiles an accumulator takes or the
    merge order, so all must give the same bits."""
    lens = [5000, 3001, 777]
    L = 16
    pool, sess, tables, q = direct_case(pkg, lens, L=L, seed=4, max_batch=L * len(lens))
    mid = np.pad(tables, ((0, 0), (0, 600 - tables.shape[1])), constant_values=-1)
    wide = np.pad(tables, ((0, 0), (0, 2048 - tables.shape[1])), constant_values=-1)
    # per layer, 313-block tables: 5 splits x 4 kv-heads x 3 rows = 60 CTAs (8 warps);
    # per layer, 600-block tables: 10 x 4 x 3 = 120 CTAs (8 warps);
    # per layer, tables 2048 blocks wide: 16 x 4 x 3 = 192 CTAs (4 warps, 3-deep);
    # all 16 layers in one call: 5 x 4 x 48 = 960 CTAs (4 warps, 2-deep)
    narrow = np.concatenate([gpu_decode(pool, l, q, tables, lens) for l in range(L)])
    middle = np.concatenate([gpu_decode(pool, l, q, mid, lens) for l in range(L)])
    padded = np.concatenate([gpu_decode(pool, l, q, wide, lens) for l in range(L)])
    whole = gpu_decode(pool, -1, q, tables, lens)
    assert np.array_equal(narrow.view(np.int64), middle.view(np.int64))
    assert np.array_equal(narrow.view(np.int64), padded.view(np.int64))
    assert np.array_equal(narrow.view(np.int64), whole.view(np.int64))
    ref = oracle.paged_decode(host_hot(pool, 4, sess, lens, tables), q.cpu().view(torch.int16)
                              .numpy().view(np.uint16), tables, lens, 1 / math.sqrt(128), 32)
    assert scaled_err(narrow, ref) <= TOL
    assert pool.check_device() == 0


def test_merge_paths_bit_identical(pkg):
    """A session of several splits is merged by the split kernel (the last
    CTA of each of its kv-heads to finish; sessions of up to 4 splits in a
    grid of at least 8 CTAs per SM) or by a combine kernel (one warp per
    query head from registers for tables of up to 16 splits, else four warps
    per head). All fold the same four chains of splits in the same order, so
    a session's output is the same bits whichever merges it. The all-layer
    calls reuse batch rows for sessions of other split counts, which also
    checks that every call leaves its split-arrival counters at zero."""
    lens = [1500, 4000, 4500, 8000, 12800, 16000, 3001]   # 2, 4, 5, 8, 13, 16, 3 splits
    L = 4
    pool, sess, tables, q = direct_case(pkg, lens, L=L, seed=31, max_batch=L * len(lens))
    n = len(lens)
    # per layer, all sessions: 16 x 4 x 7 = 448 CTAs: every session merges in the
    # register combine (tables of 1 000 blocks, 16 splits at most)
    batch = np.concatenate([gpu_decode(pool, l, q, tables, lens) for l in range(L)])
    # one session per call, in tables 2 048 blocks wide (32K tokens: 16 splits) and
    # 2 112 blocks wide (17 splits: the four-warp combine)
    alone = np.zeros_like(batch)
    wide = np.pad(tables, ((0, 0), (0, 2112 - tables.shape[1])), constant_values=-1)
    alone_wide = np.zeros_like(batch)
    for i in range(n):
        qi = q[:, i:i + 1].contiguous()
        for l in range(L):
            alone[l, i] = gpu_decode(pool, l, qi, tables[i:i + 1], lens[i:i + 1])[0, 0]
            alone_wide[l, i] = gpu_decode(pool, l, qi, wide[i:i + 1], lens[i:i + 1])[0, 0]
    # rows reversed, so each row holds a session of another split count than before
    rev = list(reversed(range(n)))
    qr = q[:, rev].contiguous()
    back = np.concatenate([gpu_decode(pool, l, qr, tables[rev], [lens[i] for i in rev])
                           for l in range(L)])[:, rev]
    # all layers in one call: 16 x 4 x 28 = 1 792 CTAs, at least 8 per SM: the split
    # kernel merges the sessions of up to 4 splits (1 500, 3 001 and 4 000 tokens),
    # first with these rows, then with the rows reversed
    whole = gpu_decode(pool, -1, q, tables, lens)
    whole_back = gpu_decode(pool, -1, qr, tables[rev], [lens[i] for i in rev])[:, rev]
    for other in (alone, alone_wide, back, whole, whole_back):
        assert np.array_equal(batch.view(np.int64), other.view(np.int64))
    ref = oracle.paged_decode(host_hot(pool, 31, sess, lens, tables), q.cpu().view(torch.int16)
                              .numpy().view(np.uint16), tables, lens, 1 / math.sqrt(128), 32)
    assert scaled_err(batch, ref) <= TOL
    assert pool.check_device() == 0


def test_overlapped_calls_bit_identical(pkg):
    """Per-layer calls launched with KV_DECODE_OVERLAP_PREVIOUS (each one
    overlapping the previous call's end) give the same bits as serialised
    calls, over several rounds on one stream."""
    lens = [77, 1500, 4100, 9000, 33]
    L = 6
    pool, sess, tables, q = direct_case(pkg, lens, L=L, seed=12)
    dev = torch.device("cuda:0")
    t = torch.as_tensor(tables, device=dev)
    s = torch.as_tensor(np.asarray(lens, dtype=np.int32), device=dev)
    st = torch.cuda.Stream()
    torch.cuda.synchronize()     # inputs were made on the default stream
    outs = []
    for overlap in (False, True, True):
        out = torch.full((L, len(lens), 32, 128), float("nan"), dtype=torch.float32, device=dev)
        for rnd in range(2):
            for l in range(L):
                pool.decode_attention(l, q[l].contiguous(), t, s, len(lens), t.shape[1],
                                      1 / math.sqrt(128), out[l], st,
                                      overlap_previous=overlap and (l > 0 or rnd > 0))
        torch.cuda.synchronize()
        outs.append(out.clone())
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])
    ref = oracle.paged_decode(host_hot(pool, 12, sess, lens, tables),
                              q.cpu().view(torch.int16).numpy().view(np.uint16), tables, lens,
                              1 / math.sqrt(128), 32)
    assert scaled_err(outs[1].double().cpu().numpy(), ref) <= TOL
    assert pool.check_device() == 0


def test_bf16_output_is_rounded_fp32(pkg):
    """KV_DECODE_OUT_BF16: each output is the fp32 result rounded to nearest
    even, both from one-split sessions (split kernel) and merged ones."""
    lens = [5, 700, 2047, 5000, 13000]
    pool, sess, tables, q = direct_case(pkg, lens, L=2, seed=14)
    dev = torch.device("cuda:0")
    t = torch.as_tensor(tables, device=dev)
    s = torch.as_tensor(np.asarray(lens, dtype=np.int32), device=dev)
    o32 = torch.empty(2, len(lens), 32, 128, dtype=torch.float32, device=dev)
    o16 = torch.empty(2, len(lens), 32, 128, dtype=torch.bfloat16, device=dev)
    pool.decode_attention(-1, q, t, s, len(lens), t.shape[1], 1 / math.sqrt(128), o32)
    pool.decode_attention(-1, q, t, s, len(lens), t.shape[1], 1 / math.sqrt(128), o16)
    torch.cuda.synchronize()
    assert torch.equal(o16.view(torch.int16), o32.to(torch.bfloat16).view(torch.int16))
    ref = oracle.paged_decode(host_hot(pool, 14, sess, lens, tables),
                              q.cpu().view(torch.int16).numpy().view(np.uint16), tables, lens,
                              1 / math.sqrt(128), 32)
    assert scaled_err(o16.double().cpu().numpy(), ref) <= TOL
    assert pool.check_device() == 0


def test_nan_tail_slots_do_not_leak(pkg):
    lens = [17, 100, 529]
    pool, sess, tables, q = direct_case(pkg, lens, L=1, seed=6)
    hv = pool.hot_view()
    for b, T in enumerate(lens):         # poison every slot past T, K and V
        j = (T - 1) // 16
        hv[int(tables[b, j]), :, :, :, T % 16 or 16:, :] = float("nan")
    got = gpu_decode(pool, 0, q, tables, lens)
    assert np.all(np.isfinite(got))
    ref = oracle.paged_decode(host_hot(pool, 6, sess, lens, tables),
                              q.cpu().view(torch.int16).numpy().view(np.uint16), tables, lens,
                              1 / math.sqrt(128), 32)
    assert scaled_err(got, ref) <= TOL


def test_device_check_flags(pkg):
    lens = [40]
    pool, sess, tables, q = direct_case(pkg, lens, L=1, seed=7)
    bad = tables.copy()
    bad[0, 1] = pool.num_hot_blocks + 3          # outside the pool: flagged, not read
    gpu_decode(pool, 0, q, bad, lens)
    assert pool.check_device() & 1
    gpu_decode(pool, 0, q, tables, [tables.shape[1] * 16 + 1])   # longer than its table row
    assert pool.check_device() & 2
    gpu_decode(pool, 0, q, tables, lens)
    assert pool.check_device() == 0


# ------------------------------------------------------------ migration

def np_bits(t):
    return t.contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def test_resume_pack_append_bit_exact(pkg):
    """resume-unpack, append and pause-pack against the oracle's copies, and
    the block tables against the oracle's free-list contract."""
    dev = torch.device("cuda:0")
    L, Hkv, bt, seed, NB = 3, 4, 16, 9, 120
    pool = pkg.Pool(num_layers=L, num_hot_blocks=NB, cold_bytes=1 << 26, max_sessions=4,
                    max_batch=8, max_context=1024, alloc_seed=21)
    ref_fl = oracle.FreeList(NB, 21)
    hot_ref = np.zeros((NB, L, 2, Hkv, bt, 128), dtype=np.uint16)
    T0, cap = 301, 700
    s = pool.session_create_paused(cap, T0)
    synth.fill_image_torch(pool.image(s), seed, s, L, Hkv, 128, T0)
    img_ref = np_bits(pool.image(s))
    pool.session_resume(s)
    row = ref_fl.pop(-(-T0 // bt))
    assert pool.session_block_table(s) == list(row)
    oracle.unpack(img_ref, T0, row, hot_ref)
    torch.cuda.synchronize()
    hot = np_bits(pool.hot_view())
    for j, p in enumerate(row):
        n = min(bt, T0 - j * bt)
        assert np.array_equal(hot[p, :, :, :, :n], hot_ref[p, :, :, :, :n])

    # append 3 chunks crossing block boundaries
    T = T0
    for n in (3, 40, 1):
        k, v = synth.kv_logical_torch(seed + 1, s, range(L), Hkv, 128, T, T + n, dev)
        kk, vv = k.permute(0, 2, 1, 3).contiguous(), v.permute(0, 2, 1, 3).contiguous()
        pool.session_append(s, kk, vv)
        need = -(-(T + n) // bt) - len(row)
        if need > 0:
            row = np.concatenate([row, ref_fl.pop(need)])
        oracle.append(hot_ref, row, T, np_bits(kk), np_bits(vv))
        T += n
    assert pool.session_block_table(s) == list(row)
    torch.cuda.synchronize()
    hot = np_bits(pool.hot_view())
    for j, p in enumerate(row):
        n = min(bt, T - j * bt)
        assert np.array_equal(hot[p, :, :, :, :n], hot_ref[p, :, :, :, :n])

    # pause packs only [T0, T): the image's first T0 tokens are not rewritten
    before = pool.stats()["bytes_packed"]
    img_dev = pool.image(s)
    img_dev[:, :, :, :T0] = 0        # if pack touched these rows they would change
    pool.session_pause(s)
    ref_fl.push(row)
    exp = np.zeros_like(img_ref)
    written = oracle.pack(hot_ref, row, T0, T, exp)
    torch.cuda.synchronize()
    img = np_bits(pool.image(s))
    assert np.array_equal(img[:, :, :, T0:T], exp[:, :, :, T0:T])
    assert not np.any(img[:, :, :, :T0])
    assert pool.stats()["bytes_packed"] - before == written
    assert pool.free_list() == list(ref_fl.contents())
    assert pool.check_device() == 0


@pytest.mark.parametrize("T", [1, 16, 17, 1000])
def test_round_trip_byte_identical(pkg, T):
    """append -> pause (pack) -> resume (unpack into other blocks): the image
    equals the appended tokens and the new blocks equal the image."""
    dev = torch.device("cuda:0")
    L, bt, NB, Hkv = 2, 16, 200, 4
    pool = pkg.Pool(num_layers=L, num_hot_blocks=NB, cold_bytes=1 << 26, max_sessions=2,
                    max_batch=4, max_context=2048, alloc_seed=T)
    s = pool.session_create(1031)
    k, v = synth.kv_logical_torch(13, s, range(L), Hkv, 128, 0, T, dev)
    pool.session_append(s, k.permute(0, 2, 1, 3).contiguous(), v.permute(0, 2, 1, 3).contiguous())
    old = pool.session_block_table(s)
    pool.session_pause(s)
    img = pool.image(s)
    torch.cuda.synchronize()
    assert torch.equal(img[:, 0, :, :T].view(torch.int16), k.view(torch.int16))
    assert torch.equal(img[:, 1, :, :T].view(torch.int16), v.view(torch.int16))
    pool.shuffle_free(T + 1)
    pool.session_resume(s)
    row = pool.session_block_table(s)
    assert len(row) == len(old)
    hv = pool.hot_view()
    blocks = hv[torch.as_tensor(row, device=dev, dtype=torch.int64)]
    as_img = blocks.permute(1, 2, 3, 0, 4, 5).reshape(L, 2, Hkv, -1, 128)[:, :, :, :T]
    torch.cuda.synchronize()
    assert torch.equal(as_img.view(torch.int16), img[:, :, :, :T].view(torch.int16))
    assert pool.check_device() == 0


@pytest.mark.parametrize("bt,T1,T2", [(16, 37, 87), (64, 37, 87), (64, 64, 65), (64, 1, 300),
                                       (64, 130, 1000)])
def test_incremental_pack_resume_bit_exact(pkg, bt, T1, T2):
    """Two pause/resume cycles: the second pack starts at the image's
    watermark T1 (mid-block and mid-chunk for most cases), every resume
    scatters into reshuffled blocks; images and blocks stay bit-exact."""
    dev = torch.device("cuda:0")
    L, NB, Hkv, D = 2, 80, 4, 128
    pool = pkg.Pool(num_layers=L, num_hot_blocks=NB, cold_bytes=1 << 26, max_sessions=2,
                    max_batch=4, max_context=2048, alloc_seed=T2, block_tokens=bt)
    s = pool.session_create(1024)
    k, v = synth.kv_logical_torch(21, s, range(L), Hkv, D, 0, T2, dev)
    kk, vv = k.permute(0, 2, 1, 3).contiguous(), v.permute(0, 2, 1, 3).contiguous()
    pool.session_append(s, kk[:, :T1].contiguous(), vv[:, :T1].contiguous())
    for cycle, T in enumerate((T1, T2)):
        if cycle == 1:
            pool.session_append(s, kk[:, T1:].contiguous(), vv[:, T1:].contiguous())
        pool.session_pause(s)
        torch.cuda.synchronize()
        img = pool.image(s)
        assert torch.equal(img[:, 0, :, :T].view(torch.int16), k[:, :, :T].view(torch.int16))
        assert torch.equal(img[:, 1, :, :T].view(torch.int16), v[:, :, :T].view(torch.int16))
        assert int(pool.session_info(s).cold_valid) == T
        pool.shuffle_free(7 * T + cycle)
        pool.session_resume(s)
        row = pool.session_block_table(s)
        assert len(row) == -(-T // bt)
        blocks = pool.hot_view()[torch.as_tensor(row, device=dev, dtype=torch.int64)]
        as_img = blocks.permute(1, 2, 3, 0, 4, 5).reshape(L, 2, Hkv, -1, D)[:, :, :, :T]
        torch.cuda.synchronize()
        assert torch.equal(as_img.view(torch.int16), img[:, :, :, :T].view(torch.int16))
    assert pool.stats()["bytes_packed"] == T2 * pool.token_bytes     # each token written once
    assert pool.check_device() == 0
    pool.close()


def test_empty_session_pause_resume(pkg):
    """A session with no tokens pauses and resumes (nothing to move; the only
    way to have an empty paused session), then takes tokens and decodes like
    any other."""
    dev = torch.device("cuda:0")
    L = 2
    pool = pkg.Pool(num_layers=L, num_hot_blocks=16, cold_bytes=1 << 24, max_sessions=3,
                    max_batch=4, max_context=256)
    a = pool.session_create(256)
    b = pool.session_create(256)
    for s in (a, b):
        pool.session_pause(s)
        pool.session_resume(s)
    for s in (a, b):
        assert pool.session_block_table(s) == [] and int(pool.session_info(s).tokens) == 0
        k, v = synth.kv_logical_torch(5, s, range(L), 4, 128, 0, 20, dev)
        pool.session_append(s, k.permute(0, 2, 1, 3).contiguous(), v.permute(0, 2, 1, 3).contiguous())
    tables = torch.empty(2, 16, dtype=torch.int32, device=dev)
    lens = torch.empty(2, dtype=torch.int32, device=dev)
    pool.batch_tables([a, b], tables, 16, lens)
    q = synth.queries_torch(5, [a, b], range(L), 32, 128, dev)
    out = torch.empty(L, 2, 32, 128, dtype=torch.float32, device=dev)
    pool.decode_attention(-1, q, tables, lens, 2, 16, 1 / math.sqrt(128), out)
    torch.cuda.synchronize()
    rows = np.full((2, 16), -1, dtype=np.int32)
    for r, s in enumerate((a, b)):
        row = pool.session_block_table(s)
        rows[r, :len(row)] = row
    hot = synth.hot_pool_np(5, [a, b], [20, 20], rows, 16, L, 4, 128, 16)
    ref = oracle.paged_decode(hot, q.cpu().view(torch.int16).numpy().view(np.uint16), rows,
                              [20, 20], 1 / math.sqrt(128), 32)
    assert scaled_err(out.cpu().double().numpy(), ref) <= TOL
    assert pool.check_device() == 0
    pool.close()


def test_config1_scenario(pkg):
    """Tiny single-layer case: 4 sessions (512..2048 tokens, one partial tail)
    decode; a 5th 1024-token session is packed, its blocks freed, the free
    list scrambled, and it is resumed into 64 other blocks; the step re-run
    gives bit-identical outputs for all 5 sessions."""
    dev = torch.device("cuda:0")
    L, Hq, Hkv, bt, seed = 1, 32, 4, 16, 0
    lens = [int(x) for x in synth.session_lengths(seed, 4, 512, 2048, bt)] + [1024]
    NB = sum(-(-t // bt) for t in lens) + 64 + 32
    pool = pkg.Pool(num_layers=L, num_hot_blocks=NB, cold_bytes=64 << 20, max_sessions=8,
                    max_batch=8, max_context=2048, alloc_seed=seed)
    k_scale = 1 / math.sqrt(128)
    sids = []
    for T in lens:
        s = pool.session_create(2048)
        k, v = synth.kv_logical_torch(seed, s, range(L), Hkv, 128, 0, T, dev, k_scale)
        pool.session_append(s, k.permute(0, 2, 1, 3).contiguous(), v.permute(0, 2, 1, 3).contiguous())
        sids.append(s)
    q = synth.queries_torch(seed, sids, range(L), Hq, 128, dev)
    mb = 128
    tables = torch.empty(len(sids), mb, dtype=torch.int32, device=dev)
    slens = torch.empty(len(sids), dtype=torch.int32, device=dev)

    def step():
        pool.batch_tables(sids, tables, mb, slens)
        out = torch.empty(L, len(sids), Hq, 128, dtype=torch.float32, device=dev)
        pool.decode_attention(-1, q, tables, slens, len(sids), mb, 1.0, out)
        torch.cuda.synchronize()
        return out.clone()

    out1 = step()
    rows = [pool.session_block_table(s) for s in sids]
    tab_h = np.full((len(sids), mb), -1, dtype=np.int32)
    for i, r in enumerate(rows):
        tab_h[i, :len(r)] = r
    hot_h = synth.hot_pool_np(seed, sids, lens, tab_h, NB, L, Hkv, 128, bt, k_scale)
    ref = oracle.paged_decode(hot_h, np_bits(q), tab_h, lens, 1.0, Hq)
    assert scaled_err(out1.cpu().double().numpy(), ref) <= TOL

    s5 = sids[4]
    pool.session_pause(s5)
    pool.shuffle_free(12345)
    pool.session_resume(s5)
    new_row = pool.session_block_table(s5)
    assert len(new_row) == 64 and new_row != rows[4]
    out2 = step()
    assert torch.equal(out1, out2)
    assert pool.check_device() == 0


@pytest.mark.parametrize("mig_ctas", [1, 8, 152])
def test_migration_cta_cap_bit_exact(pkg, mig_ctas):
    """kv_pool_set_migration_limit caps the migration grids (the copies then
    walk their items grid-stride with fewer warps): resume-unpack through the
    one-launch path and the table-reading path (more than 2 048 blocks),
    append and pause-pack stay bit-exact against the oracle's copies."""
    dev = torch.device("cuda:0")
    L, Hkv, bt, seed = 2, 4, 16, 19
    lens = [700, 33000]
    NB = sum(-(-t // bt) for t in lens) + 300
    pool = pkg.Pool(num_layers=L, num_hot_blocks=NB, cold_bytes=(sum(lens) + 2000) * L * 2 * Hkv * 256
                    + 4096, max_sessions=4, max_batch=8, max_context=34000, alloc_seed=mig_ctas)
    pool_h = pool.handle
    pkg.kvtier.kv_pool_set_migration_limit(pool_h, mig_ctas)
    ref_fl = oracle.FreeList(NB, mig_ctas)
    hot_ref = np.zeros((NB, L, 2, Hkv, bt, 128), dtype=np.uint16)
    sids, rows, imgs = [], [], []
    for T in lens:
        s = pool.session_create_paused(T + 100, T)
        synth.fill_image_torch(pool.image(s), seed, s, L, Hkv, 128, T)
        sids.append(s)
    torch.cuda.synchronize()
    for s, T in zip(sids, lens):
        imgs.append(np_bits(pool.image(s)))
        pool.session_resume(s)
        row = ref_fl.pop(-(-T // bt))
        assert pool.session_block_table(s) == list(row)
        oracle.unpack(imgs[-1], T, row, hot_ref)
        rows.append(row)
    torch.cuda.synchronize()
    hot = np_bits(pool.hot_view())
    for row, T in zip(rows, lens):
        for j, p in enumerate(row):
            n = min(bt, T - j * bt)
            assert np.array_equal(hot[p, :, :, :, :n], hot_ref[p, :, :, :, :n])
    # 50 more tokens each, then the pause packs exactly them
    for i, (s, T) in enumerate(zip(sids, lens)):
        k, v = synth.kv_logical_torch(seed + 1, s, range(L), Hkv, 128, T, T + 50, dev)
        kk, vv = k.permute(0, 2, 1, 3).contiguous(), v.permute(0, 2, 1, 3).contiguous()
        pool.session_append(s, kk, vv)
        need = -(-(T + 50) // bt) - len(rows[i])
        if need > 0:
            rows[i] = np.concatenate([rows[i], ref_fl.pop(need)])
        oracle.append(hot_ref, rows[i], T, np_bits(kk), np_bits(vv))
        pool.session_pause(s)
        ref_fl.push(rows[i])
        exp = imgs[i].copy()
        oracle.pack(hot_ref, rows[i], T, T + 50, exp)
        torch.cuda.synchronize()
        assert np.array_equal(np_bits(pool.image(s))[:, :, :, :T + 50], exp[:, :, :, :T + 50])
    assert pool.free_list() == list(ref_fl.contents())
    assert pool.check_device() == 0
    pool.close()


@pytest.mark.parametrize("case", ["scale50", "planted64", "planted1024"])
def test_decode_extreme_logits(pkg, case):
    """The online softmax's edge cases: scale 50 spreads the logits over
    hundreds (a near one-hot softmax); a planted key k = c * q (c = 64 or
    1 024) in a late split puts one token above all others by about 700 or
    11 600 for the first head of each group, so every other exponent
    underflows to zero and the merge across splits must still weigh the
    splits correctly. Outputs must be finite and within the tolerance of
    the fp64 oracle."""
    dev = torch.device("cuda:0")
    lens = [37, 1500, 5000, 17000]
    pool, sess, tables, q = direct_case(pkg, lens, L=1, seed=40)
    hot = host_hot(pool, 40, sess, lens, tables)
    scale = 50.0 if case == "scale50" else 1 / math.sqrt(128)
    if case.startswith("planted"):
        c = 64.0 if case == "planted64" else 1024.0
        hv = pool.hot_view()
        qc = q.cpu()
        for b, T in enumerate(lens):
            t = (3 * T) // 4                      # past the first split when there are several
            blk, r = int(tables[b, t // 16]), t % 16
            for g in range(4):
                kk = (qc[0, b, g * 8].float() * c).to(torch.bfloat16)   # exact: c is 2^k
                hot[blk, 0, 0, g, r] = kk.view(torch.int16).numpy().view(np.uint16)
                hv[blk, 0, 0, g, r] = kk.to(dev)
    pool._scale = scale
    ref = oracle.paged_decode(hot, q.cpu().view(torch.int16).numpy().view(np.uint16), tables,
                              lens, scale, 32)
    got = gpu_decode(pool, -1, q, tables, lens)
    assert np.all(np.isfinite(got))
    assert scaled_err(got, ref) <= TOL
    if case == "planted1024":   # head 0 of each group attends to its planted token alone
        for b, T in enumerate(lens):
            t = (3 * T) // 4
            blk, r = int(tables[b, t // 16]), t % 16
            v = hot[blk, 0, 1, :, r].astype(np.uint32) << 16
            v = v.view(np.float32)
            for g in range(4):
                assert np.allclose(got[0, b, g * 8], v[g], rtol=1e-5, atol=1e-6)
    assert pool.check_device() == 0


def test_device_table_row_matches_host_row(pkg):
    """session_block_table_device: the address of a session's row in the
    pool's device table arena, fixed for the pool's life; after appends and
    after a pause and a resume into other blocks it holds the same ids as
    the host copy (read here through the CUDA array interface)."""
    dev = torch.device("cuda:0")
    pool = pkg.Pool(num_layers=2, num_hot_blocks=64, cold_bytes=1 << 24, max_sessions=2,
                    max_batch=4, max_context=512, alloc_seed=5)
    s = pool.session_create(512)
    k, v = synth.kv_logical_torch(1, s, range(2), 4, 128, 0, 300, dev)
    pool.session_append(s, k.permute(0, 2, 1, 3).contiguous(), v.permute(0, 2, 1, 3).contiguous())
    addr, n = pool.session_block_table_device(s)
    assert n == len(pool.session_block_table(s)) == -(-300 // 16)

    class Row:
        __cuda_array_interface__ = {"shape": (n,), "typestr": "<i4", "data": (addr, False),
                                    "version": 2}

    row = torch.as_tensor(Row(), device=dev)
    torch.cuda.synchronize()
    assert row.cpu().tolist() == pool.session_block_table(s)
    old = pool.session_block_table(s)
    pool.session_pause(s)
    pool.shuffle_free(9)
    pool.session_resume(s)
    torch.cuda.synchronize()
    assert pool.session_block_table_device(s) == (addr, n)
    assert row.cpu().tolist() == pool.session_block_table(s) != old
    assert pool.check_device() == 0
    pool.close()

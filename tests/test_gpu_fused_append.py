"""The fused decode step (data paths 3 and 1 in one kernel) on the GPU.

kv_pool_batch_reserve gives each session of a batch its next position, and
decode_append_attention writes that token's K/V into the pool while it
attends over it. Against the unfused sequence (session_append of the token,
then decode_attention) outputs and pool contents must be bit-identical; the
outputs must also agree with the oracle over the grown sessions, and a
pause afterwards must pack the fused tokens into the images.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

TOL = 1e-2
HQ, HKV, D = 32, 4, 128
SEED = 3


@pytest.fixture(scope="module")
def pkg(cuda_dev):
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_25782_gb300 as P
    return P


def bits(t):
    return t.contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def token_rows(sids, pos, L, dev):
    """K and V [L][B][Hkv][D] of token pos[b] of session sids[b]."""
    ks, vs = [], []
    for sid, t in zip(sids, pos):
        k, v = synth.kv_logical_torch(SEED, sid, range(L), HKV, D, t, t + 1, dev)
        ks.append(k[:, :, 0])
        vs.append(v[:, :, 0])
    return torch.stack(ks, 1).contiguous(), torch.stack(vs, 1).contiguous()


def run(P, fused, lens0, steps, L=2, bt=16, mode="layer", overlap=False, nb=None):
    dev = torch.device("cuda:0")
    B = len(lens0)
    cap = max(lens0) + steps + 1
    nb = nb or sum(-(-(t + steps) // bt) for t in lens0) + 8
    tok_bytes = L * 2 * HKV * D * 2
    pool = P.Pool(num_layers=L, num_hot_blocks=nb, cold_bytes=B * (cap * tok_bytes + 256),
                  block_tokens=bt, max_sessions=B, max_batch=L * B, max_context=cap,
                  alloc_seed=5)
    sids = [pool.session_create(cap) for _ in lens0]
    for sid, t in zip(sids, lens0):
        if t:
            k, v = synth.kv_logical_torch(SEED, sid, range(L), HKV, D, 0, t, dev)
            pool.session_append(sid, k.permute(0, 2, 1, 3).contiguous(),
                                v.permute(0, 2, 1, 3).contiguous())
    q = synth.queries_torch(SEED, sids, range(L), HQ, D, dev)
    mb = -(-cap // bt)
    tables = torch.empty(B, mb, dtype=torch.int32, device=dev)
    slens = torch.empty(B, dtype=torch.int32, device=dev)
    scale = 1 / math.sqrt(D)
    T = list(lens0)
    outs = []
    for _ in range(steps):
        kn, vn = token_rows(sids, T, L, dev)
        out = torch.full((L, B, HQ, D), float("nan"), dtype=torch.float32, device=dev)
        if fused:
            pool.batch_reserve(sids, tables, mb, slens)
            if mode == "all":
                pool.decode_append_attention(-1, q, kn, vn, tables, slens, B, mb, scale, out)
            else:
                for l in range(L):
                    pool.decode_append_attention(l, q[l], kn[l], vn[l], tables, slens, B, mb,
                                                 scale, out[l], overlap_previous=overlap and l > 0)
        else:
            for b, sid in enumerate(sids):
                pool.session_append(sid, kn[:, b:b + 1].contiguous(), vn[:, b:b + 1].contiguous())
            pool.batch_tables(sids, tables, mb, slens)
            if mode == "all":
                pool.decode_attention(-1, q, tables, slens, B, mb, scale, out)
            else:
                for l in range(L):
                    pool.decode_attention(l, q[l], tables, slens, B, mb, scale, out[l],
                                          overlap_previous=overlap and l > 0)
        outs.append(out)
        T = [t + 1 for t in T]
    torch.cuda.synchronize()
    assert pool.check_device() == 0
    return pool, sids, T, [o.cpu() for o in outs], q


def check_pool_holds_sessions(pool, sids, T, L, bt):
    hv = pool.hot_view()
    for sid, t in zip(sids, T):
        k, v = synth.session_kv_np(SEED, sid, range(L), HKV, D, t)
        for j, blk in enumerate(pool.session_block_table(sid)):
            n = min(bt, t - j * bt)
            hb = bits(hv[blk])
            assert np.array_equal(hb[:, 0, :, :n], k[:, :, j * bt:j * bt + n]), (sid, j)
            assert np.array_equal(hb[:, 1, :, :n], v[:, :, j * bt:j * bt + n]), (sid, j)


def oracle_out(pool, sids, T, q, L, bt):
    mb = max(len(pool.session_block_table(s)) for s in sids)
    rows = np.full((len(sids), mb), -1, dtype=np.int32)
    for b, s in enumerate(sids):
        r = pool.session_block_table(s)
        rows[b, :len(r)] = r
    hot = synth.hot_pool_np(SEED, sids, T, rows, pool.num_hot_blocks, L, HKV, D, bt)
    return oracle.paged_decode(hot, bits(q), rows, T, 1 / math.sqrt(D), HQ)


LENS = [0, 1, 14, 15, 16, 17, 47, 63, 64, 100, 1023, 1024, 3000, 5000]


@pytest.mark.parametrize("bt,mode,overlap", [(16, "layer", False), (16, "layer", True),
                                             (16, "all", False), (64, "layer", True),
                                             (64, "all", False)])
def test_fused_step_equals_append_then_decode(pkg, bt, mode, overlap):
    L, steps = 2, 3
    pf, sids, T, of, q = run(pkg, True, LENS, steps, L=L, bt=bt, mode=mode, overlap=overlap)
    pu, _, _, ou, _ = run(pkg, False, LENS, steps, L=L, bt=bt, mode=mode, overlap=overlap)
    for a, b in zip(of, ou):
        assert torch.equal(a.view(torch.int32), b.view(torch.int32))   # bit-identical
    for s in sids:
        assert pf.session_block_table(s) == pu.session_block_table(s)
    assert pf.stats()["bytes_appended"] == pu.stats()["bytes_appended"]
    check_pool_holds_sessions(pf, sids, T, L, bt)
    ref = oracle_out(pf, sids, T, q, L, bt)
    got = of[-1].double().numpy()
    assert np.max(np.abs(got - ref) / np.maximum(1.0, np.abs(ref))) <= TOL
    # a pause packs the fused tokens: every image holds the session's KV
    for s, t in zip(sids, T):
        pf.session_pause(s)
    torch.cuda.synchronize()
    for s, t in zip(sids, T):
        k, v = synth.session_kv_np(SEED, s, range(L), HKV, D, t)
        img = bits(pf.image(s)[:, :, :, :t])
        assert np.array_equal(img[:, 0], k) and np.array_equal(img[:, 1], v)
    pf.close()
    pu.close()


def test_fused_steps_cross_blocks_and_splits(pkg):
    """Forty steps: every session crosses at least two block boundaries and
    the long ones change split count; the fused run stays bit-identical."""
    lens = [5, 30, 2040, 4090, 8180]
    pf, sids, T, of, q = run(pkg, True, lens, 40, L=1, mode="layer")
    pu, _, _, ou, _ = run(pkg, False, lens, 40, L=1, mode="layer")
    for a, b in zip(of, ou):
        assert torch.equal(a.view(torch.int32), b.view(torch.int32))
    check_pool_holds_sessions(pf, sids, T, 1, 16)
    ref = oracle_out(pf, sids, T, q, 1, 16)
    assert np.max(np.abs(of[-1].double().numpy() - ref) / np.maximum(1.0, np.abs(ref))) <= TOL
    pf.close()
    pu.close()


def test_fused_steps_one_cta_per_sm(pkg):
    """A batch small enough for one CTA per SM (3 splits x 4 kv-heads x 3
    sessions = 36 CTAs) runs the 8-warp kernel, one accumulator per warp,
    while larger grids run 4 warps with two accumulators each. Over twenty
    steps the token that arrives with the call lands in different warps and
    accumulators; the fused run stays bit-identical to append-then-decode
    and agrees with the oracle."""
    lens = [70, 1100, 2030]
    pf, sids, T, of, q = run(pkg, True, lens, 20, L=2, mode="layer")
    pu, _, _, ou, _ = run(pkg, False, lens, 20, L=2, mode="layer")
    for a, b in zip(of, ou):
        assert torch.equal(a.view(torch.int32), b.view(torch.int32))
    check_pool_holds_sessions(pf, sids, T, 2, 16)
    ref = oracle_out(pf, sids, T, q, 2, 16)
    assert np.max(np.abs(of[-1].double().numpy() - ref) / np.maximum(1.0, np.abs(ref))) <= TOL
    assert pf.check_device() == 0
    pf.close()
    pu.close()


def test_fused_argument_errors(pkg):
    dev = torch.device("cuda:0")
    pool = pkg.Pool(num_layers=1, num_hot_blocks=16, cold_bytes=1 << 20, max_sessions=2,
                    max_batch=2, max_context=64)
    sid = pool.session_create(64)
    tables = torch.empty(1, 4, dtype=torch.int32, device=dev)
    slens = torch.empty(1, dtype=torch.int32, device=dev)
    pool.batch_reserve([sid], tables, 4, slens)
    q = torch.zeros(1, HQ, D, dtype=torch.bfloat16, device=dev)
    kn = torch.zeros(1 * HKV * D + 8, dtype=torch.bfloat16, device=dev)
    out = torch.empty(1, HQ, D, dtype=torch.float32, device=dev)
    from paper_2609_25782_gb300 import kvtier
    with pytest.raises(kvtier.KVError) as e:    # misaligned k_new: refused before any launch
        pool.decode_append_attention(0, q, kn[1:], kn[:HKV * D], tables, slens, 1, 4, 1.0, out)
    assert e.value.code == kvtier.KV_ERR_INVALID_ARG
    with pytest.raises(kvtier.KVError) as e:
        kvtier.decode_append_attention(pool.handle, 0, q, None, kn, tables, slens, 1, 4, 1.0, out)
    assert e.value.code == kvtier.KV_ERR_INVALID_ARG
    with pytest.raises(kvtier.KVError) as e:
        pool.batch_reserve([sid, sid], tables, 4, slens)
    assert e.value.code == kvtier.KV_ERR_INVALID_ARG
    pool.decode_append_attention(0, q, kn[:HKV * D], kn[:HKV * D], tables, slens, 1, 4, 1.0, out)
    torch.cuda.synchronize()
    assert pool.check_device() == 0
    assert torch.all(out == 0)     # one token of zeros: softmax weight 1 on a zero V row
    pool.close()


def test_fused_step_bf16_output(pkg):
    """The fused step writing bf16 output gives the fp32 fused result rounded
    to nearest even, and the same pool contents."""
    dev = torch.device("cuda:0")
    lens = [15, 16, 300, 3000]
    outs = []
    for dtype in (torch.float32, torch.bfloat16):
        L, B, bt = 2, len(lens), 16
        cap = max(lens) + 2
        pool = pkg.Pool(num_layers=L, num_hot_blocks=sum(-(-(t + 1) // bt) for t in lens) + 8,
                        cold_bytes=B * (cap * L * 2 * HKV * D * 2 + 256), max_sessions=B,
                        max_batch=L * B, max_context=cap, alloc_seed=5)
        sids = [pool.session_create(cap) for _ in lens]
        for sid, t in zip(sids, lens):
            k, v = synth.kv_logical_torch(SEED, sid, range(L), HKV, D, 0, t, dev)
            pool.session_append(sid, k.permute(0, 2, 1, 3).contiguous(),
                                v.permute(0, 2, 1, 3).contiguous())
        q = synth.queries_torch(SEED, sids, range(L), HQ, D, dev)
        mb = -(-cap // bt)
        tables = torch.empty(B, mb, dtype=torch.int32, device=dev)
        slens = torch.empty(B, dtype=torch.int32, device=dev)
        kn, vn = token_rows(sids, lens, L, dev)
        pool.batch_reserve(sids, tables, mb, slens)
        out = torch.empty(L, B, HQ, D, dtype=dtype, device=dev)
        for l in range(L):
            pool.decode_append_attention(l, q[l], kn[l], vn[l], tables, slens, B, mb,
                                         1 / math.sqrt(D), out[l], overlap_previous=l > 0)
        torch.cuda.synchronize()
        assert pool.check_device() == 0
        outs.append(out.cpu())
        check_pool_holds_sessions(pool, sids, [t + 1 for t in lens], L, bt)
        pool.close()
    assert torch.equal(outs[0].to(torch.bfloat16).view(torch.int16), outs[1].view(torch.int16))

"""Residency mode (LRU, write-on-evict) on the GPU: data, not just decisions.

A random sequence of appends, pauses, resumes and decode batches runs on a
small pool under pressure, with the residency oracle in lock step (it fixes
which blocks are hot and which tokens each image holds). At every batch the
decode output is checked against the attention oracle; at the end every hot
block and every image prefix must hold the generator's values bit for bit.
"""
import math
import random

import numpy as np
import pytest
import torch

import oracle
import synth
from oracle.residency import NoHotBlocks, ResidencyOracle

pytestmark = pytest.mark.gpu

TOL = 1e-2


def bits(t):
    return t.contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


@pytest.mark.parametrize("fused,bt,mig_ctas", [(False, 16, 0), (True, 16, 0), (True, 64, 0),
                                               (True, 16, 1), (True, 64, 8)])
def test_residency_random_sequence(cuda_dev, fused, bt, mig_ctas):
    """fused: decode batches take their step token with the decode
    (kv_pool_batch_reserve + decode_append_attention, all layers). bt 64:
    evictions and fetches move 64-token blocks as four 16-token chunks.
    mig_ctas > 0: the evictions and fetches run capped at that many CTAs."""
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import Pool, kvtier

    L, Hq, Hkv, D, seed = 2, 32, 4, 128, 8
    nb = 40 if bt == 16 else 16                     # about the same pressure in tokens
    cap = 600
    pool = Pool(num_layers=L, num_hot_blocks=nb, cold_bytes=10 * cap * pool_token_bytes(L, Hkv),
                max_sessions=10, max_batch=L * 4, max_context=cap, alloc_seed=seed,
                lru_residency=True, block_tokens=bt)
    kvtier.kv_pool_set_migration_limit(pool.handle, mig_ctas)
    o = ResidencyOracle(nb, bt, seed=seed, token_bytes=pool.token_bytes)
    rnd = random.Random(seed)
    st = torch.cuda.Stream()
    live, T = [], {}
    q = synth.queries_torch(seed, range(4), range(L), Hq, D, cuda_dev)
    mb = -(-cap // bt)
    tables = torch.empty(4, mb, dtype=torch.int32, device=cuda_dev)
    slens = torch.empty(4, dtype=torch.int32, device=cuda_dev)
    torch.cuda.synchronize()     # q was made on the default stream
    checked = 0
    for step in range(260):
        r = rnd.random()
        if r < 0.1 and len(live) < 8:
            if rnd.random() < 0.5:
                n0 = rnd.randint(20, 200)
                sid = pool.session_create_paused(cap, n0)
                with torch.cuda.stream(st):   # on the stream the pool's work uses
                    synth.fill_image_torch(pool.image(sid), seed, sid, L, Hkv, D, n0)
                o.create_paused(sid, cap, n0)
                T[sid] = n0
            else:
                sid = pool.session_create(cap)
                o.create(sid, cap)
                T[sid] = 0
            live.append(sid)
            continue
        if not live:
            continue
        sid = rnd.choice(live)
        if o.s[sid].state == "paused":
            try:
                o.resume(sid)
            except NoHotBlocks:
                with pytest.raises(kvtier.KVError):
                    pool.session_resume(sid, st)
                continue
            pool.session_resume(sid, st)
        elif r < 0.55:
            n = rnd.randint(1, 40)
            if T[sid] + n > cap:
                continue
            try:
                o.append(sid, n)
            except NoHotBlocks:
                continue
            with torch.cuda.stream(st):       # values made on the appending stream
                k, v = synth.kv_logical_torch(seed, sid, range(L), Hkv, D, T[sid], T[sid] + n,
                                              cuda_dev)
                pool.session_append(sid, k.permute(0, 2, 1, 3).contiguous(),
                                    v.permute(0, 2, 1, 3).contiguous(), st)
            T[sid] += n
        elif r < 0.7:
            o.pause(sid)
            pool.session_pause(sid, st)
        elif r < 0.78:          # the next step's blocks ahead of it (same stream here)
            act = [x for x in live if o.s[x].state == "active"]
            nxt = rnd.sample(act, k=min(len(act), rnd.randint(1, 3)))
            busy = rnd.sample(act, k=min(len(act), rnd.randint(0, 2)))
            try:
                o.prefetch(nxt, busy)
            except NoHotBlocks:
                with pytest.raises(kvtier.KVError):
                    pool.prefetch(nxt, busy, st)
                continue
            pool.prefetch(nxt, busy, st)
        else:
            batch = [x for x in live if o.s[x].state == "active" and
                     (T[x] < cap if fused else T[x] > 0)]
            batch = rnd.sample(batch, k=min(len(batch), rnd.randint(1, 4)))
            if not batch:
                continue
            try:
                o.batch_reserve(batch) if fused else o.batch(batch)
            except NoHotBlocks:
                with pytest.raises(kvtier.KVError):
                    (pool.batch_reserve if fused else pool.batch_tables)(batch, tables, mb, slens, st)
                continue
            with torch.cuda.stream(st):
                out = torch.empty(L, len(batch), Hq, D, dtype=torch.float32, device=cuda_dev)
                qb = q[:, :len(batch)].contiguous()
                if fused:
                    ks, vs = [], []
                    for x in batch:
                        k, v = synth.kv_logical_torch(seed, x, range(L), Hkv, D, T[x], T[x] + 1,
                                                      cuda_dev)
                        ks.append(k[:, :, 0])
                        vs.append(v[:, :, 0])
                    kn, vn = torch.stack(ks, 1).contiguous(), torch.stack(vs, 1).contiguous()
                    pool.batch_reserve(batch, tables, mb, slens, st)
                    pool.decode_append_attention(-1, qb, kn, vn, tables, slens, len(batch), mb,
                                                 1 / math.sqrt(D), out, st)
                    for x in batch:
                        T[x] += 1
                else:
                    pool.batch_tables(batch, tables, mb, slens, st)
                    pool.decode_attention(-1, qb, tables, slens, len(batch), mb, 1 / math.sqrt(D),
                                          out, st)
            torch.cuda.synchronize()
            rows = np.full((len(batch), mb), -1, dtype=np.int32)
            for i, x in enumerate(batch):
                rows[i, :len(o.row(x))] = o.row(x)
            lens = [T[x] for x in batch]
            hot = synth.hot_pool_np(seed, batch, lens, rows, nb, L, Hkv, D, bt)
            ref = oracle.paged_decode(hot, bits(q[:, :len(batch)]), rows, lens, 1 / math.sqrt(D), Hq)
            got = out.double().cpu().numpy()
            assert np.max(np.abs(got - ref) / np.maximum(1.0, np.abs(ref))) <= TOL
            checked += 1
        assert pool.session_block_table(sid) == o.row(sid)
    torch.cuda.synchronize()
    assert pool.check_device() == 0
    stats = pool.stats()
    for key in ("bytes_packed", "bytes_unpacked", "blocks_evicted", "resume_blocks_hit",
                "resume_blocks_missed", "batch_blocks_fetched", "blocks_prefetched"):
        assert stats[key] == o.stats[key], key
    assert stats["blocks_evicted"] > 10 and checked > 10 and stats["blocks_prefetched"] > 0
    hv = pool.hot_view()
    for sid in live:
        s = o.s[sid]
        k, v = synth.session_kv_np(seed, sid, range(L), Hkv, D, s.T)
        img = bits(pool.image(sid))
        for j, slot in enumerate(s.slots):
            n = min(bt, s.T - j * bt)
            if slot >= 0:                     # hot copy: the whole block
                hb = bits(hv[slot])
                assert np.array_equal(hb[:, 0, :, :n], k[:, :, j * bt:j * bt + n])
                assert np.array_equal(hb[:, 1, :, :n], v[:, :, j * bt:j * bt + n])
            m = s.img[j]                       # cold copy: the tokens written so far
            assert np.array_equal(img[:, 0, :, j * bt:j * bt + m], k[:, :, j * bt:j * bt + m])
            assert np.array_equal(img[:, 1, :, j * bt:j * bt + m], v[:, :, j * bt:j * bt + m])
            if slot < 0:
                assert m == n
    pool.close()


def pool_token_bytes(L, Hkv):
    return L * 2 * Hkv * 128 * 2


def test_fetch_waits_for_an_eviction_on_another_stream(cuda_dev):
    """A block evicted on one stream (its tokens written to the image) and
    fetched back on another must be fetched after that write. Stream A is
    held back by a spin before a resume that evicts all of session Y's
    blocks; stream B then batches Y, fetching them from Y's image, and
    decodes. A fetch that did not wait would read the image before the
    eviction wrote it."""
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import Pool

    L, Hq, Hkv, D, bt, seed, cap = 2, 32, 4, 128, 16, 31, 64
    pool = Pool(num_layers=L, num_hot_blocks=6, cold_bytes=4 * cap * pool_token_bytes(L, Hkv),
                max_sessions=4, max_batch=L, max_context=cap, alloc_seed=seed,
                lru_residency=True)
    o = ResidencyOracle(6, bt, seed=seed, token_bytes=pool.token_bytes)
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()

    def append(sid, n):
        with torch.cuda.stream(sa):
            k, v = synth.kv_logical_torch(seed, sid, range(L), Hkv, D, 0, n, cuda_dev)
            pool.session_append(sid, k.permute(0, 2, 1, 3).contiguous(),
                                v.permute(0, 2, 1, 3).contiguous(), sa)

    y = pool.session_create(cap)
    o.create(y, cap)
    append(y, 40)                       # three blocks, none of them in the image yet
    o.append(y, 40)
    x = pool.session_create_paused(cap, 48)
    o.create_paused(x, cap, 48)
    with torch.cuda.stream(sa):
        synth.fill_image_torch(pool.image(x), seed, x, L, Hkv, D, 48)
    z = pool.session_create(cap)
    o.create(z, cap)
    append(z, 48)                       # the pool is full
    o.append(z, 48)
    q = synth.queries_torch(seed, [y], range(L), Hq, D, cuda_dev)
    mb = cap // bt
    tables = torch.empty(1, mb, dtype=torch.int32, device=cuda_dev)
    slens = torch.empty(1, dtype=torch.int32, device=cuda_dev)
    out = torch.full((L, 1, Hq, D), float("nan"), dtype=torch.float32, device=cuda_dev)
    torch.cuda.synchronize()

    with torch.cuda.stream(sa):
        torch.cuda._sleep(200_000_000)  # about 0.1 s of stream A before the eviction
    pool.session_resume(x, sa)          # evicts Y's three blocks, writing its 40 tokens
    o.resume(x)
    assert o.row(y) == [-1, -1, -1] and o.stats["bytes_packed"] == 40 * pool.token_bytes
    pool.batch_tables([y], tables, mb, slens, sb)    # Y's blocks back from its image
    o.batch([y])
    pool.decode_attention(-1, q, tables, slens, 1, mb, 1 / math.sqrt(D), out, sb)
    torch.cuda.synchronize()
    assert pool.check_device() == 0
    assert pool.session_block_table(y) == o.row(y)
    rows = np.full((1, mb), -1, dtype=np.int32)
    rows[0, :3] = o.row(y)
    hot = synth.hot_pool_np(seed, [y], [40], rows, 6, L, Hkv, D, bt)
    ref = oracle.paged_decode(hot, bits(q), rows, [40], 1 / math.sqrt(D), Hq)
    got = out.double().cpu().numpy()
    assert np.all(np.isfinite(got))
    assert np.max(np.abs(got - ref) / np.maximum(1.0, np.abs(ref))) <= TOL
    k, v = synth.session_kv_np(seed, y, range(L), Hkv, D, 40)
    hv = pool.hot_view()
    for j, slot in enumerate(o.row(y)):
        n = min(bt, 40 - j * bt)
        hb = bits(hv[slot])
        assert np.array_equal(hb[:, 0, :, :n], k[:, :, j * bt:j * bt + n])
        assert np.array_equal(hb[:, 1, :, :n], v[:, :, j * bt:j * bt + n])
    pool.close()


def test_prefetch_beside_a_running_step(cuda_dev):
    """kv_pool_prefetch as the trace driver uses it: while step k (sessions
    A, B) is still queued on the decode stream behind a spin, the prefetch of
    step k+1's sessions (C, two of whose blocks were evicted, and D) runs on
    the migration stream, evicting only the idle session E. Both steps must
    match the oracle, and step k+1 must find nothing left to fetch."""
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import Pool

    L, Hq, Hkv, D, bt, seed, cap = 2, 32, 4, 128, 16, 41, 200
    nb = 19                            # exactly the five sessions' blocks
    pool = Pool(num_layers=L, num_hot_blocks=nb, cold_bytes=6 * cap * pool_token_bytes(L, Hkv),
                max_sessions=6, max_batch=L * 2, max_context=cap, alloc_seed=seed,
                lru_residency=True)
    o = ResidencyOracle(nb, bt, seed=seed, token_bytes=pool.token_bytes)
    dst, mst = torch.cuda.Stream(), torch.cuda.Stream()
    T = {}

    def create(n0):
        sid = pool.session_create_paused(cap, n0)
        with torch.cuda.stream(mst):
            synth.fill_image_torch(pool.image(sid), seed, sid, L, Hkv, D, n0)
        o.create_paused(sid, cap, n0)
        T[sid] = n0
        return sid

    e, c, a, b, d = (create(n) for n in (96, 80, 48, 48, 32))
    for sid in (c, e, a, b, d):        # C least recent, then E; the pool is full
        pool.session_resume(sid, mst)
        o.resume(sid)
    k_, v_ = synth.kv_logical_torch(seed, d, range(L), Hkv, D, T[d], T[d] + 32, cuda_dev)
    with torch.cuda.stream(mst):       # D grows by two blocks: C's blocks 0 and 1 go
        pool.session_append(d, k_.permute(0, 2, 1, 3).contiguous(),
                            v_.permute(0, 2, 1, 3).contiguous(), mst)
    o.append(d, 32)
    T[d] += 32
    torch.cuda.synchronize()
    assert o.row(c)[:2] == [-1, -1] and min(o.row(c)[2:]) >= 0

    mb = -(-cap // bt)
    tables = [torch.empty(2, mb, dtype=torch.int32, device=cuda_dev) for _ in range(2)]
    slens = [torch.empty(2, dtype=torch.int32, device=cuda_dev) for _ in range(2)]
    q = synth.queries_torch(seed, range(2), range(L), Hq, D, cuda_dev)
    outs = []
    torch.cuda.synchronize()

    def step(i, batch, spin):
        with torch.cuda.stream(dst):
            if spin:
                torch.cuda._sleep(100_000_000)   # hold the step back (about 50 ms)
            pool.batch_tables(batch, tables[i], mb, slens[i], dst)
            o.batch(batch)
            out = torch.empty(L, 2, Hq, D, dtype=torch.float32, device=cuda_dev)
            pool.decode_attention(-1, q, tables[i], slens[i], 2, mb, 1 / math.sqrt(D), out, dst)
            done = torch.cuda.Event()
            done.record(dst)
        rows = np.full((2, mb), -1, dtype=np.int32)
        for r, x in enumerate(batch):
            rows[r, :len(o.row(x))] = o.row(x)
        outs.append((out, rows, [T[x] for x in batch], batch))
        return done

    done_k = step(0, [a, b], spin=True)
    pool.prefetch([c, d], busy=[a, b], stream=mst)   # beside step k; victims outside A-D
    o.prefetch([c, d], [a, b])
    assert o.stats["blocks_prefetched"] == 2 and o.row(e)[:2] == [-1, -1]
    mst.wait_event(done_k)
    fetched = o.stats["batch_blocks_fetched"]
    step(1, [c, d], spin=False)
    assert o.stats["batch_blocks_fetched"] == fetched   # nothing left for step k+1
    torch.cuda.synchronize()
    assert pool.check_device() == 0
    for key in ("blocks_evicted", "bytes_packed", "bytes_unpacked", "blocks_prefetched",
                "batch_blocks_fetched"):
        assert pool.stats()[key] == o.stats[key], key
    for out, rows, lens, batch in outs:
        hot = synth.hot_pool_np(seed, batch, lens, rows, nb, L, Hkv, D, bt)
        ref = oracle.paged_decode(hot, bits(q), rows, lens, 1 / math.sqrt(D), Hq)
        got = out.double().cpu().numpy()
        assert np.all(np.isfinite(got))
        assert np.max(np.abs(got - ref) / np.maximum(1.0, np.abs(ref))) <= TOL
    pool.close()

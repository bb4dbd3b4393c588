"""decode_attention_noalloc, the decode entry point that allocates nothing.

It serves callers that cannot let a library allocate device memory: an
engine that has budgeted nearly all HBM for its own arenas, or code that
cannot accept the device-wide synchronisation a cudaMalloc may cause. Its
split partials live in the library's fixed device scratch array, which
keeps whatever the previous call left there, so the test makes calls in a
row on different batches. It runs the same kernels with the same split plan
as the pool-based decode_attention, so each output must be bit-identical to
that call's on the same inputs; one call is also checked against the CPU
oracle with the parity tolerance of the other decode tests. The device's
free memory must not change across the calls. (The test itself allocates
its inputs with torch; only the entry point under test must not allocate.)
"""
import math

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

TOL = 1e-2


def _case(Pool, cuda_dev, lens, L, bt, seed, max_batch):
    nb = sum(-(-t // bt) for t in lens) + 5
    pool = Pool(num_layers=L, num_hot_blocks=nb, cold_bytes=256, block_tokens=bt,
                max_sessions=4, max_batch=max_batch, max_context=max(lens))
    tables = synth.random_block_tables(seed, lens, bt, nb)
    sess = list(range(len(lens)))
    synth.fill_hot_pool_torch(pool.hot, seed, sess, lens, tables, L, 4, 128, bt)
    q = synth.queries_torch(seed, sess, range(L), 32, 128, cuda_dev)
    return pool, nb, tables, sess, q


def _inputs(cuda_dev, tables, lens, rows, q, layer):
    tab = torch.as_tensor(tables[rows], device=cuda_dev).contiguous()
    sl = torch.as_tensor(np.asarray(lens[rows], dtype=np.int32), device=cuda_dev)
    qq = q[:, rows].contiguous() if layer < 0 else q[layer, rows].contiguous()
    return tab, sl, qq


def test_noalloc_bit_identical_to_pool_decode_and_allocates_nothing(cuda_dev):
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import Pool, kvtier

    L, Hq, bt, seed = 2, 32, 16, 17
    lens_a = [1, 15, 513, 4097, 9000]
    lens_b = [2049, 31, 700]
    lens = lens_a + lens_b
    pool, nb, tables, sess, q_all = _case(Pool, cuda_dev, lens, L, bt, seed, L * len(lens_a))
    cfg = kvtier.make_config(num_layers=L, num_q_heads=Hq, num_kv_heads=4, block_tokens=bt,
                             num_hot_blocks=nb, hot_base=pool.hot, device=0)
    scale = 1 / math.sqrt(128)

    # two calls in a row: all layers over batch a, then layer 1 over batch b
    calls = []
    for layer, rows in [(-1, slice(0, len(lens_a))), (1, slice(len(lens_a), len(lens)))]:
        tab, sl, q = _inputs(cuda_dev, tables, lens, rows, q_all, layer)
        shape = (L if layer < 0 else 1, tab.shape[0], Hq, 128)
        ref = torch.full(shape, float("nan"), dtype=torch.float32, device=cuda_dev)
        got = torch.full(shape, float("nan"), dtype=torch.float32, device=cuda_dev)
        calls.append((layer, rows, tab, sl, q, ref, got))

    def run_noalloc():
        for layer, _, tab, sl, q, _, got in calls:
            kvtier.decode_attention_noalloc(cfg, layer, q, tab, sl, tab.shape[0], tab.shape[1],
                                            scale, got)

    for layer, _, tab, sl, q, ref, _ in calls:
        pool.decode_attention(layer, q, tab, sl, tab.shape[0], tab.shape[1], scale, ref)
    run_noalloc()                   # first calls: per-device set-up, kernels loaded
    torch.cuda.synchronize()
    for _, _, _, _, _, ref, got in calls:
        assert torch.equal(got, ref)
        got.fill_(float("nan"))

    # the same two calls again, with the device's free memory watched
    free0 = torch.cuda.mem_get_info()[0]
    run_noalloc()
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    for _, _, _, _, _, ref, got in calls:
        assert torch.equal(got, ref)

    # the all-layer call against the CPU oracle
    hot = synth.hot_pool_np(seed, sess, lens, tables, nb, L, 4, 128, bt)
    rows = calls[0][1]
    want = oracle.paged_decode(hot, q_all[:, rows].cpu().view(torch.int16).numpy().view(np.uint16),
                               tables[rows], lens[rows], scale, Hq)
    g = calls[0][6].double().cpu().numpy()
    assert np.all(np.isfinite(g))
    assert np.max(np.abs(g - want) / np.maximum(1.0, np.abs(want))) <= TOL

    # a request larger than the fixed scratch is refused before any work
    tab = torch.as_tensor(tables[:1], device=cuda_dev)
    sl = torch.as_tensor(np.asarray(lens[:1], dtype=np.int32), device=cuda_dev)
    out = torch.empty(L, 64, Hq, 128, dtype=torch.float32, device=cuda_dev)
    with pytest.raises(kvtier.KVError) as e:
        kvtier.decode_attention_noalloc(cfg, -1, q_all, tab, sl, 64, 8192, scale, out)
    assert e.value.code == kvtier.KV_ERR_INVALID_ARG
    assert "scratch" in kvtier.kv_last_error()
    pool.close()


def test_noalloc_block_64(cuda_dev):
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import Pool, kvtier

    L, Hq, bt, seed = 2, 32, 64, 23
    lens = [1, 63, 64, 65, 3001, 5000]
    pool, nb, tables, sess, q = _case(Pool, cuda_dev, lens, L, bt, seed, L * len(lens))
    cfg = kvtier.make_config(num_layers=L, num_q_heads=Hq, num_kv_heads=4, block_tokens=bt,
                             num_hot_blocks=nb, hot_base=pool.hot, device=0)
    scale = 1 / math.sqrt(128)
    tab = torch.as_tensor(tables, device=cuda_dev)
    sl = torch.as_tensor(np.asarray(lens, dtype=np.int32), device=cuda_dev)
    ref = torch.full((L, len(lens), Hq, 128), float("nan"), dtype=torch.float32, device=cuda_dev)
    got = torch.full_like(ref, float("nan"))
    pool.decode_attention(-1, q, tab, sl, len(lens), tab.shape[1], scale, ref)
    for _ in range(2):
        kvtier.decode_attention_noalloc(cfg, -1, q, tab, sl, len(lens), tab.shape[1], scale, got)
        torch.cuda.synchronize()
        assert torch.equal(got, ref)
    hot = synth.hot_pool_np(seed, sess, lens, tables, nb, L, 4, 128, bt)
    want = oracle.paged_decode(hot, q.cpu().view(torch.int16).numpy().view(np.uint16), tables,
                               lens, scale, Hq)
    g = got.double().cpu().numpy()
    assert np.max(np.abs(g - want) / np.maximum(1.0, np.abs(want))) <= TOL
    pool.close()

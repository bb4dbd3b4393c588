"""decode_attention_noalloc, the decode entry point that allocates nothing.

It serves callers that cannot let a library allocate device memory: an
engine that has budgeted nearly all HBM for its own arenas, or code that
cannot accept the device-wide synchronisation a cudaMalloc may cause. Its
split partials live in the library's fixed device scratch array, which
keeps whatever the previous call left there, so the test makes two calls in
a row on different batches and checks each against the pool-based
decode_attention on the same inputs, with the parity tolerance of the other
decode tests. (The test itself allocates its inputs with torch; only the
entry point under test must not allocate.)
"""
import math

import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

TOL = 1e-2


def test_noalloc_matches_pool_decode_on_two_calls(cuda_dev):
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import Pool, kvtier

    L, Hq, Hkv, bt, seed = 2, 32, 4, 16, 17
    lens_a = [1, 15, 513, 4097, 9000]
    lens_b = [2049, 31, 700]
    lens = lens_a + lens_b
    nb = sum(-(-t // bt) for t in lens) + 5
    pool = Pool(num_layers=L, num_hot_blocks=nb, cold_bytes=256, max_sessions=4,
                max_batch=L * len(lens_a), max_context=max(lens))
    tables_all = synth.random_block_tables(seed, lens, bt, nb)
    sess = list(range(len(lens)))
    synth.fill_hot_pool_torch(pool.hot, seed, sess, lens, tables_all, L, Hkv, 128, bt)
    q_all = synth.queries_torch(seed, sess, range(L), Hq, 128, cuda_dev)
    cfg = kvtier.make_config(num_layers=L, num_q_heads=Hq, num_kv_heads=Hkv, block_tokens=bt,
                             num_hot_blocks=nb, hot_base=pool.hot, device=0)
    scale = 1 / math.sqrt(128)

    calls = [(-1, slice(0, len(lens_a))), (1, slice(len(lens_a), len(lens)))]
    for layer, rows in calls:
        tab = torch.as_tensor(tables_all[rows], device=cuda_dev).contiguous()
        sl = torch.as_tensor(np.asarray(lens[rows], dtype=np.int32), device=cuda_dev)
        q = q_all[:, rows].contiguous() if layer < 0 else q_all[layer, rows].contiguous()
        B = tab.shape[0]
        shape = (L if layer < 0 else 1, B, Hq, 128)
        ref = torch.full(shape, float("nan"), dtype=torch.float32, device=cuda_dev)
        got = torch.full(shape, float("nan"), dtype=torch.float32, device=cuda_dev)
        pool.decode_attention(layer, q, tab, sl, B, tab.shape[1], scale, ref)
        kvtier.decode_attention_noalloc(cfg, layer, q, tab, sl, B, tab.shape[1], scale, got)
        torch.cuda.synchronize()
        r = ref.double().cpu().numpy()
        g = got.double().cpu().numpy()
        assert np.all(np.isfinite(g))
        assert np.max(np.abs(g - r) / np.maximum(1.0, np.abs(r))) <= TOL

    # a request larger than the fixed scratch is refused before any work
    tab = torch.as_tensor(tables_all[:1], device=cuda_dev)
    sl = torch.as_tensor(np.asarray(lens[:1], dtype=np.int32), device=cuda_dev)
    out = torch.empty(L, 64, Hq, 128, dtype=torch.float32, device=cuda_dev)
    with pytest.raises(kvtier.KVError) as e:
        kvtier.decode_attention_noalloc(cfg, -1, q_all, tab, sl, 64, 8192, scale, out)
    assert e.value.code == kvtier.KV_ERR_INVALID_ARG
    assert "scratch" in kvtier.kv_last_error()
    pool.close()

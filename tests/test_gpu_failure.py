"""Failure detection on the GPU without a fault.

A decode wait that runs out: the test hook makes one warp of one CTA expect
16 bytes more than its first tile copy delivers, so that warp's bounded wait
(2 s) expires although every copy lands. The kernel must set
KV_DEVICE_TIMEOUT and finish; the host must see the flag through
kv_pool_check_device; and the same CUDA context must then decode correctly
again.

Split-arrival counters left non-zero (as decode calls that overlapped on
the GPU would leave them): kv_pool_check_device must report
KV_DEVICE_STALE_COUNTERS and reset them, after decode calls whose sessions
the split kernel merged itself left them at zero.
"""
import math
import time

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

TOL = 1e-2


def test_decode_wait_timeout_is_reported_and_context_survives(cuda_dev):
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import Pool, kvtier

    L, Hq, Hkv, D, bt, seed = 1, 32, 4, 128, 16, 6
    lens = [300, 77]
    nb = sum(-(-t // bt) for t in lens) + 4
    pool = Pool(num_layers=L, num_hot_blocks=nb, cold_bytes=256, max_sessions=2, max_batch=2,
                max_context=512)
    tables = synth.random_block_tables(seed, lens, bt, nb)
    synth.fill_hot_pool_torch(pool.hot, seed, [0, 1], lens, tables, L, Hkv, D, bt)
    q = synth.queries_torch(seed, [0, 1], range(L), Hq, D, cuda_dev)
    t = torch.as_tensor(tables, device=cuda_dev)
    s = torch.as_tensor(np.asarray(lens, dtype=np.int32), device=cuda_dev)
    hot = synth.hot_pool_np(seed, [0, 1], lens, tables, nb, L, Hkv, D, bt)
    ref = oracle.paged_decode(hot, q.cpu().view(torch.int16).numpy().view(np.uint16), tables,
                              lens, 1 / math.sqrt(D), Hq)

    def decode():
        out = torch.full((L, 2, Hq, D), float("nan"), dtype=torch.float32, device=cuda_dev)
        pool.decode_attention(0, q[0], t, s, 2, t.shape[1], 1 / math.sqrt(D), out[0])
        torch.cuda.synchronize()
        return out.double().cpu().numpy()

    def err(got):
        return np.max(np.abs(got - ref) / np.maximum(1.0, np.abs(ref)))

    assert err(decode()) <= TOL and pool.check_device() == 0

    kvtier.kv_pool_inject_decode_timeout(pool.handle, 1)
    t0 = time.monotonic()
    decode()                                   # returns: the wait is bounded
    elapsed = time.monotonic() - t0
    flags = pool.check_device()
    assert flags == kvtier.KV_DEVICE_TIMEOUT
    assert 1.5 < elapsed < 60                  # one 2 s limit (plus the bounded drain)
    assert "timed out" in kvtier.kv_last_error() or "flags 4" in kvtier.kv_last_error()

    # the hook disarmed itself and the context is intact
    t0 = time.monotonic()
    got = decode()
    assert time.monotonic() - t0 < 1.0
    assert err(got) <= TOL and pool.check_device() == 0
    pool.close()


def test_stale_arrival_counters_are_reported_and_reset(cuda_dev):
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import Pool, kvtier

    # all layers in one call: 16 sessions x 4 splits x 4 kv-heads x 8 layers = 2 048 CTAs,
    # at least 8 per SM, so the split kernel merges these sessions of 2..4 splits itself
    L, Hq, Hkv, D, bt, seed = 8, 32, 4, 128, 16, 9
    lens = [4096, 3000, 2049, 1025, 4000, 3500, 2600, 1100] * 2
    sess = list(range(len(lens)))
    nb = sum(-(-t // bt) for t in lens) + 4
    pool = Pool(num_layers=L, num_hot_blocks=nb, cold_bytes=256, max_sessions=len(lens),
                max_batch=L * len(lens), max_context=max(lens))
    tables = synth.random_block_tables(seed, lens, bt, nb)
    synth.fill_hot_pool_torch(pool.hot, seed, sess, lens, tables, L, Hkv, D, bt)
    q = synth.queries_torch(seed, sess, range(L), Hq, D, cuda_dev)
    t = torch.as_tensor(tables, device=cuda_dev)
    s = torch.as_tensor(np.asarray(lens, dtype=np.int32), device=cuda_dev)

    def decode():
        out = torch.full((L, len(lens), Hq, D), float("nan"), dtype=torch.float32,
                         device=cuda_dev)
        pool.decode_attention(-1, q, t, s, len(lens), t.shape[1], 1 / math.sqrt(D), out)
        torch.cuda.synchronize()
        return out.cpu().numpy()

    first = decode()
    assert pool.check_device() == 0            # every call leaves the counters at zero
    hot = synth.hot_pool_np(seed, sess, lens, tables, nb, L, Hkv, D, bt)
    ref = oracle.paged_decode(hot, q.cpu().view(torch.int16).numpy().view(np.uint16), tables,
                              lens, 1 / math.sqrt(D), Hq)
    assert np.max(np.abs(first - ref) / np.maximum(1.0, np.abs(ref))) <= TOL

    kvtier.kv_pool_inject_stale_counter(pool.handle)
    assert pool.check_device() == kvtier.KV_DEVICE_STALE_COUNTERS
    assert pool.check_device() == 0            # reset by the check
    again = decode()
    assert np.array_equal(first.view(np.int32), again.view(np.int32))
    assert pool.check_device() == 0
    pool.close()

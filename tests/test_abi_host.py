"""C-ABI library: symbol exports and the pool's host logic, without a GPU.

The pool is created with KV_POOL_HOST_LOGIC_ONLY: no CUDA call is made and no
data moves, so these tests exercise placement, session states, capacity
errors, write-on-evict accounting and the no-change-on-error rule. Placement
is checked against the oracle's restatement of the free-list contract.
"""
import os
import re

import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def kv():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import kvtier
    return kvtier


def header_functions():
    src = open(os.path.join(ROOT, "include", "kvtier.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(\w+)\s*\(", src, flags=re.M)))


def test_library_exports_every_declared_symbol(kv):
    names = header_functions()
    assert len(names) >= 20
    for n in names:
        assert hasattr(kv.lib, n), f"libkvtier.so does not export {n}"
    assert sorted(kv.EXPORTS) == names


def test_sizes_match_paper_shape(kv):
    cfg = kv.make_config(num_layers=48, num_hot_blocks=1)
    assert kv.kv_token_bytes(cfg) == oracle.kv_bytes_per_token(48, 4, 128) == 96 * 1024
    assert kv.kv_block_bytes(cfg) == 1536 * 1024


def test_decode_split_bound(kv):
    """S(t) is the tight bound of the per-session split count over T <= t, for
    splits of clamp(ceil(tiles/16), 64, 128) 16-token tiles."""
    import numpy as np
    T = np.arange(1, 140_001)
    tiles = -(-T // 16)
    st = np.clip(-(-tiles // 16), 64, 128)
    running = np.maximum.accumulate(-(-tiles // st))
    for t in (1, 1024, 1025, 4096, 16384, 16385, 32768, 32769, 65536, 131072, 140000):
        assert kv.kv_decode_splits(t) == running[t - 1], t
    assert [kv.kv_decode_splits(t) for t in (1024, 1025, 16384, 32768, 32769, 131072)] == \
        [1, 2, 16, 16, 17, 64]
    assert kv.kv_decode_splits(0) == 0 and kv.kv_decode_splits(-5) == 0


def host_pool(kv, nb=40, seed=7, L=2, bt=16, cold_tokens=10000, max_sessions=8, max_context=4096):
    cfg = kv.make_config(num_layers=L, num_hot_blocks=nb, block_tokens=bt, alloc_seed=seed,
                         max_sessions=max_sessions, max_context=max_context,
                         cold_bytes=cold_tokens * L * 2 * 4 * 128 * 2,
                         flags=kv.KV_POOL_HOST_LOGIC_ONLY)
    return kv.kv_pool_create(cfg), cfg


def snapshot(kv, pool, sids):
    infos = {}
    for s in sids:
        i = kv.session_info(pool, s)
        infos[s] = (i.state, i.num_blocks, i.tokens, i.capacity, i.cold_valid,
                    tuple(kv.session_block_table(pool, s)))
    return kv.kv_pool_free_list(pool), infos, kv.kv_pool_get_stats(pool)


def test_placement_follows_free_list_contract(kv):
    pool, cfg = host_pool(kv, nb=40, seed=7)
    ref = oracle.FreeList(40, 7)
    assert kv.kv_pool_free_list(pool) == list(ref.contents())
    a = kv.session_create(pool, 2000)
    b = kv.session_create(pool, 2000)
    kv.session_append(pool, a, None, None, 37, None)      # 3 blocks
    exp_a = list(ref.pop(3))
    kv.session_append(pool, b, None, None, 16, None)      # 1 block
    exp_b = list(ref.pop(1))
    kv.session_append(pool, a, None, None, 11, None)      # 48 tokens: still 3 blocks
    kv.session_append(pool, a, None, None, 1, None)       # 49: a 4th block
    exp_a += list(ref.pop(1))
    assert kv.session_block_table(pool, a) == exp_a
    assert kv.session_block_table(pool, b) == exp_b
    kv.session_pause(pool, a, None)
    ref.push(exp_a)
    assert kv.kv_pool_free_list(pool) == list(ref.contents())
    kv.kv_pool_shuffle_free(pool, 1234)
    ref.shuffle(1234)
    assert kv.kv_pool_free_list(pool) == list(ref.contents())
    kv.session_resume(pool, a, None)
    assert kv.session_block_table(pool, a) == list(ref.pop(4))
    assert kv.kv_pool_free_list(pool) == list(ref.contents())
    kv.kv_pool_destroy(pool)


def test_state_machine_errors(kv):
    pool, _ = host_pool(kv)
    s = kv.session_create(pool, 100)
    with pytest.raises(kv.KVError) as e:
        kv.session_resume(pool, s, None)
    assert e.value.code == kv.KV_ERR_BAD_STATE
    kv.session_append(pool, s, None, None, 5, None)
    kv.session_pause(pool, s, None)
    for fn in (lambda: kv.session_pause(pool, s, None),
               lambda: kv.session_append(pool, s, None, None, 1, None)):
        with pytest.raises(kv.KVError) as e:
            fn()
        assert e.value.code == kv.KV_ERR_BAD_STATE
    with pytest.raises(kv.KVError) as e:
        kv.decode_attention(pool, 0, 256, 512, 768, 1, 1, 1.0, 1024, None)   # aligned dummies
    assert e.value.code == kv.KV_ERR_BAD_STATE
    with pytest.raises(kv.KVError) as e:
        kv.session_info(pool, 5)
    assert e.value.code == kv.KV_ERR_INVALID_ARG
    kv.kv_pool_destroy(pool)


def test_capacity_errors_change_nothing(kv):
    pool, _ = host_pool(kv, nb=5, cold_tokens=300, max_sessions=3)
    s = kv.session_create(pool, 100)
    kv.session_append(pool, s, None, None, 60, None)        # 4 blocks of 5
    before = snapshot(kv, pool, [s])
    with pytest.raises(kv.KVError) as e:
        kv.session_append(pool, s, None, None, 41, None)    # past capacity 100
    assert e.value.code == kv.KV_ERR_INVALID_ARG
    t = kv.session_create(pool, 100)
    before = snapshot(kv, pool, [s, t])
    with pytest.raises(kv.KVError) as e:
        kv.session_append(pool, t, None, None, 32, None)    # needs 2 blocks, 1 free
    assert e.value.code == kv.KV_ERR_NO_HOT_BLOCKS
    assert snapshot(kv, pool, [s, t]) == before
    with pytest.raises(kv.KVError) as e:
        kv.session_create(pool, 200)                        # cold arena: 300 tokens total
    assert e.value.code == kv.KV_ERR_NO_COLD_SPACE
    kv.session_pause(pool, s, None)
    kv.session_append(pool, t, None, None, 65, None)        # takes all 5 blocks
    with pytest.raises(kv.KVError) as e:
        kv.session_resume(pool, s, None)
    assert e.value.code == kv.KV_ERR_NO_HOT_BLOCKS
    assert kv.session_info(pool, s).state == kv.KV_SESSION_PAUSED
    kv.kv_pool_destroy(pool)


def test_cold_arena_first_fit_and_coalescing(kv):
    pool, _ = host_pool(kv, cold_tokens=300, max_sessions=8)
    a = kv.session_create(pool, 100)
    b = kv.session_create(pool, 100)
    c = kv.session_create(pool, 100)
    with pytest.raises(kv.KVError):
        kv.session_create(pool, 1)
    kv.session_destroy(pool, b)
    kv.session_destroy(pool, c)
    d = kv.session_create(pool, 200)     # b's and c's ranges coalesced
    assert kv.kv_pool_get_stats(pool)["cold_bytes_used"] == 300 * 2 * 2 * 4 * 128 * 2
    kv.session_destroy(pool, a)
    kv.session_destroy(pool, d)
    assert kv.kv_pool_get_stats(pool)["cold_bytes_used"] == 0
    kv.kv_pool_destroy(pool)


def test_write_on_evict_accounting(kv):
    pool, cfg = host_pool(kv)
    tb = kv.kv_token_bytes(cfg)
    s = kv.session_create(pool, 1000)
    kv.session_append(pool, s, None, None, 100, None)
    kv.session_pause(pool, s, None)
    assert kv.kv_pool_get_stats(pool)["bytes_packed"] == 100 * tb
    assert kv.session_info(pool, s).cold_valid == 100
    kv.session_resume(pool, s, None)
    assert kv.kv_pool_get_stats(pool)["bytes_unpacked"] == 100 * tb
    kv.session_pause(pool, s, None)      # nothing new: no bytes written (at most once)
    assert kv.kv_pool_get_stats(pool)["bytes_packed"] == 100 * tb
    kv.session_resume(pool, s, None)
    kv.session_append(pool, s, None, None, 7, None)
    kv.session_pause(pool, s, None)      # only the 7 new tokens
    st = kv.kv_pool_get_stats(pool)
    assert st["bytes_packed"] == 107 * tb
    assert st["pauses"] == 3 and st["resumes"] == 2
    kv.kv_pool_destroy(pool)


def test_paused_session_creation(kv):
    pool, _ = host_pool(kv, nb=40)
    s = kv.session_create_paused(pool, 500, 130)
    i = kv.session_info(pool, s)
    assert (i.state, i.tokens, i.cold_valid, i.num_blocks) == (kv.KV_SESSION_PAUSED, 130, 130, 0)
    kv.session_resume(pool, s, None)
    assert kv.session_info(pool, s).num_blocks == 9
    kv.kv_pool_destroy(pool)


@pytest.mark.parametrize("op", ["append", "pause", "resume"])
def test_injected_cuda_failure_is_atomic(kv, op):
    pool, _ = host_pool(kv)
    s = kv.session_create(pool, 1000)
    kv.session_append(pool, s, None, None, 40, None)
    if op == "resume":
        kv.session_pause(pool, s, None)
    run = {"append": lambda: kv.session_append(pool, s, None, None, 30, None),
           "pause": lambda: kv.session_pause(pool, s, None),
           "resume": lambda: kv.session_resume(pool, s, None)}[op]
    failures = 0
    for n in range(1, 20):
        before = snapshot(kv, pool, [s])
        kv.kv_pool_inject_cuda_failure(pool, n)
        try:
            run()
        except kv.KVError as e:
            assert e.code == kv.KV_ERR_CUDA
            assert "injected" in kv.kv_last_error()
            assert snapshot(kv, pool, [s]) == before
            failures += 1
            continue
        break
    assert failures >= 2   # the op makes several device calls; each failure point was covered
    kv.kv_pool_inject_cuda_failure(pool, 0)
    kv.kv_pool_destroy(pool)


def test_bad_configs_rejected(kv):
    bad = [dict(head_dim=64), dict(block_tokens=32), dict(num_q_heads=24),
           dict(num_kv_heads=16, num_q_heads=16), dict(num_q_heads=48, num_kv_heads=4)]
    for over in bad:
        args = dict(num_layers=2, num_hot_blocks=10, flags=kv.KV_POOL_HOST_LOGIC_ONLY)
        args.update(over)
        with pytest.raises(kv.KVError) as e:
            kv.kv_pool_create(kv.make_config(**args))
        assert e.value.code == kv.KV_ERR_INVALID_ARG
    with pytest.raises(kv.KVError):   # real pools need arenas
        kv.kv_pool_create(kv.make_config(num_layers=2, num_hot_blocks=10))


def test_decode_arguments_checked_before_any_launch(kv):
    """Every argument of a decode call is validated before the pool's state
    (a host-logic pool then refuses to compute): layer, batch size, table
    width, the workspace the call needs, the scale."""
    cfg = kv.make_config(num_layers=4, num_hot_blocks=64, max_batch=2, max_context=1024,
                         flags=kv.KV_POOL_HOST_LOGIC_ONLY)
    pool = kv.kv_pool_create(cfg)
    q, tab, lens, out = 256, 512, 768, 1024            # aligned stand-ins, never dereferenced
    cases = [
        dict(layer=4), dict(layer=-2), dict(B=0), dict(B=65536), dict(layer=-1, B=16384),
        dict(max_blocks=0), dict(max_blocks=(1 << 26) + 1),
        dict(max_blocks=1024),                  # 16K-token tables: 16 splits x 32 heads > 2 x 32 x 1
        dict(layer=-1, B=2),                    # 4 layers x 2 rows x 32 heads > 64 rows
        dict(scale=float("nan")), dict(scale=float("inf")),
    ]
    for c in cases:
        a = dict(layer=0, B=1, max_blocks=64, scale=1.0) | c
        with pytest.raises(kv.KVError) as e:
            kv.decode_attention(pool, a["layer"], q, tab, lens, a["B"], a["max_blocks"], a["scale"],
                                out, None)
        assert e.value.code == kv.KV_ERR_INVALID_ARG, c
    for ok in (dict(layer=0, B=2, max_blocks=64), dict(layer=3, B=1, max_blocks=64)):
        with pytest.raises(kv.KVError) as e:    # valid arguments: the pool cannot compute
            kv.decode_attention(pool, ok["layer"], q, tab, lens, ok["B"], ok["max_blocks"], 1.0,
                                out, None)
        assert e.value.code == kv.KV_ERR_BAD_STATE, ok
    kv.kv_pool_destroy(pool)

"""Random calls, many of them invalid, against the C ABI's host logic.

Every call must either succeed or return one of the documented error codes,
and the pool's invariants must hold after each: every hot block is free or
owned by exactly one session, the free list holds no duplicates, session
lengths never exceed their capacity, and the cold arena accounting matches
the live sessions.
"""
import random

import pytest

CODES = None


@pytest.fixture(scope="module")
def kv():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import kvtier
    global CODES
    CODES = {kvtier.KV_ERR_INVALID_ARG, kvtier.KV_ERR_BAD_STATE, kvtier.KV_ERR_NO_HOT_BLOCKS,
             kvtier.KV_ERR_NO_COLD_SPACE}
    return kvtier


def check_invariants(kv, pool, nb, sids, token_bytes, lru):
    free = kv.kv_pool_free_list(pool)
    assert len(free) == len(set(free))
    owned = []
    cold = 0
    for sid in sids:
        info = kv.session_info(pool, sid)
        row = kv.session_block_table(pool, sid)
        hot = [b for b in row if b >= 0]
        owned += hot
        assert info.tokens <= info.capacity
        assert info.num_blocks == len(hot)
        if not lru and info.state == kv.KV_SESSION_PAUSED:
            assert not hot                    # simple mode frees on pause
        if info.state == kv.KV_SESSION_ACTIVE and not lru:
            assert len(row) == -(-info.tokens // 16)
        cold += -(-(info.capacity * token_bytes) // 256) * 256
    assert len(owned) == len(set(owned))
    assert not set(owned) & set(free)
    assert sorted(owned + free) == list(range(nb))
    st = kv.kv_pool_get_stats(pool)
    assert st["cold_bytes_used"] == cold
    assert st["free_blocks"] == len(free) and st["used_blocks"] == len(owned)


@pytest.mark.parametrize("lru", [False, True])
@pytest.mark.parametrize("seed", [0, 1, 2])
def test_random_calls_keep_invariants(kv, lru, seed):
    rnd = random.Random(seed * 7 + lru)
    nb = 24
    flags = kv.KV_POOL_HOST_LOGIC_ONLY | (kv.KV_POOL_LRU_RESIDENCY if lru else 0)
    cfg = kv.make_config(num_layers=1, num_hot_blocks=nb, alloc_seed=seed, max_sessions=6,
                         max_context=512, max_batch=8, cold_bytes=2000 * 1 * 2 * 4 * 128 * 2,
                         flags=flags)
    tb = kv.kv_token_bytes(cfg)
    pool = kv.kv_pool_create(cfg)
    sids = []
    ok = errs = 0
    for _ in range(1500):
        op = rnd.randrange(10)
        sid = rnd.choice(sids + [-1, 99, rnd.randrange(-3, 9)]) if rnd.random() < 0.9 and sids \
            else rnd.randrange(-3, 9)
        try:
            if op == 0:
                cap = rnd.choice([0, 1, 17, 300, 512, 513, 2000])
                if rnd.random() < 0.5:
                    s = kv.session_create(pool, cap)
                else:
                    s = kv.session_create_paused(pool, cap, rnd.choice([-1, 0, 1, 40, cap, cap + 1]))
                sids.append(s)
            elif op == 1:
                kv.session_append(pool, sid, None, None, rnd.choice([-1, 0, 1, 5, 33, 600]), None)
            elif op == 2:
                kv.session_pause(pool, sid, None)
            elif op == 3:
                kv.session_resume(pool, sid, None)
            elif op == 4 and rnd.random() < 0.3:
                kv.session_destroy(pool, sid)
                if sid in sids:
                    sids.remove(sid)
            elif op == 5:
                kv.kv_pool_shuffle_free(pool, rnd.randrange(1 << 40))
            elif op == 6 and lru:
                batch = rnd.sample(sids + [42], k=min(len(sids) + 1, rnd.randint(1, 3)))
                kv.kv_pool_batch_tables(pool, batch, None, rnd.choice([0, 1, 64]), None)
            elif op == 7:
                kv.session_info(pool, sid)
            elif op == 8:
                kv.kv_pool_set_migration_limit(pool, rnd.choice([-1, 0, 64]))
            elif op == 9:
                batch = [rnd.choice(sids + [-1, 77]) if sids else -1
                         for _ in range(rnd.randint(1, 3))]
                kv.kv_pool_batch_reserve(pool, batch, None, rnd.choice([0, 1, 64]), None)
            ok += 1
        except kv.KVError as e:
            assert e.code in CODES, (op, e)
            assert kv.kv_last_error()
            errs += 1
        check_invariants(kv, pool, nb, sids, tb, lru)
    assert ok > 200 and errs > 200
    kv.kv_pool_destroy(pool)


def test_decode_flags_and_arguments_rejected(kv):
    cfg = kv.make_config(num_layers=2, num_hot_blocks=8, flags=kv.KV_POOL_HOST_LOGIC_ONLY,
                         cold_bytes=1 << 24)
    pool = kv.kv_pool_create(cfg)
    with pytest.raises(kv.KVError) as e:
        kv.decode_attention_ex(pool, 0, 1, 1, 1, 1, 1, 1.0, 1, 1 << 7, None)
    assert e.value.code == kv.KV_ERR_INVALID_ARG       # unknown flag
    with pytest.raises(kv.KVError) as e:
        kv.kv_pool_set_migration_limit(pool, -5)
    assert e.value.code == kv.KV_ERR_INVALID_ARG
    for kn, vn, code in ((None, 256, kv.KV_ERR_INVALID_ARG), (256, None, kv.KV_ERR_INVALID_ARG),
                         (264, 256, kv.KV_ERR_INVALID_ARG),       # not 16-byte aligned
                         (256, 512, kv.KV_ERR_BAD_STATE)):        # host-logic pool: no decode
        with pytest.raises(kv.KVError) as e:
            kv.decode_append_attention(pool, 0, 1024, kn, vn, 2048, 4096, 1, 1, 1.0, 8192)
        assert e.value.code == code
    for args in ((1026, 2048, 4096, 8192), (1024, 2048, 4096, 8200), (1024, 2050, 4096, 8192)):
        with pytest.raises(kv.KVError) as e:       # misaligned q, out, block_tables
            kv.decode_attention(pool, 0, args[0], args[1], args[2], 1, 1, 1.0, args[3], None)
        assert e.value.code == kv.KV_ERR_INVALID_ARG and "align" in kv.kv_last_error()
    sid = kv.session_create(pool, 64)
    with pytest.raises(kv.KVError) as e:
        kv.session_append(pool, sid, 1032, 1024, 1, None)
    assert e.value.code == kv.KV_ERR_INVALID_ARG
    kv.session_append(pool, sid, 1024, 2048, 1, None)   # aligned: accepted (host logic only)
    with pytest.raises(kv.KVError) as e:               # misaligned batch outputs
        kv.kv_pool_batch_reserve(pool, [sid], 1026, 4, 2048, None)
    assert e.value.code == kv.KV_ERR_INVALID_ARG
    kv.kv_pool_inject_decode_timeout(pool, 1)          # armed, then disarmed: host state only
    kv.kv_pool_inject_decode_timeout(pool, 0)
    with pytest.raises(kv.KVError) as e:               # no device workspace to touch
        kv.kv_pool_inject_stale_counter(pool)
    assert e.value.code == kv.KV_ERR_BAD_STATE
    kv.kv_pool_destroy(pool)
    with pytest.raises(kv.KVError) as e:
        kv.kv_pool_inject_stale_counter(None)
    assert e.value.code == kv.KV_ERR_INVALID_ARG
    with pytest.raises(kv.KVError) as e:
        kv.kv_pool_inject_decode_timeout(None, 1)
    assert e.value.code == kv.KV_ERR_INVALID_ARG
    with pytest.raises(kv.KVError) as e:              # no-alloc path: misaligned out
        kv.decode_attention_noalloc(kv.make_config(num_layers=2, num_hot_blocks=8, hot_base=256),
                                    0, 1024, 2048, 4096, 1, 1, 1.0, 8200)
    assert e.value.code == kv.KV_ERR_INVALID_ARG
    with pytest.raises(kv.KVError) as e:              # no-alloc path: bad shapes, before any CUDA call
        kv.decode_attention_noalloc(kv.make_config(num_layers=2, num_hot_blocks=8, head_dim=64,
                                                   hot_base=256), 0, 1, 1, 1, 1, 1, 1.0, 1)
    assert e.value.code == kv.KV_ERR_INVALID_ARG

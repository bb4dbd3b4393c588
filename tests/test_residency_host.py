"""Block residency (LRU, write-on-evict) on the host, without a GPU.

First the oracle's restatement of the policy is pinned to properties the
paper states and to a scenario worked by hand; then the library's
bookkeeping (a host-logic-only pool in residency mode) is compared with the
oracle decision by decision on random operation sequences under pressure.
"""
import random

import pytest

import oracle
from oracle.residency import NoHotBlocks, ResidencyOracle

BT, TB = 16, 1000          # block tokens; bytes per token (any constant)


def pack_tokens(o):
    """token -> number of times it was written to the cold tier"""
    cnt = {}
    for kind, sid, j, slot, t0, t1 in o.log:
        if kind == "pack":
            for t in range(j * BT + t0, j * BT + t1):
                cnt[(sid, t)] = cnt.get((sid, t), 0) + 1
    return cnt


def test_hand_worked_eviction_scenario():
    o = ResidencyOracle(6, BT, seed=3, token_bytes=TB)
    start = list(o.fl.contents())
    o.create(0, 1000)
    o.append(0, 40)            # A: 3 blocks, time 1
    o.create(1, 1000)
    o.append(1, 32)            # B: 2 blocks, time 2
    assert o.fl.n == 1
    a_slots = o.row(0)
    assert a_slots == [start[5], start[4], start[3]]     # popped from the end
    o.pause(0)
    o.create(2, 1000)
    o.append(2, 40)            # C needs 3 blocks: 1 free + A's blocks 0 and 1 (A least recent)
    assert o.row(0) == [-1, -1, a_slots[2]]
    assert o.stats["blocks_evicted"] == 2
    assert o.stats["bytes_packed"] == 32 * TB             # two full blocks, written once
    o.resume(0)                # A's blocks 0,1 missing: evict B's (LRU among B, C), hit = 1
    assert o.stats["resume_blocks_hit"] == 1 and o.stats["resume_blocks_missed"] == 2
    assert o.row(1) == [-1, -1]
    assert o.stats["bytes_packed"] == 64 * TB             # + B's 32 tokens
    assert o.stats["bytes_unpacked"] == 32 * TB           # A's two blocks back
    o.pause(0)
    o.resume(0)                # nothing evicted since: all hits, nothing moves
    assert o.stats["resume_blocks_hit"] == 4 and o.stats["bytes_unpacked"] == 32 * TB


def test_each_token_written_at_most_once():
    rnd = random.Random(5)
    o = ResidencyOracle(10, BT, seed=1, token_bytes=TB)
    for sid in range(4):
        o.create(sid, 10_000)
    for _ in range(400):
        sid = rnd.randrange(4)
        s = o.s[sid]
        try:
            if s.state == "active":
                if rnd.random() < 0.7:
                    o.append(sid, rnd.randint(1, 30))
                else:
                    o.pause(sid)
            else:
                o.resume(sid)
        except NoHotBlocks:
            pass
    cnt = pack_tokens(o)
    assert cnt and max(cnt.values()) == 1
    total = sum(s.T for s in o.s.values())
    assert o.stats["bytes_packed"] <= total * TB


def test_no_pressure_no_eviction_full_hits():
    o = ResidencyOracle(100, BT, seed=2, token_bytes=TB)
    for sid in range(3):
        o.create(sid, 1000)
        o.append(sid, 100)
        o.pause(sid)
    for sid in range(3):
        o.resume(sid)
    assert o.stats["blocks_evicted"] == 0 and o.stats["bytes_packed"] == 0
    assert o.stats["resume_blocks_missed"] == 0 and o.stats["resume_blocks_hit"] == 21


def test_recency_keeps_the_active_set_hot():
    """Batched every step, the active sessions are always the most recent:
    with room for them, only idle sessions' blocks are evicted."""
    o = ResidencyOracle(40, BT, seed=4, token_bytes=TB)
    active, idle = [0, 1, 2], [3, 4, 5, 6]
    for sid in active + idle:
        o.create(sid, 10_000)
    for sid in idle:
        o.append(sid, 64)
        o.pause(sid)
    for sid in active:
        o.append(sid, 100)
    for step in range(100):    # the active set grows to 3 x 13 = 39 of 40 blocks
        o.batch(active)
        for sid in active:
            o.append(sid, 1)
        assert all(slot >= 0 for sid in active for slot in o.row(sid))
    assert o.stats["blocks_evicted"] > 0
    evicted_active = [l for l in o.log if l[0] == "pack" and l[1] in active]
    assert not evicted_active


def test_no_pinning_spills_instead_of_failing():
    o = ResidencyOracle(8, BT, seed=6, token_bytes=TB)
    o.create(0, 1000)
    o.append(0, 64)            # 4 blocks
    o.create(1, 1000)
    o.append(1, 64)            # 4 blocks: pool full, both active
    o.append(0, 16)            # needs one more: session 1 (active, older) spills a block
    assert o.row(1)[0] == -1
    o.batch([1])               # bringing it back evicts session 0's oldest block
    assert all(x >= 0 for x in o.row(1)) and o.row(0)[0] == -1
    with pytest.raises(NoHotBlocks):
        o.batch([0, 1])        # 9 blocks can never fit in 8


def test_batch_reserve_hand_worked():
    o = ResidencyOracle(6, BT, seed=7, token_bytes=TB)
    start = list(o.fl.contents())
    o.create(0, 1000)
    o.append(0, 32)            # A: 2 full blocks
    o.create(1, 1000)
    o.append(1, 20)            # B: 2 blocks, tail holds 4 tokens
    o.create(2, 1000)
    o.append(2, 20)            # C: 2 blocks; pool full
    o.pause(2)
    c_row = o.row(2)
    o.batch_reserve([0, 1])    # A's tail is full: one block, taken from C's block 0 (LRU)
    assert o.row(2) == [-1, c_row[1]]
    assert o.row(0) == [start[5], start[4], c_row[0]]
    assert o.s[0].T == 33 and o.s[1].T == 21
    assert o.stats["bytes_packed"] == 16 * TB and o.stats["blocks_evicted"] == 1
    assert o.stats["bytes_appended"] == (32 + 20 + 20 + 2) * TB
    o.resume(2)                # C's block 0 back: evicts from the least recent of A, B
    o.batch_reserve([2])       # C at 21 tokens: no new block
    assert o.s[2].T == 21 and len(o.row(2)) == 2
    with pytest.raises(AssertionError):
        o.batch_reserve([0, 0])


def test_batch_reserve_equals_appends_then_batch_without_pressure():
    """With free blocks to spare, reserving a step's tokens for a batch is
    one-token appends in batch order followed by batching them."""
    a = ResidencyOracle(200, BT, seed=9, token_bytes=TB)
    b = ResidencyOracle(200, BT, seed=9, token_bytes=TB)
    rnd = random.Random(3)
    for o in (a, b):
        for sid in range(5):
            o.create(sid, 10_000)
    for step in range(120):
        batch = rnd.sample(range(5), k=rnd.randint(1, 5))
        a.batch_reserve(batch)
        for sid in batch:
            b.append(sid, 1)
        b.batch(batch)
        assert [a.row(s) for s in range(5)] == [b.row(s) for s in range(5)]
        assert list(a.fl.contents()) == list(b.fl.contents())
    assert a.stats == b.stats


# ------------------------------------------------ library vs oracle

@pytest.fixture(scope="module")
def kv():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import kvtier
    return kvtier


def lib_pool(kv, nb, seed):
    cfg = kv.make_config(num_layers=1, num_hot_blocks=nb, block_tokens=BT, alloc_seed=seed,
                         max_sessions=8, max_context=4096, max_batch=8,
                         cold_bytes=8 * 4096 * 2 * 4 * 128 * 2,
                         flags=kv.KV_POOL_HOST_LOGIC_ONLY | kv.KV_POOL_LRU_RESIDENCY)
    return kv.kv_pool_create(cfg), kv.kv_token_bytes(cfg)


def compare(kv, pool, o, sids):
    assert kv.kv_pool_free_list(pool) == list(o.fl.contents())
    for sid in sids:
        assert kv.session_block_table(pool, sid) == o.row(sid)
        info = kv.session_info(pool, sid)
        assert info.tokens == o.s[sid].T
        assert info.state == (kv.KV_SESSION_ACTIVE if o.s[sid].state == "active"
                              else kv.KV_SESSION_PAUSED)
    st = kv.kv_pool_get_stats(pool)
    for k, v in o.stats.items():
        assert st[k] == v, k


@pytest.mark.parametrize("seed", [0, 1, 2, 3])
def test_library_matches_oracle_on_random_sequences(kv, seed):
    rnd = random.Random(seed)
    nb = 14
    pool, tb = lib_pool(kv, nb, seed)
    o = ResidencyOracle(nb, BT, seed=seed, token_bytes=tb)
    live = []
    fails = reserved = prefetched = 0
    for step in range(500):
        r = rnd.random()
        try:
            if r < 0.08 and len(live) < 6:
                if rnd.random() < 0.5:
                    T = rnd.randint(1, 90)
                    sid = kv.session_create_paused(pool, 400, T)
                    o.create_paused(sid, 400, T)
                else:
                    sid = kv.session_create(pool, 400)
                    o.create(sid, 400)
                live.append(sid)
            elif r < 0.12 and live:
                sid = rnd.choice(live)
                kv.session_destroy(pool, sid)
                o.destroy(sid)
                live.remove(sid)
            elif r < 0.14:
                s = rnd.randrange(1 << 30)
                kv.kv_pool_shuffle_free(pool, s)
                o.shuffle(s)
            elif live:
                sid = rnd.choice(live)
                state = o.s[sid].state
                if state == "paused":
                    exp = None
                    try:
                        o.resume(sid)
                    except NoHotBlocks:
                        exp = kv.KV_ERR_NO_HOT_BLOCKS
                    try:
                        kv.session_resume(pool, sid)
                        assert exp is None
                    except kv.KVError as e:
                        assert e.code == exp
                        fails += 1
                elif r < 0.6:
                    n = rnd.randint(1, 24)
                    if o.s[sid].T + n > 400:
                        continue
                    exp = None
                    try:
                        o.append(sid, n)
                    except NoHotBlocks:
                        exp = kv.KV_ERR_NO_HOT_BLOCKS
                    try:
                        kv.session_append(pool, sid, None, None, n, None)
                        assert exp is None
                    except kv.KVError as e:
                        assert e.code == exp
                        fails += 1
                elif r < 0.75:
                    o.pause(sid)
                    kv.session_pause(pool, sid, None)
                elif r < 0.87:
                    batch = [x for x in live if o.s[x].state == "active" and o.s[x].T > 0]
                    batch = rnd.sample(batch, k=min(len(batch), rnd.randint(1, 3)))
                    if not batch:
                        continue
                    exp = None
                    try:
                        o.batch(batch)
                    except NoHotBlocks:
                        exp = kv.KV_ERR_NO_HOT_BLOCKS
                    try:
                        kv.kv_pool_batch_tables(pool, batch, None, 64, None)
                        assert exp is None
                    except kv.KVError as e:
                        assert e.code == exp
                        fails += 1
                elif r < 0.92:      # the next step's blocks, ahead of it
                    act = [x for x in live if o.s[x].state == "active"]
                    if not act:
                        continue
                    nxt = rnd.sample(act, k=min(len(act), rnd.randint(1, 3)))
                    busy = rnd.sample(act, k=min(len(act), rnd.randint(0, 2)))
                    exp = None
                    try:
                        o.prefetch(nxt, busy)
                    except NoHotBlocks:
                        exp = kv.KV_ERR_NO_HOT_BLOCKS
                    try:
                        kv.kv_pool_prefetch(pool, nxt, busy)
                        assert exp is None
                        prefetched += 1
                    except kv.KVError as e:
                        assert e.code == exp
                        fails += 1
                else:               # a fused decode step's token for each member
                    batch = [x for x in live if o.s[x].state == "active" and o.s[x].T < 400]
                    batch = rnd.sample(batch, k=min(len(batch), rnd.randint(1, 3)))
                    if not batch:
                        continue
                    exp = None
                    try:
                        o.batch_reserve(batch)
                    except NoHotBlocks:
                        exp = kv.KV_ERR_NO_HOT_BLOCKS
                    try:
                        kv.kv_pool_batch_reserve(pool, batch, None, 64, None)
                        assert exp is None
                        reserved += 1
                    except kv.KVError as e:
                        assert e.code == exp
                        fails += 1
        finally:
            pass
        compare(kv, pool, o, live)
    st = kv.kv_pool_get_stats(pool)
    assert st["blocks_evicted"] > 20 and st["resume_blocks_missed"] > 0 and reserved > 10
    assert prefetched > 5 and st["blocks_prefetched"] > 0
    kv.kv_pool_destroy(pool)


def test_batch_reserve_simple_mode_equals_one_token_appends(kv):
    """Without residency, a batch reservation pops exactly the blocks that
    one-token appends in batch order would, and fails atomically."""
    def pool():
        cfg = kv.make_config(num_layers=1, num_hot_blocks=40, block_tokens=BT, alloc_seed=5,
                             max_sessions=6, max_context=4096, max_batch=8,
                             cold_bytes=6 * 4096 * 2 * 4 * 128 * 2,
                             flags=kv.KV_POOL_HOST_LOGIC_ONLY)
        p = kv.kv_pool_create(cfg)
        for _ in range(5):
            kv.session_create(p, 300)
        return p
    a, b = pool(), pool()
    rnd = random.Random(11)
    for step in range(150):
        batch = rnd.sample(range(5), k=rnd.randint(1, 5))
        if any(kv.session_info(a, s).tokens >= 300 for s in batch):
            continue
        kv.kv_pool_batch_reserve(a, batch, None, 64, None)
        for sid in batch:
            kv.session_append(b, sid, None, None, 1, None)
        assert [kv.session_block_table(a, s) for s in range(5)] == \
            [kv.session_block_table(b, s) for s in range(5)]
        assert kv.kv_pool_free_list(a) == kv.kv_pool_free_list(b)
    sa, sb = kv.kv_pool_get_stats(a), kv.kv_pool_get_stats(b)
    assert sa == sb
    # errors leave everything as it was
    before = ([kv.session_block_table(a, s) for s in range(5)], kv.kv_pool_free_list(a))
    for bad, code in (([0, 0], kv.KV_ERR_INVALID_ARG), ([0, 9], kv.KV_ERR_INVALID_ARG)):
        with pytest.raises(kv.KVError) as e:
            kv.kv_pool_batch_reserve(a, bad, None, 64, None)
        assert e.value.code == code
    assert before == ([kv.session_block_table(a, s) for s in range(5)], kv.kv_pool_free_list(a))
    kv.session_pause(a, 1, None)
    before = ([kv.session_block_table(a, s) for s in range(5)], kv.kv_pool_free_list(a),
              kv.session_info(a, 0).tokens)
    with pytest.raises(kv.KVError) as e:
        kv.kv_pool_batch_reserve(a, [0, 1], None, 64, None)   # member 0 is fine, 1 is paused
    assert e.value.code == kv.KV_ERR_BAD_STATE
    assert before == ([kv.session_block_table(a, s) for s in range(5)], kv.kv_pool_free_list(a),
                      kv.session_info(a, 0).tokens)
    kv.kv_pool_destroy(a)
    kv.kv_pool_destroy(b)


def test_prefetch_hand_worked():
    """One step ahead: the next batch's evicted blocks come back with victims
    outside both the next batch and the batch still decoding; the next
    batch is stamped as used; a prefetch that cannot find room changes
    nothing; after a prefetch the step itself fetches nothing."""
    o = ResidencyOracle(8, BT, seed=12, token_bytes=TB)
    for sid in range(4):
        o.create(sid, 1000)
        o.append(sid, 32)      # A, B, C, D: two full blocks each, times 1..4; pool full
    o.pause(2)                 # C idles
    o.batch([1, 3])            # B and D decode: time 5
    a_row, c_row = o.row(0), o.row(2)
    o.append(1, 16)            # B grows: the LRU block is A's block 0 (time 1)
    assert o.row(0) == [-1, a_row[1]]
    assert o.stats["bytes_packed"] == 16 * TB
    b_new = o.row(1)[2]
    assert b_new == a_row[0]
    o.prefetch([0], busy=[1])  # A is next; B still decodes: victim from C (time 3) or D (5)
    assert o.row(2) == [-1, c_row[1]]                  # C's block 0, the least recent
    assert o.row(0) == [c_row[0], a_row[1]]
    assert o.stats["blocks_prefetched"] == 1 and o.stats["prefetches"] == 1
    assert o.stats["bytes_packed"] == 32 * TB          # + C's 16 tokens, written once
    assert o.stats["bytes_unpacked"] == 16 * TB        # A's block back
    assert o.s[0].time > o.s[1].time                   # A stamped after B's append
    o.batch_reserve([0])       # A's tail is full: one new block (victim C's block 1)
    assert o.stats["batch_blocks_fetched"] == 0
    assert o.row(2) == [-1, -1]
    o.append(3, 16)            # D grows: the LRU outside D is B (its append came before A's stamps)
    assert o.row(1)[0] == -1
    before = ([o.row(s) for s in range(4)], list(o.fl.contents()), dict(o.stats))
    with pytest.raises(NoHotBlocks):
        o.prefetch([1], busy=[0, 3])       # C holds no hot block: no victim outside A, B, D
    assert before == ([o.row(s) for s in range(4)], list(o.fl.contents()), dict(o.stats))
    o.resume(2)
    o.prefetch([2], busy=[0])  # nothing missing: only the stamp
    assert o.stats["blocks_prefetched"] == 1 and o.stats["prefetches"] == 2


def test_prefetch_then_step_fetches_nothing_without_interference():
    """Prefetching step k+1's batch during step k leaves step k+1 nothing to
    fetch when no other allocation comes in between; the blocks it reads
    are those the prefetch placed."""
    o = ResidencyOracle(24, BT, seed=14, token_bytes=TB)
    rnd = random.Random(8)
    n = 8
    for sid in range(n):
        o.create(sid, 10_000)
        o.append(sid, 32)      # 8 x 2 blocks: 16 of 24
    cur = [0, 1, 2]
    done = 0
    for step in range(80):
        o.batch_reserve(cur)
        nxt = sorted(rnd.sample(range(n), k=3))
        for sid in nxt:        # a paused member of the next batch resumes first
            if o.s[sid].state == "paused":
                o.resume(sid)
        for sid in range(n):   # sessions outside both batches idle
            if sid not in cur and sid not in nxt and o.s[sid].state == "active":
                o.pause(sid)
        try:
            o.prefetch(nxt, busy=cur)
        except NoHotBlocks:
            cur = nxt
            continue
        fetched = o.stats["batch_blocks_fetched"]
        rows = {s: o.row(s) for s in nxt}
        assert all(x >= 0 for s in nxt for x in rows[s])
        o.batch_reserve(nxt)
        assert o.stats["batch_blocks_fetched"] == fetched
        assert all(o.row(s)[:len(rows[s])] == rows[s] for s in nxt)
        done += 1
        cur = nxt
    assert done > 40
    assert o.stats["blocks_evicted"] > 0 and o.stats["blocks_prefetched"] > 0

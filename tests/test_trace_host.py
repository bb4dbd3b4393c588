"""The agentic trace's schedule on a host-logic-only pool, without a GPU.

The schedule is a function of the seeded trace alone (no timing enters it),
so its rules are checked here by stepping the driver on the CPU: at most N_a
sessions decode or wait to join, a resumed session joins the batch
admit_lead steps later, every decode burst lasts exactly its drawn length,
no session is in two places at once, the pool's token counts follow the
driver's, and no token reaches the cold tier twice (write-on-evict).
"""
import dataclasses
import math

import numpy as np
import pytest


@pytest.fixture(scope="module")
def tr():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import kvtier, trace
    return kvtier, trace


def small_cfg(trace, **kw):
    base = dict(sessions=12, t0_min=40, t0_max=500, burst_mean=12.0, pause_mean_s=0.6,
                append_median=48.0, append_max=400, active_cap=4, steps=400, dt_s=0.075,
                layers=2, seed=5)
    base.update(kw)
    return trace.TraceConfig(**base)


def host_pool(kv, cfg, trace_list, lru_blocks=None):
    tok_bytes = cfg.layers * 2 * cfg.num_kv_heads * 128 * 2
    flags = kv.KV_POOL_HOST_LOGIC_ONLY | (kv.KV_POOL_LRU_RESIDENCY if lru_blocks else 0)
    c = kv.make_config(num_layers=cfg.layers, num_q_heads=cfg.num_q_heads,
                       num_kv_heads=cfg.num_kv_heads, block_tokens=cfg.block_tokens,
                       max_sessions=cfg.sessions, max_batch=cfg.active_cap, max_context=1 << 16,
                       num_hot_blocks=lru_blocks or 100000,
                       cold_bytes=cfg.sessions * (1 << 16) * tok_bytes, flags=flags)
    pool = kv.kv_pool_create(c)
    for t in trace_list:
        kv.session_create_paused(pool, 1 << 16, t.t0)
    return pool, tok_bytes


def test_generate_is_seeded_and_follows_its_distributions(tr):
    _, trace = tr
    cfg = trace.TraceConfig(seed=3)
    a, b = trace.generate(cfg), trace.generate(cfg)
    assert [dataclasses.asdict(x) for x in a] == [dataclasses.asdict(x) for x in b]
    assert trace.generate(dataclasses.replace(cfg, seed=4))[0].t0 != a[0].t0 or \
        trace.generate(dataclasses.replace(cfg, seed=4))[0].bursts != a[0].bursts
    assert len(a) == cfg.sessions
    assert all(cfg.t0_min <= x.t0 <= cfg.t0_max for x in a)
    assert all(0.0 <= x.first_ready_s <= cfg.pause_mean_s for x in a)
    bursts = np.concatenate([x.bursts for x in a])
    pauses = np.concatenate([x.pauses for x in a])
    appends = np.concatenate([x.appends for x in a])
    assert bursts.min() >= 1 and abs(bursts.mean() / cfg.burst_mean - 1) < 0.1
    assert pauses.min() >= 0 and abs(pauses.mean() / cfg.pause_mean_s - 1) < 0.1
    assert appends.min() >= 1 and appends.max() <= cfg.append_max
    assert abs(np.median(appends) / cfg.append_median - 1) < 0.1
    # lognormal: the log of the uncapped draws has the configured spread
    below_cap = appends[appends < cfg.append_max]
    assert abs(np.std(np.log(below_cap)) / cfg.append_sigma - 1) < 0.15


@pytest.mark.parametrize("lead,fused", [(1, True), (3, True), (1, False)])
def test_schedule_rules_hold_every_step(tr, lead, fused):
    kv, trace = tr
    cfg = small_cfg(trace, admit_lead=lead, fused_append=fused)
    tl = trace.generate(cfg)
    pool, tok_bytes = host_pool(kv, cfg, tl)
    d = trace.TraceDriver(cfg, pool, tl, gpu=False)
    decoded = {}                      # (session, turn) -> decode steps in that turn
    first_decode = {}                 # (session, turn) -> step of its first decode
    admitted = {}                     # (session, turn) -> step of its resume
    expect_tokens = [t.t0 for t in tl]
    try:
        for k in range(cfg.steps):
            turn_before = list(d.turn)
            joining_before = {i for _, i in d.joining}
            resumes_before = d.counts["resumes"]
            d.step(k)
            new = [i for _, i in d.joining if i not in joining_before]
            assert d.counts["resumes"] - resumes_before == len(new)
            for i in new:
                admitted[(i, d.turn[i])] = k
                expect_tokens[i] += tl[i].appends[d.turn[i]]
            members = sorted(d.active)
            joining = [i for _, i in d.joining]
            queued = [i for _, i in d.queue]
            # N_a bounds the batch and the sessions about to join it
            assert len(members) + len(joining) <= cfg.active_cap
            # a session is decoding, joining or paused in the queue: one of them
            placed = members + joining + queued
            assert sorted(placed) == list(range(cfg.sessions))
            for i in members:
                key = (i, d.turn[i])
                assert d.turn[i] == turn_before[i]      # a decoding session's turn holds
                decoded[key] = decoded.get(key, 0) + 1
                first_decode.setdefault(key, k)
                expect_tokens[i] += 1
            for i in range(cfg.sessions):
                info = kv.session_info(pool, d.sids[i])
                assert info.tokens == d.tokens[i] == expect_tokens[i]
                want = kv.KV_SESSION_PAUSED if i in queued else kv.KV_SESSION_ACTIVE
                assert info.state == want
                if want == kv.KV_SESSION_PAUSED:
                    assert info.cold_valid == info.tokens   # a pause packed every new token
        # simple mode packs each token once: the cold writes are exactly what
        # the images gained beyond the initial contexts
        gained = sum(kv.session_info(pool, d.sids[i]).cold_valid - tl[i].t0
                     for i in range(cfg.sessions))
        assert kv.kv_pool_get_stats(pool)["bytes_packed"] == gained * tok_bytes > 0
    finally:
        kv.kv_pool_destroy(pool)
    finished = [(i, t) for (i, t) in decoded if t < d.turn[i]]
    assert len(finished) > 3 * cfg.sessions          # many complete turns were exercised
    for (i, t) in finished:
        assert decoded[(i, t)] == tl[i].bursts[t]   # a burst lasts its drawn length
        assert first_decode[(i, t)] - admitted[(i, t)] == max(1, lead)


def test_dry_run_is_deterministic(tr):
    _, trace = tr
    cfg = small_cfg(trace)
    tl = trace.generate(cfg)
    a, b = trace.plan(cfg, tl), trace.plan(cfg, tl)
    assert a["counts"] == b["counts"] and a["stats"] == b["stats"] and a["caps"] == b["caps"]
    assert a["counts"]["resumes"] > cfg.sessions and a["counts"]["pauses"] > cfg.sessions


@pytest.mark.parametrize("mode", ["simple", "lru"])
def test_no_token_written_to_the_cold_tier_twice(tr, mode):
    """Write-on-evict: over the whole run the cold tier receives at most the
    tokens generated after each session's initial context (which starts in
    its image), once each."""
    kv, trace = tr
    cfg = small_cfg(trace, lru=mode == "lru")
    tl = trace.generate(cfg)
    hot = None
    if mode == "lru":
        peak = trace.plan(dataclasses.replace(cfg, lru=False), tl)["peak_blocks"]
        hot = int(math.ceil(1.2 * peak))
    r = trace.plan(cfg, tl, hot_blocks=hot)
    tok_bytes = cfg.layers * 2 * cfg.num_kv_heads * 128 * 2
    grown = sum(cap - t.t0 for cap, t in zip(r["caps"], tl))
    assert 0 < r["stats"]["bytes_packed"] <= grown * tok_bytes
    assert r["stats"]["bytes_packed"] % tok_bytes == 0
    if mode == "simple":
        # every pause packs the session's new tokens: nothing generated and then
        # paused is left out
        assert r["stats"]["pauses"] == r["counts"]["pauses"]
    else:
        s = r["stats"]
        assert s["resume_blocks_hit"] + s["resume_blocks_missed"] > 0
        assert s["blocks_evicted"] > 0                # the pool was under pressure


def test_lru_trace_with_prefetch_matches_the_residency_oracle(tr, monkeypatch):
    """The residency-mode schedule with the one-step-ahead prefetch, each pool
    call mirrored on the residency oracle: block tables, free list and
    counters equal after every step; the prefetch takes fetches out of the
    steps themselves without changing the schedule."""
    import oracle
    from oracle.residency import NoHotBlocks, ResidencyOracle
    kv, trace = tr
    base = small_cfg(trace, lru=True, steps=300)
    tl = trace.generate(base)
    peak = trace.plan(dataclasses.replace(base, lru=False), tl)["peak_blocks"]
    nb = int(math.ceil(1.05 * peak))
    tok_bytes = base.layers * 2 * base.num_kv_heads * 128 * 2
    pool, _ = host_pool(kv, base, tl, lru_blocks=nb)
    o = ResidencyOracle(nb, base.block_tokens, seed=0, token_bytes=tok_bytes)
    for i, t in enumerate(tl):
        o.create_paused(i, 1 << 16, t.t0)

    def mirror(name, fn):
        real = getattr(kv, name)

        def call(*a, **k):
            err = None
            try:
                fn(*a, **k)
            except NoHotBlocks:
                err = kv.KV_ERR_NO_HOT_BLOCKS
            try:
                real(*a, **k)
            except kv.KVError as e:
                assert e.code == err
                raise
            assert err is None
        monkeypatch.setattr(kv, name, call)

    mirror("session_resume", lambda p, sid, st=None: o.resume(sid))
    mirror("session_pause", lambda p, sid, st=None: o.pause(sid))
    mirror("session_append", lambda p, sid, k, v, n, st=None: o.append(sid, n))
    mirror("kv_pool_batch_reserve", lambda p, sids, *a: o.batch_reserve(list(sids)))
    mirror("kv_pool_prefetch", lambda p, sids, busy=(), st=None: o.prefetch(list(sids), list(busy)))
    d = trace.TraceDriver(base, pool, tl, gpu=False)
    try:
        for k in range(base.steps):
            d.step(k)
            assert kv.kv_pool_free_list(pool) == list(o.fl.contents())
            for i in range(base.sessions):
                assert kv.session_block_table(pool, i) == o.row(i)
        st = kv.kv_pool_get_stats(pool)
        for key, v in o.stats.items():
            assert st[key] == v, key
    finally:
        kv.kv_pool_destroy(pool)
    assert st["prefetches"] > 0 and st["blocks_evicted"] > 0
    monkeypatch.undo()
    # the same schedule without the prefetch: the steps fetch more themselves
    off = trace.plan(dataclasses.replace(base, prefetch=False), tl, hot_blocks=nb)
    on = trace.plan(base, tl, hot_blocks=nb)
    assert on["counts"]["resumes"] == off["counts"]["resumes"]
    assert on["counts"]["decode_tokens"] == off["counts"]["decode_tokens"]
    assert on["stats"]["batch_blocks_fetched"] < off["stats"]["batch_blocks_fetched"]
    assert off["stats"]["blocks_prefetched"] == 0

"""The agentic trace driver end to end on a small configuration.

Sessions cycle through resume -> turn append -> decode burst -> pause many
times on two streams. At sampled steps the decode outputs are checked against
the oracle (values regenerated on the host from their logical positions),
and at the end every cold image must hold exactly the session's logical KV
for the tokens it has packed.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

TOL = 1e-2


@pytest.mark.parametrize("lead", [1, 2])
def test_small_trace_parity(cuda_dev, lead):
    """lead: steps between a session's resume and its first decode (2: the
    admitted session waits a step longer, its resume further ahead)."""
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import Pool, kvtier
    from paper_2609_25782_gb300 import trace as tr

    cfg = tr.TraceConfig(sessions=6, t0_min=100, t0_max=700, burst_mean=8.0, pause_mean_s=0.6,
                         append_median=40.0, append_sigma=1.0, append_max=300, active_cap=2,
                         steps=150, dt_s=0.1, layers=2, seed=5, admit_lead=lead)
    trace = tr.generate(cfg)
    plan = tr.plan(cfg, trace)
    assert plan["counts"]["pauses"] >= 10
    L, Hkv, Hq, D, bt = cfg.layers, cfg.num_kv_heads, cfg.num_q_heads, 128, cfg.block_tokens
    nb = plan["peak_blocks"] + 40
    pool = Pool(num_layers=L, num_hot_blocks=nb, cold_bytes=plan["cold_bytes"] + 4096,
                max_sessions=cfg.sessions, max_batch=cfg.active_cap,
                max_context=plan["max_context"], alloc_seed=9)
    for i, t in enumerate(trace):
        sid = pool.session_create_paused(plan["caps"][i], t.t0)
        assert sid == i
        synth.fill_image_torch(pool.image(sid), cfg.seed, sid, L, Hkv, D, t.t0)

    def kv_source(sid, t0, t1):
        k, v = synth.kv_logical_torch(cfg.seed, sid, range(L), Hkv, D, t0, t1, cuda_dev)
        return k.permute(0, 2, 1, 3).contiguous(), v.permute(0, 2, 1, 3).contiguous()

    q = synth.queries_torch(cfg.seed, range(cfg.active_cap), range(L), Hq, D, cuda_dev)
    out = torch.empty(L, cfg.active_cap, Hq, D, dtype=torch.float32, device=cuda_dev)
    max_blocks = -(-plan["max_context"] // bt)
    tables = torch.empty(cfg.active_cap, max_blocks, dtype=torch.int32, device=cuda_dev)
    seq_lens = torch.empty(cfg.active_cap, dtype=torch.int32, device=cuda_dev)
    dstream, mstream = torch.cuda.Stream(), torch.cuda.Stream()
    torch.cuda.synchronize()     # inputs made on the default stream are complete
    checked = []

    def on_step(k, members):
        if k % 13 != 5:
            return
        torch.cuda.synchronize()
        got = out[:, :len(members)].double().cpu().numpy()
        lens = [int(kvtier.session_info(pool.handle, m).tokens) for m in members]
        tab = np.full((len(members), max_blocks), -1, dtype=np.int32)
        for r, m in enumerate(members):
            row = pool.session_block_table(m)
            tab[r, :len(row)] = row
        hot = synth.hot_pool_np(cfg.seed, members, lens, tab, nb, L, Hkv, D, bt)
        qh = q[:, :len(members)].contiguous().cpu().view(torch.int16).numpy().view(np.uint16)
        ref = oracle.paged_decode(hot, qh, tab, lens, 1 / math.sqrt(D), Hq)
        err = np.max(np.abs(got - ref) / np.maximum(1.0, np.abs(ref)))
        assert err <= TOL, f"step {k}: scaled error {err}"
        checked.append(k)

    d = tr.TraceDriver(cfg, pool.handle, trace, gpu=True, kv_source=kv_source, q=q, out=out,
                       decode_stream=dstream, mig_stream=mstream, tables=tables,
                       seq_lens=seq_lens, max_blocks=max_blocks, on_step=on_step)
    d.run()
    torch.cuda.synchronize()
    assert len(checked) >= 5
    assert d.counts == plan["counts"]          # same schedule as the dry run
    assert pool.check_device() == 0
    st = pool.stats()
    assert st["pauses"] == plan["counts"]["pauses"] and st["resumes"] == plan["counts"]["resumes"]
    # every image holds the session's logical KV for its packed prefix
    for i in range(cfg.sessions):
        info = kvtier.session_info(pool.handle, i)
        n = int(info.cold_valid)
        img = pool.image(i)[:, :, :, :n].contiguous().cpu().view(torch.int16).numpy().view(np.uint16)
        k, v = synth.session_kv_np(cfg.seed, i, range(L), Hkv, D, n)
        assert np.array_equal(img[:, 0], k) and np.array_equal(img[:, 1], v)
    pool.close()


def test_full_trace_sampled_parity(cuda_dev):
    """The benchmark's trace (48 sessions, N_a = 16, 2 000 steps, 48 layers),
    with appended tokens taking their logical values so the oracle can
    regenerate any session: at sampled steps two members of the batch are
    checked on one layer each; at the end every image prefix is checked."""
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import Pool, kvtier
    from paper_2609_25782_gb300 import trace as tr

    cfg = tr.TraceConfig(seed=0)
    L, Hkv, Hq, D, bt = cfg.layers, cfg.num_kv_heads, cfg.num_q_heads, 128, cfg.block_tokens
    trace = tr.generate(cfg)
    plan = tr.plan(cfg, trace)
    nb = plan["peak_blocks"] + 256
    pool = Pool(num_layers=L, num_hot_blocks=nb, cold_bytes=plan["cold_bytes"] + 4096,
                max_sessions=cfg.sessions, max_batch=cfg.active_cap,
                max_context=plan["max_context"], alloc_seed=cfg.seed)
    for i, t in enumerate(trace):
        sid = pool.session_create_paused(plan["caps"][i], t.t0)
        synth.fill_image_torch(pool.image(sid), cfg.seed, sid, L, Hkv, D, t.t0)

    def kv_source(sid, t0, t1):
        k, v = synth.kv_logical_torch(cfg.seed, sid, range(L), Hkv, D, t0, t1, cuda_dev)
        return k.permute(0, 2, 1, 3).contiguous(), v.permute(0, 2, 1, 3).contiguous()

    q = synth.queries_torch(cfg.seed, range(cfg.active_cap), range(L), Hq, D, cuda_dev)
    out = torch.empty(L, cfg.active_cap, Hq, D, dtype=torch.float32, device=cuda_dev)
    max_blocks = -(-plan["max_context"] // bt)
    tables = torch.empty(cfg.active_cap, max_blocks, dtype=torch.int32, device=cuda_dev)
    seq_lens = torch.empty(cfg.active_cap, dtype=torch.int32, device=cuda_dev)
    torch.cuda.synchronize()     # inputs made on the default stream are complete
    rng = np.random.default_rng(1)
    sample_steps = {400, 1200, 1999}
    checked = []

    def on_step(k, members):
        if k not in sample_steps:
            return
        torch.cuda.synchronize()
        for r in rng.choice(len(members), size=2, replace=False):
            m = members[int(r)]
            l = int(rng.integers(0, L))
            T = int(kvtier.session_info(pool.handle, m).tokens)
            kk, vv = synth.session_kv_np(cfg.seed, m, [l], Hkv, D, T)
            nblk = -(-T // bt)
            host = np.full((nblk, 1, 2, Hkv, bt, D), synth.BF16_NAN, dtype=np.uint16)
            for j in range(nblk):
                n = min(bt, T - j * bt)
                host[j, 0, 0, :, :n] = kk[0, :, j * bt:j * bt + n]
                host[j, 0, 1, :, :n] = vv[0, :, j * bt:j * bt + n]
            qh = q[l:l + 1, int(r):int(r) + 1].contiguous().cpu().view(torch.int16).numpy().view(np.uint16)
            ref = oracle.paged_decode(host, qh, np.arange(nblk, dtype=np.int32)[None], [T],
                                      1 / math.sqrt(D), Hq)
            got = out[l:l + 1, int(r):int(r) + 1].double().cpu().numpy()
            err = np.max(np.abs(got - ref) / np.maximum(1.0, np.abs(ref)))
            assert err <= TOL, (k, m, l, err)
            checked.append((k, m))

    d = tr.TraceDriver(cfg, pool.handle, trace, gpu=True, kv_source=kv_source, q=q, out=out,
                       decode_stream=torch.cuda.Stream(priority=-1), mig_stream=torch.cuda.Stream(),
                       tables=tables, seq_lens=seq_lens, max_blocks=max_blocks, on_step=on_step)
    d.run()
    torch.cuda.synchronize()
    assert len(checked) == 6
    assert d.counts == plan["counts"]
    assert pool.check_device() == 0
    # every image holds its session's logical KV for the packed prefix (sampled layers)
    for i in range(cfg.sessions):
        n = int(kvtier.session_info(pool.handle, i).cold_valid)
        l = i % L
        img = pool.image(i)[l, :, :, :n].contiguous().cpu().view(torch.int16).numpy().view(np.uint16)
        kk, vv = synth.session_kv_np(cfg.seed, i, [l], Hkv, D, n)
        assert np.array_equal(img[0], kk[0]) and np.array_equal(img[1], vv[0])
    pool.close()


@pytest.mark.parametrize("prefetch,lead", [(True, 1), (False, 1), (True, 2)])
def test_small_trace_residency_under_pressure(cuda_dev, prefetch, lead):
    """The small trace in residency mode (LRU, write-on-evict) with a hot pool
    of exactly the simple mode's peak: paused sessions' blocks are evicted and
    fetched back, step tokens go through the fused decode. At sampled steps
    the decode must match the oracle over the members' logical KV (so every
    block fetched back holds the right bytes), and the run's counters must
    equal the residency dry run's. Without the one-step-ahead prefetch some
    blocks are fetched inside the steps (victims of admissions on the
    migration stream), which exercises fetches after evictions made on the
    other stream."""
    import dataclasses

    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import Pool, kvtier
    from paper_2609_25782_gb300 import trace as tr

    base = tr.TraceConfig(sessions=6, t0_min=100, t0_max=700, burst_mean=8.0, pause_mean_s=0.6,
                          append_median=40.0, append_sigma=1.0, append_max=300, active_cap=2,
                          steps=150, dt_s=0.1, layers=2, seed=5, admit_lead=lead)
    trace = tr.generate(base)
    simple = tr.plan(base, trace)
    cfg = dataclasses.replace(base, lru=True, prefetch=prefetch)
    nb = simple["peak_blocks"]
    dry = tr.plan(cfg, trace, hot_blocks=nb)["stats"]
    assert dry["blocks_evicted"] > 0 and dry["resume_blocks_missed"] > 0
    assert (dry["prefetches"] > 0) == prefetch
    if not prefetch:
        assert dry["batch_blocks_fetched"] > 0
    L, Hkv, Hq, D, bt = cfg.layers, cfg.num_kv_heads, cfg.num_q_heads, 128, cfg.block_tokens
    pool = Pool(num_layers=L, num_hot_blocks=nb, cold_bytes=simple["cold_bytes"] + 4096,
                max_sessions=cfg.sessions, max_batch=cfg.active_cap,
                max_context=simple["max_context"], alloc_seed=cfg.seed, lru_residency=True)
    for i, t in enumerate(trace):
        sid = pool.session_create_paused(simple["caps"][i], t.t0)
        synth.fill_image_torch(pool.image(sid), cfg.seed, sid, L, Hkv, D, t.t0)

    def kv_source(sid, t0, t1):
        k, v = synth.kv_logical_torch(cfg.seed, sid, range(L), Hkv, D, t0, t1, cuda_dev)
        return k.permute(0, 2, 1, 3).contiguous(), v.permute(0, 2, 1, 3).contiguous()

    q = synth.queries_torch(cfg.seed, range(cfg.active_cap), range(L), Hq, D, cuda_dev)
    out = torch.empty(L, cfg.active_cap, Hq, D, dtype=torch.float32, device=cuda_dev)
    max_blocks = -(-simple["max_context"] // bt)
    tables = torch.empty(cfg.active_cap, max_blocks, dtype=torch.int32, device=cuda_dev)
    seq_lens = torch.empty(cfg.active_cap, dtype=torch.int32, device=cuda_dev)
    torch.cuda.synchronize()
    checked = []

    def on_step(k, members):
        if k % 7 != 3:
            return
        torch.cuda.synchronize()
        got = out[:, :len(members)].double().cpu().numpy()
        lens = [int(kvtier.session_info(pool.handle, m).tokens) for m in members]
        tab = np.full((len(members), max_blocks), -1, dtype=np.int32)
        for r, m in enumerate(members):
            row = pool.session_block_table(m)
            assert min(row) >= 0                   # the batch's blocks are all hot
            tab[r, :len(row)] = row
        hot = synth.hot_pool_np(cfg.seed, members, lens, tab, nb, L, Hkv, D, bt)
        qh = q[:, :len(members)].contiguous().cpu().view(torch.int16).numpy().view(np.uint16)
        ref = oracle.paged_decode(hot, qh, tab, lens, 1 / math.sqrt(D), Hq)
        err = np.max(np.abs(got - ref) / np.maximum(1.0, np.abs(ref)))
        assert err <= TOL, f"step {k}: scaled error {err}"
        checked.append(k)

    d = tr.TraceDriver(cfg, pool.handle, trace, gpu=True, kv_source=kv_source, q=q, out=out,
                       decode_stream=torch.cuda.Stream(), mig_stream=torch.cuda.Stream(),
                       tables=tables, seq_lens=seq_lens, max_blocks=max_blocks, on_step=on_step)
    d.run()
    torch.cuda.synchronize()
    assert len(checked) >= 10
    assert pool.check_device() == 0
    st = pool.stats()
    for key in ("bytes_packed", "bytes_unpacked", "blocks_evicted", "resume_blocks_hit",
                "resume_blocks_missed", "resumes", "pauses", "batch_blocks_fetched",
                "blocks_prefetched", "prefetches"):
        assert st[key] == dry[key], key
    pool.close()


def test_trace_graph_replay_bit_identical_to_direct_calls(cuda_dev):
    """The driver replays each step's per-layer calls from a CUDA graph cached
    per (batch size, table width rounded up to 1 024 tokens), the step's new
    K/V staged in a fixed buffer. On the same schedule the outputs of every
    step must be bit-identical to launching the calls directly (the wider
    tables change the launch shape only)."""
    import dataclasses

    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import Pool
    from paper_2609_25782_gb300 import trace as tr

    base = tr.TraceConfig(sessions=6, t0_min=100, t0_max=1500, burst_mean=8.0, pause_mean_s=0.6,
                          append_median=40.0, append_sigma=1.0, append_max=300, active_cap=3,
                          steps=80, dt_s=0.1, layers=2, seed=7)
    trace = tr.generate(base)
    plan = tr.plan(base, trace)
    L, Hkv, Hq, D, bt = base.layers, base.num_kv_heads, base.num_q_heads, 128, base.block_tokens
    outs = {}
    for graphs in (True, False):
        cfg = dataclasses.replace(base, graphs=graphs)
        pool = Pool(num_layers=L, num_hot_blocks=plan["peak_blocks"] + 40,
                    cold_bytes=plan["cold_bytes"] + 4096, max_sessions=cfg.sessions,
                    max_batch=cfg.active_cap, max_context=plan["max_context"], alloc_seed=3)
        for i, t in enumerate(trace):
            sid = pool.session_create_paused(plan["caps"][i], t.t0)
            synth.fill_image_torch(pool.image(sid), cfg.seed, sid, L, Hkv, D, t.t0)

        def kv_source(sid, t0, t1):
            k, v = synth.kv_logical_torch(cfg.seed, sid, range(L), Hkv, D, t0, t1, cuda_dev)
            return k.permute(0, 2, 1, 3).contiguous(), v.permute(0, 2, 1, 3).contiguous()

        q = synth.queries_torch(cfg.seed, range(cfg.active_cap), range(L), Hq, D, cuda_dev)
        out = torch.empty(L, cfg.active_cap, Hq, D, dtype=torch.float32, device=cuda_dev)
        max_blocks = -(-plan["max_context"] // bt)
        tables = torch.empty(cfg.active_cap, max_blocks, dtype=torch.int32, device=cuda_dev)
        seq_lens = torch.empty(cfg.active_cap, dtype=torch.int32, device=cuda_dev)
        torch.cuda.synchronize()
        got = {}

        def on_step(k, members, out=out, got=got):
            torch.cuda.synchronize()
            got[k] = (tuple(members), out[:, :len(members)].clone())

        d = tr.TraceDriver(cfg, pool.handle, trace, gpu=True, kv_source=kv_source, q=q, out=out,
                           decode_stream=torch.cuda.Stream(), mig_stream=torch.cuda.Stream(),
                           tables=tables, seq_lens=seq_lens, max_blocks=max_blocks,
                           on_step=on_step)
        d.run()
        torch.cuda.synchronize()
        assert pool.check_device() == 0
        if graphs:
            assert 0 < len(d.graphs) < len(got)      # shapes repeat: graphs are replayed
        outs[graphs] = got
        pool.close()
    assert outs[True].keys() == outs[False].keys() and len(outs[True]) > 40
    for k in outs[True]:
        mg, og = outs[True][k]
        md, od = outs[False][k]
        assert mg == md
        assert torch.equal(og.view(torch.int32), od.view(torch.int32)), k

"""Benchmark of the hot/cold KV hot path on GB300.

Headline workload: one decode-attention step of 32 active sessions over all
48 layers of a Qwen3-Coder-30B-A3B-shaped KV cache (4 KV heads, head_dim 128,
32 query heads, 16-token blocks, 96 KiB of KV per token), contexts uniform in
[8K, 32K] tokens (about 64 GB of hot KV at seeded random physical blocks).
A step is 48 per-layer decode_attention calls (split-KV kernel + combine).

  value     decode-attention KV GB/s, inputs resident in HBM
  e2e       the same metric with, every step, Q and the batch tables copied
            host->device from pinned memory and the outputs copied back
  roofline  the decode kernels against the measured HBM copy bandwidth
  secondary resume-unpack and pause-pack of 8 x 32K-token sessions

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
Under torchrun each rank runs an independent replica on its own sessions
(sessions shard across GPUs with no exchange); value sums over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

L, HQ, HKV, D, BT = 48, 32, 4, 128, 16
B2, TMIN2, TMAX2 = 32, 8192, 32768
TOKEN_BYTES = L * 2 * HKV * D * 2
PEAKS = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_HBM = 6800.0


def hbm_peak():
    try:
        with open(PEAKS) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM, "fallback"


TRAFFIC_RECORD = "decode_split_kernel_traffic_2L_B32_8K-32K.txt"


def recorded_traffic():
    """DRAM bytes per launch of the decode split kernel from the committed ncu
    capture, or None when the kernel source changed since it was taken."""
    try:
        rec, shas = {}, {}
        with open(os.path.join(ROOT, "profiles", TRAFFIC_RECORD)) as f:
            for line in f:
                if line.startswith("#") or ": " not in line:
                    continue
                key, val = line.rstrip("\n").split(": ", 1)
                if key.startswith("sha256 "):
                    shas[key[len("sha256 "):]] = val
                else:
                    rec[key] = val
        if not shas:
            return None
        for path, sha in shas.items():
            with open(os.path.join(ROOT, path), "rb") as f:
                if hashlib.sha256(f.read()).hexdigest() != sha:
                    return None
        return int(rec["dram_bytes_per_launch"])
    except Exception:
        return None


def replica_seed(seed: int, rank: int) -> int:
    """Each rank serves its own sessions: disjoint seeded draws per rank."""
    return seed + 1000 * rank


def reduce_over_ranks(total_ms: float, e2e_ms: float, kv_bytes: float, device="cpu"):
    """Max of the timed regions and sum of the bytes over all ranks (the
    whole-job value divides the summed bytes by the slowest rank's time)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([total_ms, e2e_ms, kv_bytes], dtype=torch.float64, device=device)
    mx, sm = t.clone(), t.clone()
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    dist.all_reduce(sm, op=dist.ReduceOp.SUM)
    return float(mx[0]), float(mx[1]), float(sm[2])


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during a region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        time.sleep(0.5)   # let the sampler start before the timed region
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in getattr(self, "lines", []):
            p = [x.strip() for x in line.split(",")]
            if len(p) < 9:
                continue
            try:
                sm.append(float(p[1]))
                mx.append(float(p[2]))
            except ValueError:
                continue
            for n, v in zip(names, p[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------- workloads

def decode_workload(args, rank: int):
    import torch
    import synth
    from paper_2609_25782_gb300 import Pool
    dev = torch.device("cuda", torch.cuda.current_device())
    s = replica_seed(args.seed, rank)
    nl, B = args.layers, args.batch
    lens = synth.session_lengths(s, B, args.tmin, args.tmax, BT)
    nb = int(sum(-(-int(t) // BT) for t in lens)) + 64
    pool = Pool(num_layers=nl, num_hot_blocks=nb, cold_bytes=256, max_sessions=B,
                max_batch=nl * B, max_context=args.tmax, device=dev.index)
    tables = synth.random_block_tables(s, lens, BT, nb, max_blocks=-(-args.tmax // BT))
    sess = list(range(B))
    synth.fill_hot_pool_torch(pool.hot, s, sess, lens, tables, nl, HKV, D, BT, chunk_blocks=48)
    q = synth.queries_torch(s, sess, range(nl), HQ, D, dev).contiguous()
    torch.cuda.synchronize()
    return pool, lens, tables, q


def run_decode(args, ws, rank):
    import torch
    import torch.distributed as dist
    dev = torch.device("cuda", torch.cuda.current_device())
    t_setup = time.time()
    pool, lens, tables_h, q = decode_workload(args, rank)
    L, B2 = args.layers, args.batch
    setup_s = time.time() - t_setup
    tables = torch.as_tensor(tables_h, device=dev)
    lens_d = torch.as_tensor(lens.astype(np.int32), device=dev)
    max_blocks = tables.shape[1]
    out = torch.empty(L, B2, HQ, D, dtype=torch.float32, device=dev)
    scale = 1 / math.sqrt(D)
    stream = torch.cuda.Stream(device=dev)
    kv_bytes = int(lens.sum()) * L * 2 * HKV * D * 2   # per step (all layers)
    q_bytes = B2 * HQ * D * 2
    out_bytes = B2 * HQ * D * 4
    tab_bytes = int(sum(-(-int(t) // BT) for t in lens)) * 4
    launch_alg_bytes = kv_bytes / L + q_bytes + out_bytes + tab_bytes   # one layer's call

    # Layer l > 0 follows layer l-1's call on the stream, which writes only
    # `out`, so it may overlap its start with that call's end.
    ov = not args.no_overlap

    def step_calls(st):
        for l in range(L):
            pool.decode_attention(l, q[l], tables, lens_d, B2, max_blocks, scale, out[l], st,
                                  overlap_previous=ov and l > 0)

    graph = capture_graph(step_calls, stream) if args.graph else None

    def step():
        if graph is not None:
            with torch.cuda.stream(stream):
                graph.replay()
        else:
            step_calls(stream)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    torch.cuda.synchronize()
    flags = pool.check_device()
    if flags:
        raise RuntimeError(f"device check flags {flags} after warm-up")

    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    if ws > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(dev.index) as clk:
        t0.record(stream)
        for k in range(args.steps):
            step()
        t1.record(stream)
        torch.cuda.synchronize()
    if ws > 1:
        dist.barrier()
    total_ms = t0.elapsed_time(t1)
    launch_ms = total_ms / (args.steps * L)     # average decode call over the timed region

    # End to end through the C ABI with host buffers: every step copies its
    # Q, block tables and seq_lens from pinned host memory and reads its
    # outputs back. Inputs and outputs rotate through NB buffers so that step
    # k+1's upload and step k's read-back run on a copy stream while step k
    # decodes, and the host may issue up to NB steps (about 50 ms of GPU work,
    # about 500 launches: well inside the CUDA launch queue) before it waits
    # for a read-back, which a host stall of tens of ms then does not drain.
    NB = 5
    cs = torch.cuda.Stream(device=dev)
    q_h = torch.empty(q.shape, dtype=q.dtype).pin_memory()
    q_h.copy_(q.cpu())
    tab_h = torch.as_tensor(tables_h).pin_memory()
    len_h = torch.as_tensor(lens.astype(np.int32)).pin_memory()
    out_h = [torch.empty(out.shape, dtype=out.dtype).pin_memory() for _ in range(NB)]
    q_d = [torch.empty_like(q) for _ in range(NB)]
    tab_d = [torch.empty_like(tables) for _ in range(NB)]
    len_d = [torch.empty_like(lens_d) for _ in range(NB)]
    out_d = [torch.empty_like(out) for _ in range(NB)]
    up_done = [torch.cuda.Event() for _ in range(NB)]
    dec_done = [torch.cuda.Event() for _ in range(NB)]
    down_done = [torch.cuda.Event() for _ in range(NB)]
    for ev in up_done + dec_done + down_done:
        ev.record(cs)

    def upload(buf):
        with torch.cuda.stream(cs):
            cs.wait_event(dec_done[buf])          # the decode that read this buffer is done
            q_d[buf].copy_(q_h, non_blocking=True)
            tab_d[buf].copy_(tab_h, non_blocking=True)
            len_d[buf].copy_(len_h, non_blocking=True)
            up_done[buf].record(cs)

    def e2e_run(nsteps):
        upload(0)
        for k in range(nsteps):
            buf = k % NB
            if k >= NB:
                # the host consumes step k-NB's result before issuing step k, as a
                # serving loop would; a host running much further ahead fills the
                # CUDA launch queue, where a launch waiting for room can stall it
                down_done[buf].synchronize()
            if k + 1 < nsteps:
                upload((k + 1) % NB)
            stream.wait_event(up_done[buf])
            stream.wait_event(down_done[buf])     # this output buffer was read back
            for l in range(L):
                pool.decode_attention(l, q_d[buf][l], tab_d[buf], len_d[buf], B2, max_blocks,
                                      scale, out_d[buf][l], stream, overlap_previous=ov and l > 0)
            dec_done[buf].record(stream)
            with torch.cuda.stream(cs):
                cs.wait_event(dec_done[buf])
                out_h[buf].copy_(out_d[buf], non_blocking=True)
                down_done[buf].record(cs)
        stream.wait_event(down_done[(nsteps - 1) % NB])

    e2e_run(max(1, args.warmup // 2))
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    if ws > 1:
        dist.barrier()
    e0.record(stream)
    cs.wait_event(e0)
    e2e_run(args.steps)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1)
    if ws > 1:
        dist.barrier()

    # Launches per call, as the library decides them: the split kernel, plus
    # the combine when a session of the table's width can have more splits
    # than the split kernel merges itself (4 in a grid of splits x kv-heads x
    # rows of at least 8 CTAs per SM, else none).
    from paper_2609_25782_gb300 import kvtier
    splits = kvtier.kv_decode_splits(max_blocks * BT)
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    in_kernel = 4 if splits * HKV * B2 >= 8 * sms else 0
    per_call = 1 if splits <= max(1, in_kernel) else 2
    res = {
        "graph": graph is not None, "launches_per_call": per_call,
        "total_ms": total_ms, "launch_ms": launch_ms, "kv_bytes": kv_bytes, "e2e_ms": e2e_ms,
        "launch_alg_bytes": launch_alg_bytes, "setup_s": setup_s, "clocks": clk.summary(),
        "h2d": q.numel() * 2 + tables.numel() * 4 + lens_d.numel() * 4,
        "d2h": out.numel() * 4, "pool": pool, "lens": lens, "tables": tables_h,
    }
    return res


def capture_graph(calls, stream):
    """One CUDA graph of `calls(capture_stream)` (the library's launches are
    recorded like any other stream work), or None if capture fails."""
    import torch
    try:
        with torch.cuda.stream(stream):
            calls(stream)                      # warm the launch path outside capture
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            calls(torch.cuda.current_stream())
        torch.cuda.synchronize()
        return g
    except Exception as e:                     # report and fall back to direct launches
        print(f"graph capture failed, launching directly: {e}", file=sys.stderr)
        return None


def run_migration(args, rank):
    """Resume burst of 8 x 32K-token sessions (cold images -> random free
    blocks of a pool with 2x headroom) and the reverse pack."""
    import torch
    import synth
    from paper_2609_25782_gb300 import Pool
    dev = torch.device("cuda", torch.cuda.current_device())
    n_sess, T = args.mig_sessions, args.mig_tokens
    nb = 2 * n_sess * (T // BT)
    pool = Pool(num_layers=L, num_hot_blocks=nb, cold_bytes=n_sess * T * TOKEN_BYTES + 4096,
                max_sessions=2 * n_sess, max_batch=8, max_context=T, alloc_seed=args.seed + rank,
                device=dev.index)
    st = torch.cuda.Stream(device=dev)
    sids = [pool.session_create_paused(T, T) for _ in range(n_sess)]
    for s in sids:
        synth.fill_image_torch(pool.image(s), args.seed, s, L, HKV, D, T)
    torch.cuda.synchronize()
    img_bytes = T * TOKEN_BYTES

    def gate(stream):
        """Keep the stream busy (a short spin) while the host enqueues the timed
        calls, so the start event fires with their launches already queued and
        the interval is device time, not host launch latency."""
        with torch.cuda.stream(stream):
            torch.cuda._sleep(1_000_000)

    def burst(reps):
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(n_sess)]
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        tot = 0.0
        per = []
        for _ in range(reps):
            gate(st)
            a.record(st)
            for i, s in enumerate(sids):
                ev[i][0].record(st)
                pool.session_resume(s, st)
                ev[i][1].record(st)
            b.record(st)
            torch.cuda.synchronize()
            tot += a.elapsed_time(b)
            per += [e0.elapsed_time(e1) for e0, e1 in ev]
            for s in sids:            # image already valid: pause writes nothing
                pool.session_pause(s, st)
        return tot / reps, per

    burst(1)
    burst_ms, per = burst(max(2, args.steps // 4))
    alone, alone_idle = [], []
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    for rep in range(6):
        if rep % 2 == 0:
            gate(st)
        a.record(st)
        pool.session_resume(sids[0], st)
        b.record(st)
        torch.cuda.synchronize()
        (alone if rep % 2 == 0 else alone_idle).append(a.elapsed_time(b))
        pool.session_pause(sids[0], st)
    flags = pool.check_device()

    # pause-pack: fresh sessions filled by append, then packed (tokens [0, T))
    pack_ms = []
    k, v = synth.kv_logical_torch(args.seed, 0, range(L), HKV, D, 0, T, dev)
    kk = k.permute(0, 2, 1, 3).contiguous()
    vv = v.permute(0, 2, 1, 3).contiguous()
    del k, v
    for s in sids:
        pool.session_destroy(s)
    for rep in range(2):
        fresh = [pool.session_create(T) for _ in range(n_sess)]
        for s in fresh:
            pool.session_append(s, kk, vv, st)
        torch.cuda.synchronize()
        gate(st)
        a.record(st)
        for s in fresh:
            pool.session_pause(s, st)
        b.record(st)
        torch.cuda.synchronize()
        pack_ms.append(a.elapsed_time(b))
        for s in fresh:
            pool.session_destroy(s)
    flags |= pool.check_device()
    pool.close()
    peak, _ = hbm_peak()
    unpack_rw = 2 * n_sess * img_bytes / (burst_ms * 1e-3) / 1e9
    pack_ms_m = statistics.mean(pack_ms)
    pack_rw = 2 * n_sess * img_bytes / (pack_ms_m * 1e-3) / 1e9
    return {
        "resume_unpack": {
            "sessions": n_sess, "tokens": T, "image_bytes": img_bytes,
            "burst_ms": round(burst_ms, 3),
            "gbs_image": round(n_sess * img_bytes / (burst_ms * 1e-3) / 1e9, 1),
            "gbs_rw": round(unpack_rw, 1), "frac_rw": round(unpack_rw / peak, 3),
            "per_session_ms_in_burst": round(statistics.mean(per), 3),
            "per_session_ms_alone": round(statistics.median(alone), 3),
            "per_session_ms_alone_from_idle_gpu": round(statistics.median(alone_idle), 3),
        },
        "pause_pack": {
            "sessions": n_sess, "tokens": T, "burst_ms": round(pack_ms_m, 3),
            "gbs_rw": round(pack_rw, 1), "frac_rw": round(pack_rw / peak, 3),
        },
        "device_flags": flags,
    }


def run_trace(args, rank, lru_factor: float = 0.0):
    """Agentic trace: 48 sessions, N_a = 16, decode on one stream and
    pack/unpack on another; step p50/p99 from events on the decode stream.
    lru_factor > 0: block residency mode with a hot pool of lru_factor times
    the simple mode's peak; its statistics must equal the host dry run's."""
    import dataclasses
    import torch
    import synth
    from paper_2609_25782_gb300 import Pool, kvtier
    from paper_2609_25782_gb300 import trace as tr
    dev = torch.device("cuda", torch.cuda.current_device())
    cfg = tr.TraceConfig(seed=replica_seed(args.seed, rank), steps=args.trace_steps,
                         admit_lead=args.trace_admit_lead,
                         fused_append=not args.trace_unfused_append,
                         prefetch=not args.trace_no_prefetch,
                         overlap=not args.trace_no_overlap, max_ahead=args.trace_max_ahead,
                         graphs=not args.trace_no_graphs)
    trace = tr.generate(cfg)
    plan = tr.plan(cfg, trace)
    nb = plan["peak_blocks"] + 256
    dry = None
    if lru_factor > 0:
        cfg = dataclasses.replace(cfg, lru=True)
        nb = int(plan["peak_blocks"] * lru_factor)
        dry = tr.plan(cfg, trace, hot_blocks=nb)["stats"]
    pool = Pool(num_layers=cfg.layers, num_hot_blocks=nb, cold_bytes=plan["cold_bytes"] + 4096,
                max_sessions=cfg.sessions, max_batch=cfg.active_cap,
                max_context=plan["max_context"], alloc_seed=cfg.seed, device=dev.index,
                lru_residency=cfg.lru)
    kvtier.kv_pool_set_migration_limit(pool.handle, args.trace_mig_ctas)
    for i, t in enumerate(trace):
        sid = pool.session_create_paused(plan["caps"][i], t.t0)
        synth.fill_image_torch(pool.image(sid), cfg.seed, sid, cfg.layers, cfg.num_kv_heads, D,
                               t.t0)
    # appended tokens: slices of one seeded random buffer (values do not
    # change timing); flat so that any [L][n][Hkv][D] prefix is contiguous
    per_tok = cfg.layers * cfg.num_kv_heads * D
    buf_k, buf_v = synth.kv_logical_torch(cfg.seed, 4095, range(cfg.layers), cfg.num_kv_heads, D,
                                          0, cfg.append_max, dev)
    flat_k, flat_v = buf_k.reshape(-1), buf_v.reshape(-1)

    def kv_source(sid, t0, t1):
        n = t1 - t0
        shape = (cfg.layers, n, cfg.num_kv_heads, D)
        return flat_k[: n * per_tok].view(shape), flat_v[: n * per_tok].view(shape)

    def kv_step_source(sids, positions):     # the step tokens of a batch, [L][B][Hkv][D]
        shape = (cfg.layers, len(sids), cfg.num_kv_heads, D)
        n = len(sids) * per_tok
        return flat_k[:n].view(shape), flat_v[:n].view(shape)

    q = synth.queries_torch(cfg.seed, range(cfg.active_cap), range(cfg.layers), HQ, D, dev)
    out = torch.empty(cfg.layers, cfg.active_cap, HQ, D, dtype=torch.float32, device=dev)
    max_blocks = -(-plan["max_context"] // cfg.block_tokens)
    tables = torch.empty(cfg.active_cap, max_blocks, dtype=torch.int32, device=dev)
    seq_lens = torch.empty(cfg.active_cap, dtype=torch.int32, device=dev)
    dstream = torch.cuda.Stream(device=dev, priority=-1)
    mstream = torch.cuda.Stream(device=dev)
    torch.cuda.synchronize()
    d = tr.TraceDriver(cfg, pool.handle, trace, gpu=True, kv_source=kv_source, q=q, out=out,
                       decode_stream=dstream, mig_stream=mstream, tables=tables,
                       seq_lens=seq_lens, max_blocks=max_blocks, kv_step_source=kv_step_source)
    t0 = time.perf_counter()
    with torch.cuda.stream(dstream):
        d.run()
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    flags = pool.check_device()
    step_t = [(a.elapsed_time(b), tok) for a, b, _, tok in d.step_events]
    steps_ms = sorted(t for t, _ in step_t)
    # per-step decode bandwidth: separates workload size from interference
    step_gbs = sorted(tok * TOKEN_BYTES / (t * 1e-3) / 1e9 for t, tok in step_t)
    mig = {"unpack": [0.0, 0], "pack": [0.0, 0], "prefetch": [0.0, 0]}
    for kind, a, b, nbytes in d.mig_events:
        mig[kind][0] += a.elapsed_time(b)
        mig[kind][1] += nbytes
    st = pool.stats()
    pool.close()
    del buf_k, buf_v, flat_k, flat_v
    # decode/migration overlap (Section 3: eviction and resume run beside
    # decode): every interval on one device clock, relative to the first step
    overlap = None
    if d.step_events and any(n > 0 for *_, n in d.mig_events):
        ref = d.step_events[0][0]
        steps_iv = [(ref.elapsed_time(a), ref.elapsed_time(b), tok) for a, b, _, tok in d.step_events]
        # migrations that moved bytes (a residency-mode prefetch with nothing
        # missing, or a pause that packs nothing, is an empty interval)
        migs_iv = [(ref.elapsed_time(a), ref.elapsed_time(b)) for _, a, b, n in d.mig_events
                   if n > 0]
        mig_ms = sum(max(0.0, e - s0) for s0, e in migs_iv)
        inside = 0.0
        j = 0
        for s0, e in sorted(migs_iv):       # steps are disjoint and in time order
            while j < len(steps_iv) and steps_iv[j][1] <= s0:
                j += 1
            i = j
            while i < len(steps_iv) and steps_iv[i][0] < e:
                inside += max(0.0, min(e, steps_iv[i][1]) - max(s0, steps_iv[i][0]))
                i += 1
        busy, idle = [], []
        for s0, e, tok in steps_iv:
            hit = any(ms < e and me > s0 for ms, me in migs_iv)
            (busy if hit else idle).append(tok * TOKEN_BYTES / max(1e-9, (e - s0) * 1e-3) / 1e9)
        med = lambda v: round(statistics.median(v), 1) if v else None
        overlap = {"migration_ms": round(mig_ms, 2),
                   "migration_overlapping_decode_frac": round(inside / max(1e-9, mig_ms), 4),
                   "steps_with_migration": len(busy), "steps_without": len(idle),
                   "decode_kv_gbs_p50_with_migration": med(busy),
                   "decode_kv_gbs_p50_without": med(idle)}
    # host side of the run: enqueue time per step, garbage-collector pauses,
    # and what the host was doing around the slowest step
    host_ms = sorted((h[3] - h[0]) * 1e3 for h in d.host_stamps)
    worst = max(range(len(step_t)), key=lambda i: step_t[i][0]) if step_t else None
    host = {"enqueue_ms_p50": round(host_ms[len(host_ms) // 2], 3),
            "enqueue_ms_max": round(host_ms[-1], 3),
            "gc_pauses": len(d.gc_pauses),
            "gc_pause_ms_max": round(max((p[2] for p in d.gc_pauses), default=0.0) * 1e3, 3),
            # decode steps queued on the GPU when the host began a step
            "queued_steps_p50": sorted(h[5] for h in d.host_stamps)[len(d.host_stamps) // 2]}
    # time the thread spent off the CPU inside a step (blocked in a call, or
    # descheduled): wall time minus thread CPU time
    off = sorted(max(0.0, (h[3] - h[0]) - h[4]) * 1e3 for h in d.host_stamps)
    host["offcpu_ms_p99"] = round(off[int(0.99 * (len(off) - 1))], 3)
    host["offcpu_ms_max"] = round(off[-1], 3)
    host["steps_offcpu_over_1ms"] = sum(1 for x in off if x > 1.0)
    hk = max(range(len(d.host_stamps)), key=lambda i: d.host_stamps[i][3] - d.host_stamps[i][0])
    h = d.host_stamps[hk]
    host["slowest_host_step"] = {
        "step": hk, "ms": round((h[3] - h[0]) * 1e3, 3),
        "pauses_admissions_ms": round((h[1] - h[0]) * 1e3, 3),
        "reserve_ms": round(((h[2] or h[1]) - h[1]) * 1e3, 3),
        "decode_enqueue_ms": round((h[3] - (h[2] or h[1])) * 1e3, 3),
        "thread_cpu_ms": round(h[4] * 1e3, 3),
        "queued_steps_at_start": h[5],
        "gpu_ms": round(step_t[d.step_index.index(hk)][0], 3) if hk in d.step_index else None}
    if worst is not None:
        k = d.step_index[worst]
        lo = max(0, k - 8)
        t_lo, t_hi = d.host_stamps[lo][0], d.host_stamps[k][3]
        host["slowest_step"] = {
            "step": k, "ms": round(step_t[worst][0], 3),
            "host_enqueue_ms": round((d.host_stamps[k][3] - d.host_stamps[k][0]) * 1e3, 3),
            "host_ms_prev8_max": round(max((h[3] - h[0]) * 1e3 for h in d.host_stamps[lo:k + 1]), 3),
            "queued_steps_at_start": d.host_stamps[k][5],
            "queued_steps_prev8_min": min(h[5] for h in d.host_stamps[lo:k + 1]),
            "gc_ms_in_prev8": round(sum(p[2] for p in d.gc_pauses
                                        if t_lo <= p[1] <= t_hi) * 1e3, 3)}
    torch.cuda.empty_cache()

    def pct(p):
        return steps_ms[min(len(steps_ms) - 1, int(round(p / 100 * (len(steps_ms) - 1))))]

    from paper_2609_25782_gb300 import tiering_model
    sim_s = cfg.steps * cfg.dt_s
    # mean KV a resident session holds, over all steps (every session stays resident)
    mean_session = d.counts["session_tokens"] / (cfg.steps * cfg.sessions) * TOKEN_BYTES
    model = tiering_model.from_trace(
        cold_write_bytes=st["bytes_packed"], hot_read_bytes=d.counts["decode_tokens"] * TOKEN_BYTES,
        cold_read_bytes=st["bytes_unpacked"], simulated_seconds=sim_s,
        mean_session_bytes=mean_session,
        hbm_bytes=torch.cuda.get_device_properties(dev).total_memory)
    extra = {"model": {k: (round(v, 3) if isinstance(v, float) and v != float("inf") else
                           (None if v == float("inf") else v)) for k, v in model.items()},
             "simulated_s": sim_s}
    if cfg.lru:
        hit, miss = st["resume_blocks_hit"], st["resume_blocks_missed"]
        extra.update({"mode": "LRU block residency, write-on-evict", "hot_blocks": nb,
                 "hot_vs_simple_peak": lru_factor,
                 "resume_hit_rate": round(hit / max(1, hit + miss), 4),
                 "blocks_evicted": st["blocks_evicted"],
                 "cold_write_gb": round(st["bytes_packed"] / 1e9, 2),
                 "cold_read_gb": round(st["bytes_unpacked"] / 1e9, 2),
                 "prefetch": cfg.prefetch,
                 "blocks_prefetched": st["blocks_prefetched"],
                 "blocks_fetched_in_step": st["batch_blocks_fetched"],
                 "prefetch_skipped": d.counts["prefetch_skipped"],
                 "matches_dry_run": all(st[k] == dry[k] for k in (
                     "bytes_packed", "bytes_unpacked", "blocks_evicted", "resume_blocks_hit",
                     "resume_blocks_missed", "resumes", "pauses", "batch_blocks_fetched",
                     "blocks_prefetched", "prefetches"))})
    return {
        **extra,
        "admit_lead": cfg.admit_lead, "mig_ctas": args.trace_mig_ctas,
        "decode_graphs": len(d.graphs) if cfg.graphs else None, "max_ahead": cfg.max_ahead,
        "step_append": "fused into the decode kernel" if cfg.fused_append else "separate kernel",
        "steps": cfg.steps, "sessions": cfg.sessions, "active_cap": cfg.active_cap,
        "step_ms_p50": round(pct(50), 3), "step_ms_p99": round(pct(99), 3),
        "step_ms_max": round(steps_ms[-1], 3), "wall_s": round(wall, 2), "host": host,
        "overlap": overlap,
        "mean_batch": round(sum(e[2] for e in d.step_events) / max(1, len(d.step_events)), 2),
        "step_kv_gbs_p50": round(step_gbs[len(step_gbs) // 2], 1),
        "step_kv_gbs_p1": round(step_gbs[len(step_gbs) // 100], 1),
        "resumes": st["resumes"], "pauses": st["pauses"],
        "unpack_gb": round(mig["unpack"][1] / 1e9, 2),
        "unpack_gbs": round(mig["unpack"][1] / max(1e-9, mig["unpack"][0] * 1e-3) / 1e9, 1),
        "pack_gb": round(mig["pack"][1] / 1e9, 2),
        "pack_gbs": round(mig["pack"][1] / max(1e-9, mig["pack"][0] * 1e-3) / 1e9, 1),
        "decode_kv_gb": round(d.counts["decode_tokens"] * TOKEN_BYTES / 1e9, 1),
        "hot_read_share": round(d.counts["decode_tokens"] * TOKEN_BYTES /
                                (d.counts["decode_tokens"] * TOKEN_BYTES + mig["unpack"][1]), 4),
        # the hot set's share of resident KV (the paper's counterpart of the read share)
        "hot_set_capacity_share": round(d.counts["decode_tokens"] / d.counts["session_tokens"], 4),
        "device_flags": flags,
        "trace": "seeded synthetic: T0 U[2K,24K], bursts Geometric(200), pauses Exp(30 s), "
                 "turn append LogNormal(median 1536, sigma 1, cap 16K), dt 75 ms/step",
    }


SWEEP_B = (1, 8, 32, 128, 256)
SWEEP_T = (1024, 4096, 16384, 65536, 131072)
SWEEP_CAP = 120e9
# The bounded curve every default run reports (a subset of the full sweep):
# (block tokens, batch, context) decode points and resume-unpack contexts.
CURVE_DECODE = ((16, 1, 16384), (16, 1, 131072), (16, 8, 4096), (16, 8, 65536),
                (16, 32, 16384), (16, 256, 4096), (64, 1, 16384), (64, 8, 65536))
CURVE_RESUME = (1024, 131072)


def run_sweep(args, decode_points=None, resume_T=SWEEP_T):
    """Roofline-fraction curve: the resume-unpack sweep over single sessions
    (1K..128K tokens by default), then decode over (block size, batch,
    context) with total KV <= 120 GB, per-layer launches and the all-layers
    launch. decode_points: (bt, B, T) triples, default every point of the
    full grid."""
    import torch
    import synth
    from paper_2609_25782_gb300 import Pool, kvtier
    dev = torch.device("cuda", torch.cuda.current_device())
    peak, _ = hbm_peak()
    if decode_points is None:
        decode_points = [(bt, B, T) for bt in (16, 64) for B in SWEEP_B for T in SWEEP_T
                         if B * T * TOKEN_BYTES <= SWEEP_CAP]
    # resume-unpack sweep (first, before the long decode sweep loads the GPU)
    resume = []
    Tm = max(resume_T)
    pool = Pool(num_layers=L, num_hot_blocks=Tm // 16 + 64, cold_bytes=Tm * TOKEN_BYTES * 2 + 4096,
                max_sessions=len(resume_T) + 1, max_batch=4, max_context=Tm, alloc_seed=args.seed,
                device=dev.index)
    stream = torch.cuda.Stream(device=dev)
    for T in resume_T:
        s = pool.session_create_paused(T, T)
        synth.fill_image_torch(pool.image(s), args.seed, s, L, HKV, D, T)
        ms, ms_idle = [], []
        for rep in range(12):
            # even reps: device time (a spin keeps the stream busy while the host
            # enqueues the resume, so the start event fires with its launches
            # queued); odd reps: from an idle GPU, host enqueue included
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            if rep % 2 == 0:
                with torch.cuda.stream(stream):
                    torch.cuda._sleep(1_000_000)
            a.record(stream)
            pool.session_resume(s, stream)
            b.record(stream)
            torch.cuda.synchronize()
            if rep >= 4:
                (ms if rep % 2 == 0 else ms_idle).append(a.elapsed_time(b))
            pool.session_pause(s, stream)
        m = statistics.median(ms)
        rw = 2 * T * TOKEN_BYTES / (m * 1e-3) / 1e9
        resume.append({"T": T, "ms": round(m, 4), "gbs_rw": round(rw, 1), "frac": round(rw / peak, 3),
                       "ms_from_idle_gpu": round(statistics.median(ms_idle), 4)})
        pool.session_destroy(s)
    pool.close()
    del pool
    torch.cuda.empty_cache()
    scale = 1 / math.sqrt(D)
    points = []
    for bt in sorted({p[0] for p in decode_points}):
        pts = [(B, T) for b2, B, T in decode_points if b2 == bt]
        max_tok = max(B * T for B, T in pts)
        nb = max_tok // bt + 64
        Bmax = max(B for B, _ in pts)
        # workspace rows: the largest of layers x B x Hq x S(T) over the points
        splits = kvtier.kv_decode_splits
        need = max(L * B * HQ * splits(T) for B, T in pts)
        ctx = max(T for _, T in pts)
        pool = Pool(num_layers=L, num_hot_blocks=nb, cold_bytes=256, block_tokens=bt,
                    max_sessions=4, max_batch=-(-need // (HQ * splits(ctx))),
                    max_context=ctx, device=dev.index)
        # values: one synthetic session laid over the whole pool (finite N(0,1))
        synth.fill_hot_pool_torch(pool.hot, args.seed, [0], [nb * bt], [np.arange(nb)], L, HKV, D,
                                  bt, chunk_blocks=max(1, 48 * 16 // bt))
        stream = torch.cuda.Stream(device=dev)
        for B, T in pts:
            lens = np.full(B, T, dtype=np.int64)
            tables = synth.random_block_tables(args.seed + B + T, lens, bt, nb)
            tab = torch.as_tensor(tables, device=dev)
            sl = torch.as_tensor(lens.astype(np.int32), device=dev)
            q = synth.queries_torch(args.seed, range(B), range(L), HQ, D, dev).contiguous()
            out = torch.empty(L, B, HQ, D, dtype=torch.float32, device=dev)
            res = {"block_tokens": bt, "B": B, "T": T}
            def per_layer(st):
                for l in range(L):
                    pool.decode_attention(l, q[l], tab, sl, B, tab.shape[1], scale, out[l], st,
                                          overlap_previous=l > 0)

            g = capture_graph(per_layer, stream) if args.graph else None
            res["graph"] = g is not None
            for mode in ("per_layer", "all_layers"):
                def step():
                    if mode == "all_layers":
                        pool.decode_attention(-1, q, tab, sl, B, tab.shape[1], scale, out, stream)
                    elif g is not None:
                        with torch.cuda.stream(stream):
                            g.replay()
                    else:
                        per_layer(stream)
                kv = B * T * TOKEN_BYTES
                reps = max(3, min(50, int(2e11 // kv)))
                for _ in range(2):
                    step()
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                torch.cuda.synchronize()
                a.record(stream)
                for _ in range(reps):
                    step()
                b.record(stream)
                torch.cuda.synchronize()
                ms = a.elapsed_time(b) / reps
                gbs = kv / (ms * 1e-3) / 1e9
                res[mode] = {"ms": round(ms, 4), "kv_gbs": round(gbs, 1), "frac": round(gbs / peak, 3)}
            points.append(res)
            del q, out, tab, sl, g
        flags = pool.check_device()
        if flags:
            raise RuntimeError(f"device check flags {flags} in the sweep")
        pool.close()
        del pool
        torch.cuda.empty_cache()
    return {"decode": points, "resume": resume, "peak_gbs": peak}


def cpu_baseline(res, seed, budget_s=15.0):
    """The oracle on a bounded sample of the same step: layer 0 (then more
    layers while the budget lasts) of all 32 sessions, its KV read from the
    device hot pool into a compact host pool."""
    import torch
    import oracle
    import synth
    pool, lens, tables = res["pool"], res["lens"], res["tables"]
    L = pool.L
    hv = pool.hot_view()
    nblk = [-(-int(t) // BT) for t in lens]
    rows = np.concatenate([tables[b, :n] for b, n in enumerate(nblk)]).astype(np.int64)
    compact = np.full((len(nblk), max(nblk)), -1, dtype=np.int32)
    pos = 0
    for b, n in enumerate(nblk):
        compact[b, :n] = np.arange(pos, pos + n)
        pos += n
    idx = torch.as_tensor(rows, device=hv.device)
    sess = list(range(len(lens)))
    spent, layers, kv = 0.0, 0, 0
    while layers < L and spent < budget_s:
        host = hv[idx][:, layers:layers + 1].cpu().view(torch.int16).numpy().view(np.uint16)
        host = np.ascontiguousarray(host)
        qh = synth.queries_np(seed, sess, [layers], HQ, D)
        t0 = time.perf_counter()
        oracle.paged_decode(host, qh, compact, lens, 1 / math.sqrt(D), HQ)
        spent += time.perf_counter() - t0
        layers += 1
        kv += int(np.sum(lens)) * 2 * HKV * D * 2
    return {"value": round(kv / spent / 1e9, 3), "unit": "GB/s", "cores": oracle.threads(),
            "kind": "oracle",
            "sample": f"layers 0..{layers - 1} of the {len(lens)}-session step ({kv / 1e9:.2f} GB of KV), "
                      f"fp64 CPU oracle, {spent:.1f} s"}


def cpu_unpack_baseline(seed, tokens=4096, budget_s=3.0):
    """The oracle's resume copy timed on the host cores: one session image of
    `tokens` tokens in the 48-layer shape unpacked into randomly placed hot
    blocks, repeated while the budget lasts. The copy moves bit patterns, so
    the values are seeded random bytes."""
    import oracle
    rng = np.random.default_rng(seed)
    nblk = -(-tokens // BT)
    img = rng.integers(0, 1 << 16, size=(L, 2, HKV, tokens, D), dtype=np.uint16)
    hot = np.zeros((2 * nblk, L, 2, HKV, BT, D), dtype=np.uint16)
    row = rng.permutation(2 * nblk)[:nblk].astype(np.int32)
    spent, reps = 0.0, 0
    while reps < 1 or spent < budget_s:
        t0 = time.perf_counter()
        oracle.unpack(img, tokens, row, hot)
        spent += time.perf_counter() - t0
        reps += 1
    rw = 2 * tokens * TOKEN_BYTES * reps
    return {"value": round(rw / spent / 1e9, 3), "unit": "GB/s r+w", "cores": 1, "kind": "oracle",
            "sample": f"unpack of one {tokens}-token image ({tokens * TOKEN_BYTES / 1e9:.2f} GB) "
                      f"into random blocks, {reps} times, {spent:.1f} s"}


METRIC = "decode-attn KV GB/s (per step over all layers; resume-unpack GB/s and ms in secondary)"


def workload_name(args) -> str:
    """The decode workload's name, shared by both arms' JSON lines."""
    nl, nbatch = args.layers, args.batch
    if (nl, nbatch, args.tmin, args.tmax) == (L, B2, TMIN2, TMAX2):
        shape = ("Qwen3-Coder-30B-A3B KV shape (48 layers, Hq 32, Hkv 4, D 128, 16-token blocks), "
                 "32 sessions with contexts U[8K,32K]")
    else:
        shape = (f"{nl} layers (Hq 32, Hkv 4, D 128, 16-token blocks), {nbatch} sessions with "
                 f"contexts U[{args.tmin},{args.tmax}] (reduced profiling case)")
    return f"decode-attention step: {shape}, random physical blocks"


def run_reference(args):
    """The oracle timed as the reference arm on host cores: each step is one
    layer of four sessions of the decode workload (lengths from the same
    seeded draw), inputs from the shared generator."""
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    import synth
    lens = synth.session_lengths(args.seed, B2, TMIN2, TMAX2, BT)[:4]
    tables = synth.random_block_tables(args.seed, lens, BT, int(sum(-(-int(t) // BT) for t in lens)))
    hot = synth.hot_pool_np(args.seed, range(4), lens, tables, tables.size and int(tables.max()) + 1,
                            1, HKV, D, BT)
    q = synth.queries_np(args.seed, range(4), [0], HQ, D)
    for _ in range(args.warmup):
        oracle.paged_decode(hot, q, tables, lens, 1 / math.sqrt(D), HQ)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle.paged_decode(hot, q, tables, lens, 1 / math.sqrt(D), HQ)
    dt = time.perf_counter() - t0
    kv = int(np.sum(lens)) * 2 * HKV * D * 2 * args.steps
    val = kv / dt / 1e9
    line = {
        "impl": "reference", "metric": METRIC, "value": round(val, 4), "unit": "GB/s",
        "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(dt / args.steps * 1e3, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload_name(args),
                   "reference_step": "the CPU oracle on layer 0 of 4 of the sessions (bounded sample)"},
        "cpu_baseline": {"value": round(val, 4), "unit": "GB/s", "cores": oracle.threads(),
                         "kind": "oracle",
                         "sample": f"layer 0 of 4 sessions ({int(np.sum(lens))} tokens) per step"},
        "e2e": {"value": round(val, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--no-secondary", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--only-migration", action="store_true",
                    help="skip the decode step (profiling the migration kernels)")
    # workload shape; the defaults are the headline decode configuration
    ap.add_argument("--layers", type=int, default=L)
    ap.add_argument("--batch", type=int, default=B2)
    ap.add_argument("--tmin", type=int, default=TMIN2)
    ap.add_argument("--tmax", type=int, default=TMAX2)
    ap.add_argument("--mig-sessions", type=int, default=8)
    ap.add_argument("--mig-tokens", type=int, default=32768)
    ap.add_argument("--trace-steps", type=int, default=2000)
    ap.add_argument("--trace-admit-lead", type=int, default=1,
                    help="steps between a session's resume and its first decode step")
    ap.add_argument("--trace-mig-ctas", type=int, default=0,
                    help="cap on migration-kernel CTAs during the trace (0: none)")
    ap.add_argument("--only-trace", action="store_true",
                    help="run only the agentic trace (simple and residency modes)")
    ap.add_argument("--trace-max-ahead", type=int, default=30,
                    help="trace: steps the host may run ahead of the GPU (0: unbounded)")
    ap.add_argument("--trace-no-graphs", action="store_true",
                    help="trace: launch each step's decode calls directly (no CUDA graphs)")
    ap.add_argument("--trace-no-overlap", action="store_true",
                    help="trace: launch every layer's decode fully serialised")
    ap.add_argument("--trace-no-prefetch", action="store_true",
                    help="trace (residency mode): no one-step-ahead fetch of spilled blocks")
    ap.add_argument("--trace-lru-factor", type=float, default=1.5,
                    help="residency-mode hot pool as a multiple of the simple mode's peak")
    ap.add_argument("--trace-unfused-append", action="store_true",
                    help="trace: write each step's token with its own kernel before the decode")
    ap.add_argument("--no-trace", action="store_true")
    ap.add_argument("--no-curve", action="store_true",
                    help="skip the bounded roofline curve in the secondary results")
    ap.add_argument("--graph", action=argparse.BooleanOptionalAction, default=True,
                    help="replay the per-layer calls of a step from one CUDA graph")
    ap.add_argument("--no-overlap", action="store_true",
                    help="launch every decode call fully serialised (no programmatic overlap)")
    ap.add_argument("--sweep", action="store_true",
                    help="print the roofline-fraction sweep (block size x batch x context)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)

    import torch
    import torch.distributed as dist
    ws, rank, local = dist_env()
    if ws > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    import __graft_entry__
    if rank == 0 or ws == 1:
        __graft_entry__.build()
    if ws > 1:
        dist.barrier()

    if args.sweep:
        sw = run_sweep(args)
        if rank == 0:
            print(json.dumps({"sweep": sw}))
        return 0
    if args.only_migration:
        sec = run_migration(args, rank)
        if rank == 0:
            print(json.dumps({"secondary": sec}))
        return 0
    if args.only_trace:
        tr_res = {"trace": run_trace(args, rank),
                  "trace_lru": run_trace(args, rank, lru_factor=args.trace_lru_factor)}
        if rank == 0:
            print(json.dumps(tr_res))
        return 0
    res = run_decode(args, ws, rank)
    total_ms = res["total_ms"]
    e2e_ms = res["e2e_ms"]
    if ws > 1:
        total_ms, e2e_ms, all_kv = reduce_over_ranks(total_ms, e2e_ms, float(res["kv_bytes"]),
                                                     device="cuda")
    else:
        all_kv = float(res["kv_bytes"])
    value = all_kv * args.steps / (total_ms * 1e-3) / 1e9
    e2e = all_kv * args.steps / (e2e_ms * 1e-3) / 1e9
    peak, peak_kind = hbm_peak()
    achieved = res["launch_alg_bytes"] / (res["launch_ms"] * 1e-3) / 1e9

    secondary = None
    if not args.no_secondary:
        keep = res["pool"]
        res["pool"] = None
        secondary = run_migration(args, rank)
        res["pool"] = keep
    cpu = None   # the oracle baselines: rank 0 of a single-GPU run only
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(res, replica_seed(args.seed, rank))
        if secondary is not None:
            secondary["resume_unpack"]["cpu_baseline"] = cpu_unpack_baseline(args.seed)
    res["pool"].close()
    del res["pool"]
    torch.cuda.empty_cache()
    if secondary is not None and not args.no_trace:
        secondary["trace"] = run_trace(args, rank)
        secondary["trace_lru"] = run_trace(args, rank, lru_factor=args.trace_lru_factor)
    if secondary is not None and not args.no_curve:
        # the bounded roofline curve (config 5 subset); --sweep prints the full grid
        t_curve = time.time()
        secondary["sweep"] = run_sweep(args, decode_points=CURVE_DECODE, resume_T=CURVE_RESUME)
        secondary["sweep"]["seconds"] = round(time.time() - t_curve, 1)
    nl, nbatch = args.layers, args.batch
    headline = (nl, nbatch, args.tmin, args.tmax) == (L, B2, TMIN2, TMAX2)

    if rank == 0:
        line = {
            "metric": METRIC,
            "value": round(value, 1), "unit": "GB/s", "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(total_ms / args.steps, 4),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": {
                "workload": workload_name(args),
                "tokens": int(np.sum(res["lens"])), "kv_gb_per_step": round(res["kv_bytes"] / 1e9, 2),
                "launches_per_step": res["launches_per_call"] * nl, "compute": "bf16 inputs, fp32 softmax/accumulate",
                "cuda_graph": res["graph"],
                "l2": f"inputs larger than L2 (KV per layer call {res['kv_bytes'] / nl / 1e9:.2f} GB)",
                "parallelism": f"replicas x{ws} (sessions sharded, no collective)",
            },
            "e2e": {"value": round(e2e, 1), "unit": "GB/s", "h2d_bytes_per_step": res["h2d"],
                    "d2h_bytes_per_step": res["d2h"]},
            "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
                         "unit": "GB/s", "frac": round(achieved / peak, 4),
                         "traffic": recorded_traffic() if headline else None,
                         "peak_kind": peak_kind,
                         "kernel": "decode_split_kernel; achieved = algorithmic bytes of one "
                                   "decode_attention call (split kernel + dependent combine) / "
                                   "(timed region / calls)",
                         "alg_bytes_per_launch": int(res["launch_alg_bytes"])},
            "cpu_baseline": cpu,
            # every rank launches the same per-step kernels; whole-job count, like `value`
            "gpu_launches": res["launches_per_call"] * nl * args.steps * ws,
            "clocks": res["clocks"],
            "secondary": secondary,
        }
        print(json.dumps(line))
    if ws > 1:
        dist.barrier()
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())

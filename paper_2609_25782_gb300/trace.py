"""Host trace driver: agentic sessions over the hot/cold KV pool.

Sessions alternate decode bursts with pauses (tool calls, user input); a
batching scheduler keeps at most N_a sessions decoding and admits a waiting
session whenever one pauses (the paper's Section 4 methodology). On a pause
the session's new KV is packed into its cold image and its hot blocks are
freed (data path 4, write-on-evict); on admission its image is unpacked into
fresh blocks (data path 2) and the turn's new context is appended (data path
3). Decode (data path 1) runs on one stream, migrations on another, so
eviction and resume overlap decode (Section 3, data paths).

The schedule is a pure function of the seeded trace: a session admitted at
step k first decodes at step k+1 (one step of prefetch), and the decode
stream waits for its admission event, so a late migration shows up as a
longer step rather than a different schedule. The same driver runs on a
host-logic-only pool (no GPU) to size the arenas before the real run.

Every data movement is a C-ABI call into libkvtier.so; this module only
decides what to call and when.
"""
from __future__ import annotations

import dataclasses
import gc
import heapq
import math
import time
from dataclasses import dataclass, field

import numpy as np

from . import kvtier


@dataclass
class TraceConfig:
    sessions: int = 48
    t0_min: int = 2048
    t0_max: int = 24576
    burst_mean: float = 200.0        # tokens per decode burst (geometric)
    pause_mean_s: float = 30.0       # seconds (exponential)
    append_median: float = 1536.0    # tokens per turn (lognormal)
    append_sigma: float = 1.0        # assumed; only the median is specified
    append_max: int = 16384          # cap on one turn's appended context
    active_cap: int = 16             # N_a
    steps: int = 2000
    dt_s: float = 0.075              # simulated seconds per decode step (assumed)
    layers: int = 48
    num_q_heads: int = 32
    num_kv_heads: int = 4
    block_tokens: int = 16
    seed: int = 0
    lru: bool = False                # block residency with LRU write-on-evict
    admit_lead: int = 1              # steps between a resume and the session's first decode
    fused_append: bool = True        # step token written by the decode kernel itself
    prefetch: bool = True            # residency mode: next step's spilled blocks fetched ahead
    overlap: bool = True             # layer l > 0 starts while layer l-1's call drains
    # Each step's per-layer decode calls replayed from a CUDA graph, one per
    # (batch size, table width rounded up to 1 024 tokens), as a serving
    # engine replays decode graphs per batch bucket; the step's new K/V go
    # through a fixed staging buffer.
    graphs: bool = True
    # The host issues step k only after step k - max_ahead has finished on the
    # GPU; 0: never waits. The queued steps absorb host stalls (a descheduled
    # thread on a shared machine). The CUDA launch queue holds about 1 000
    # launches: about ten steps of direct calls; thirty replayed steps fit
    # (measured: no launch waited for queue space). A launch that waits for
    # queue space can itself stall the host.
    max_ahead: int = 30


@dataclass
class SessionTrace:
    t0: int
    first_ready_s: float
    bursts: list = field(default_factory=list)    # tokens per turn
    pauses: list = field(default_factory=list)    # seconds after each turn
    appends: list = field(default_factory=list)   # context tokens at each turn start


def generate(cfg: TraceConfig, max_turns: int = 64) -> list[SessionTrace]:
    """Seeded per-session turn sequences (independent arrival phases)."""
    rng = np.random.Generator(np.random.PCG64(cfg.seed ^ 0x7A3CE))
    out = []
    p = 1.0 / cfg.burst_mean
    for _ in range(cfg.sessions):
        st = SessionTrace(t0=int(rng.integers(cfg.t0_min, cfg.t0_max + 1)),
                          first_ready_s=float(rng.uniform(0.0, cfg.pause_mean_s)))
        st.bursts = [int(x) for x in rng.geometric(p, size=max_turns)]
        st.pauses = [float(x) for x in rng.exponential(cfg.pause_mean_s, size=max_turns)]
        app = rng.lognormal(math.log(cfg.append_median), cfg.append_sigma, size=max_turns)
        st.appends = [int(min(cfg.append_max, max(1, round(x)))) for x in app]
        out.append(st)
    return out


class TraceDriver:
    """Runs the schedule against a pool handle.

    gpu=False: host-logic-only pool, no CUDA; records the peak sizes.
    gpu=True : real pool; `kv_source(sid, t0, t1)` returns device bf16 K and V
    [L][t1-t0][Hkv][D] for the tokens appended at positions t0..t1-1. With
    cfg.fused_append each step's token goes through kv_pool_batch_reserve and
    decode_append_attention; `kv_step_source(sids, positions)` may supply the
    batch's K and V [L][B][Hkv][D] at once (else kv_source rows are stacked).
    """

    def __init__(self, cfg: TraceConfig, pool: int, trace: list[SessionTrace], gpu: bool,
                 kv_source=None, q=None, out=None, decode_stream=None, mig_stream=None,
                 tables=None, seq_lens=None, max_blocks: int = 0, on_step=None,
                 kv_step_source=None):
        self.cfg, self.pool, self.trace, self.gpu = cfg, pool, trace, gpu
        self.kv_source = kv_source
        self.kv_step_source = kv_step_source
        self.q, self.out = q, out
        self.dstream, self.mstream = decode_stream, mig_stream
        self.tables, self.seq_lens, self.max_blocks = tables, seq_lens, max_blocks
        self.on_step = on_step
        n = cfg.sessions
        self.sids = list(range(n))           # session i has pool id sids[i]
        self.turn = [0] * n
        self.tokens = [t.t0 for t in trace]
        self.burst_left = [0] * n
        self.queue = [(t.first_ready_s, i) for i, t in enumerate(trace)]
        heapq.heapify(self.queue)
        self.active: list[int] = []          # decoding this step
        self.joining: list[tuple[int, int]] = []   # (first decode step, session) admitted
        self.retire: list[int] = []
        self.peak_tokens = list(self.tokens)
        self.peak_blocks = 0
        self.counts = {"resumes": 0, "pauses": 0, "appended_tokens": 0, "decode_tokens": 0,
                       "turn_tokens": 0, "steps": 0, "prefetch_skipped": 0,
                       "session_tokens": 0}   # sum over steps of all sessions' lengths
        self.step_events = []                # (start, end, B, tokens) per decode step (gpu)
        self.step_index = []                 # trace step k of each step_events entry
        self.mig_events = []                 # (kind, start, end, bytes)
        # host clock (perf_counter) per trace step: begin, after pauses and
        # admissions, after the batch reservation, end of enqueue; then the
        # CPU time the thread used over the step (time.thread_time) and the
        # decode steps still queued on the GPU when the step began
        self.host_stamps = []
        self._done = 0                       # step_events[:_done] have finished
        self.gc_pauses = []                  # (generation, start, seconds) during run()
        self.admit_ev = {}
        self.last_decode_ev = None
        self.graphs = {}                     # (B, table width) -> captured decode step
        if gpu:
            import torch
            self._torch = torch
            if cfg.graphs and cfg.fused_append:
                shape = (cfg.layers, cfg.active_cap, cfg.num_kv_heads, 128)
                dev = q.device
                self.k_stage = torch.empty(shape, dtype=torch.bfloat16, device=dev)
                self.v_stage = torch.empty(shape, dtype=torch.bfloat16, device=dev)

    # ---------------------------------------------------------------- helpers
    def _event(self):
        return self._torch.cuda.Event(enable_timing=True)

    def _record_mig(self, kind, fn, nbytes):
        if not self.gpu:
            fn()
            return
        a, b = self._event(), self._event()
        a.record(self.mstream)
        fn()
        b.record(self.mstream)
        self.mig_events.append((kind, a, b, nbytes))

    def _append(self, i, n, stream):
        sid = self.sids[i]
        t0 = self.tokens[i]
        if self.gpu:
            # produce the values on the stream that consumes them (side
            # streams do not order against the default stream)
            with self._torch.cuda.stream(stream):
                k, v = self.kv_source(sid, t0, t0 + n)
                kvtier.session_append(self.pool, sid, k, v, n, stream)
        else:
            kvtier.session_append(self.pool, sid, None, None, n, None)
        self.tokens[i] += n
        self.peak_tokens[i] = max(self.peak_tokens[i], self.tokens[i])

    def _step_kv(self, members):
        """K and V [L][B][Hkv][D] of the step's new token of each member."""
        sids = [self.sids[i] for i in members]
        pos = [self.tokens[i] for i in members]
        if self.kv_step_source is not None:
            return self.kv_step_source(sids, pos)
        torch = self._torch
        rows = [self.kv_source(sid, t, t + 1) for sid, t in zip(sids, pos)]
        return (torch.cat([r[0] for r in rows], dim=1).contiguous(),
                torch.cat([r[1] for r in rows], dim=1).contiguous())

    # ------------------------------------------------------------------- step
    def step(self, k: int) -> None:
        cfg = self.cfg
        if self.gpu and cfg.max_ahead > 0 and len(self.step_events) >= cfg.max_ahead:
            self.step_events[-cfg.max_ahead][1].synchronize()
        queued = 0
        if self.gpu:
            ev = self.step_events
            while self._done < len(ev) and ev[self._done][1].query():
                self._done += 1
            queued = len(ev) - self._done
        h0 = time.perf_counter()
        c0 = time.thread_time()
        h_adm = h_res = None
        now = k * cfg.dt_s
        tok_bytes = cfg.layers * 2 * cfg.num_kv_heads * 128 * 2
        # 1. sessions whose burst ended last step pause. Simple mode packs their
        # new tokens and frees the blocks; residency mode moves nothing (the
        # blocks age until evicted). Migrations may touch blocks the last
        # decode step read, so they wait for it.
        if self.gpu and self.last_decode_ev is not None and (self.retire or cfg.lru):
            self.mstream.wait_event(self.last_decode_ev)
        for i in self.retire:
            sid = self.sids[i]
            info = kvtier.session_info(self.pool, sid)
            nbytes = 0 if cfg.lru else (info.tokens - info.cold_valid) * tok_bytes
            self._record_mig("pack", lambda: kvtier.session_pause(
                self.pool, sid, self.mstream if self.gpu else None), nbytes)
            self.active.remove(i)
            heapq.heappush(self.queue, (now + self.trace[i].pauses[self.turn[i]], i))
            self.turn[i] += 1
            self.counts["pauses"] += 1
        self.retire = []
        # sessions whose admission lead has passed join the batch now
        self.active.extend(i for j, i in self.joining if j <= k)
        self.joining = [(j, i) for j, i in self.joining if j > k]
        # 2. admit ready sessions while below the cap (resume + turn context)
        while (len(self.active) + len(self.joining) < cfg.active_cap and self.queue
               and self.queue[0][0] <= now):
            _, i = heapq.heappop(self.queue)
            sid = self.sids[i]
            before = kvtier.kv_pool_get_stats(self.pool)["bytes_unpacked"]
            self._record_mig("unpack", lambda: kvtier.session_resume(
                self.pool, sid, self.mstream if self.gpu else None), 0)
            fetched = kvtier.kv_pool_get_stats(self.pool)["bytes_unpacked"] - before
            if self.gpu:
                kind, a, b, _ = self.mig_events[-1]
                self.mig_events[-1] = (kind, a, b, fetched)
            n_ctx = self.trace[i].appends[self.turn[i]]
            self._append(i, n_ctx, self.mstream if self.gpu else None)
            self.counts["turn_tokens"] += n_ctx
            self.burst_left[i] = self.trace[i].bursts[self.turn[i]]
            if self.gpu:
                ev = self._torch.cuda.Event()
                ev.record(self.mstream)
                self.admit_ev[i] = ev
            self.joining.append((k + max(1, cfg.admit_lead), i))
            self.counts["resumes"] += 1
        # 3. decode step for the active batch
        h_adm = time.perf_counter()
        members = sorted(self.active)
        if members:
            if self.gpu:
                start, end = self._event(), self._event()
                start.record(self.dstream)
                for i in members:
                    ev = self.admit_ev.pop(i, None)
                    if ev is not None:
                        self.dstream.wait_event(ev)
            sids = [self.sids[i] for i in members]
            B = len(sids)
            # tables as wide as this batch's longest session (after its step token):
            # no launched split lies past every session's end; with graphs, rounded
            # up to 1 024 tokens so that a step's graph is reused
            mb = -(-(max(self.tokens[i] for i in members) + 1) // cfg.block_tokens)
            if self.gpu and cfg.graphs and self.max_blocks:
                r = max(1, 1024 // cfg.block_tokens)
                mb = min(self.max_blocks, -(-mb // r) * r)
            if cfg.fused_append:             # this step's token (path 3) comes with the decode
                if self.gpu:
                    with self._torch.cuda.stream(self.dstream):
                        k_new, v_new = self._step_kv(members)
                    kvtier.kv_pool_batch_reserve(self.pool, sids, self.tables, mb,
                                                 self.seq_lens, self.dstream)
                else:
                    kvtier.kv_pool_batch_reserve(self.pool, sids, None, 1 << 20, None, None)
                for i in members:
                    self.tokens[i] += 1
                    self.peak_tokens[i] = max(self.peak_tokens[i], self.tokens[i])
            else:
                for i in members:             # this step's token (path 3)
                    self._append(i, 1, self.dstream if self.gpu else None)
                if not self.gpu and cfg.lru:     # recency and spilled-block fetches
                    kvtier.kv_pool_batch_tables(self.pool, sids, None, 1 << 20, None, None)
                if self.gpu:
                    kvtier.kv_pool_batch_tables(self.pool, sids, self.tables, mb,
                                                self.seq_lens, self.dstream)
            h_res = time.perf_counter()
            self.counts["appended_tokens"] += len(members)
            blocks = sum(-(-self.tokens[i] // cfg.block_tokens)
                         for i in self.active + [i for _, i in self.joining])
            self.peak_blocks = max(self.peak_blocks, blocks)
            if self.gpu:
                if cfg.fused_append and cfg.graphs:
                    with self._torch.cuda.stream(self.dstream):   # fixed addresses
                        self.k_stage[:, :B].copy_(k_new)
                        self.v_stage[:, :B].copy_(v_new)
                    k_new, v_new = self.k_stage, self.v_stage
                g = self.graphs.get((B, mb)) if cfg.graphs else None
                if g is not None:
                    with self._torch.cuda.stream(self.dstream):
                        g.replay()
                    end.record(self.dstream)
                else:
                    self._decode_calls(B, mb, k_new, v_new)
                    end.record(self.dstream)
                    if cfg.graphs:               # record it for the next step of this shape
                        g = self._torch.cuda.CUDAGraph()
                        with self._torch.cuda.stream(self.dstream):
                            g.capture_begin(capture_error_mode="relaxed")
                            self._decode_calls(B, mb, k_new, v_new)
                            g.capture_end()
                        self.graphs[(B, mb)] = g
                self.last_decode_ev = end
                self.step_events.append((start, end, B, sum(self.tokens[i] for i in members)))
                self.step_index.append(k)
                if self.on_step is not None:
                    self.on_step(k, members)
            self.counts["decode_tokens"] += sum(self.tokens[i] for i in members)
            for i in members:
                self.burst_left[i] -= 1
                if self.burst_left[i] <= 0:
                    self.retire.append(i)
            if cfg.lru and cfg.prefetch:
                self._prefetch_next(k, sids)
        self.counts["steps"] += 1
        self.counts["session_tokens"] += sum(self.tokens)
        self.host_stamps.append((h0, h_adm, h_res, time.perf_counter(), time.thread_time() - c0,
                                 queued))

    def _decode_calls(self, B: int, mb: int, k_new, v_new) -> None:
        """The step's per-layer decode calls on the decode stream."""
        cfg = self.cfg
        for l in range(cfg.layers):
            # layer l > 0 follows layer l-1's call, which writes only `out`
            # and (fused) layer l-1's rows of the pool
            flags = kvtier.KV_DECODE_OVERLAP_PREVIOUS if l > 0 and cfg.overlap else 0
            if cfg.fused_append:
                kvtier.decode_append_attention(
                    self.pool, l, self.q[l], k_new[l], v_new[l], self.tables, self.seq_lens, B,
                    mb, 1 / math.sqrt(128), self.out[l], flags, self.dstream)
            else:
                kvtier.decode_attention_ex(
                    self.pool, l, self.q[l], self.tables, self.seq_lens, B, mb,
                    1 / math.sqrt(128), self.out[l], flags, self.dstream)

    def _prefetch_next(self, k: int, busy: list) -> None:
        """One step ahead (Section 3, "Eviction, resume and decode"): the
        sessions of step k+1 are known now (this step's members minus those
        whose burst just ended, plus the admitted sessions that join at k+1),
        so their evicted blocks are fetched on the migration stream while
        step k decodes; victims exclude both batches. The migration stream is
        already ordered after step k-1's decode (start of this step)."""
        retiring = set(self.retire)
        nxt = sorted({i for i in self.active if i not in retiring} |
                     {i for j, i in self.joining if j <= k + 1})
        if not nxt:
            return
        sids = [self.sids[i] for i in nxt]

        def call():
            try:
                kvtier.kv_pool_prefetch(self.pool, sids, busy, self.mstream if self.gpu else None)
            except kvtier.KVError as e:   # too few victims outside both batches: the
                if e.code != kvtier.KV_ERR_NO_HOT_BLOCKS:   # step's own call fetches them
                    raise
                self.counts["prefetch_skipped"] += 1

        if self.gpu:
            before = kvtier.kv_pool_get_stats(self.pool)["blocks_prefetched"]
            self._record_mig("prefetch", call, 0)
            n = kvtier.kv_pool_get_stats(self.pool)["blocks_prefetched"] - before
            kind, a, b, _ = self.mig_events[-1]
            tok_bytes = self.cfg.layers * 2 * self.cfg.num_kv_heads * 128 * 2
            self.mig_events[-1] = (kind, a, b, n * self.cfg.block_tokens * tok_bytes)
        else:
            call()

    def run(self, steps: int | None = None) -> None:
        """Run the schedule; Python garbage-collector pauses that fall inside
        it are recorded in gc_pauses (a host stall long enough to drain the
        launch queue shows up as a longer step)."""
        started = {}

        def on_gc(phase, info):
            if phase == "start":
                started["t"] = time.perf_counter()
            elif "t" in started:
                t = started.pop("t")
                self.gc_pauses.append((info.get("generation", -1), t, time.perf_counter() - t))

        gc.callbacks.append(on_gc)
        try:
            for k in range(self.cfg.steps if steps is None else steps):
                self.step(k)
        finally:
            gc.callbacks.remove(on_gc)


def plan(cfg: TraceConfig, trace: list[SessionTrace], hot_blocks: int | None = None) -> dict:
    """Dry run on a host-logic-only pool: per-session capacity and peak hot
    blocks needed by the real run (the schedule does not depend on timing).
    With cfg.lru and hot_blocks, the dry run uses a residency-mode pool of
    that size and its statistics are those the real run must reproduce."""
    lru = cfg.lru and hot_blocks is not None
    if cfg.lru and not lru:
        cfg = dataclasses.replace(cfg, lru=False)
    tok_bytes = cfg.layers * 2 * cfg.num_kv_heads * 128 * 2
    big = cfg.sessions * (1 << 22) * tok_bytes    # host-logic pool: nothing is allocated
    c = kvtier.make_config(num_layers=cfg.layers, num_q_heads=cfg.num_q_heads,
                           num_kv_heads=cfg.num_kv_heads, block_tokens=cfg.block_tokens,
                           max_sessions=cfg.sessions, max_batch=cfg.active_cap,
                           max_context=1 << 22,
                           num_hot_blocks=hot_blocks if lru else 300000, cold_bytes=big,
                           flags=kvtier.KV_POOL_HOST_LOGIC_ONLY |
                           (kvtier.KV_POOL_LRU_RESIDENCY if lru else 0))
    pool = kvtier.kv_pool_create(c)
    try:
        for t in trace:
            kvtier.session_create_paused(pool, 1 << 22, t.t0)
        d = TraceDriver(cfg, pool, trace, gpu=False)
        d.run()
        stats = kvtier.kv_pool_get_stats(pool)
    finally:
        kvtier.kv_pool_destroy(pool)
    caps = [int(x) for x in d.peak_tokens]
    return {"caps": caps, "peak_blocks": int(d.peak_blocks), "counts": d.counts, "stats": stats,
            "cold_bytes": int(sum(-(-(cap * tok_bytes) // 256) * 256 for cap in caps)),
            "max_context": int(max(caps))}

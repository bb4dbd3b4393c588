"""Oracle of the block residency policy (test infrastructure).

Restates, slowly and directly, the eviction and resume policy of the paper's
hot-cold hierarchy (Section 3, "Eviction, resume and decode" and "Memory
hierarchy and write policy"; Section 4, "Methodology"):

* every KV block is resident in HBM, in the cold tier, or both;
* when HBM has no free block, the least recently used block is evicted;
  active blocks are not pinned, recency alone keeps them hot;
* a block is written to the cold tier only when it is evicted, and only the
  tokens the cold copy does not hold yet (KV is immutable, so a block is
  written at most once);
* a resumed session fetches only its blocks that are not in HBM (the resume
  hit rate is the fraction that still is).

Recency is kept per session: appending to a session, resuming it, or
batching it for a decode step stamps all its blocks with a new time (one
time per call). The victim is the hot block with the smallest
(time, session id, block index), skipping the sessions the current call
works on. Freed and evicted blocks go to the end of the free list in that
order and allocations pop from the end (the placement contract of
oracle.FreeList).

The scan over every hot block on each eviction is deliberately naive: the
library keeps an ordered set of sessions instead, and the tests compare the
two decision by decision.
"""
from __future__ import annotations

from dataclasses import dataclass, field

from . import FreeList


class NoHotBlocks(Exception):
    pass


@dataclass
class Sess:
    state: str                     # "active" | "paused"
    T: int
    cap: int
    slots: list = field(default_factory=list)    # per logical block: slot or -1
    img: list = field(default_factory=list)      # per logical block: tokens in the image
    time: int = 0


class ResidencyOracle:
    def __init__(self, num_blocks: int, block_tokens: int, seed: int, token_bytes: int):
        self.fl = FreeList(num_blocks, seed)
        self.bt = block_tokens
        self.tb = token_bytes
        self.clock = 0
        self.s: dict[int, Sess] = {}
        self.stats = {"bytes_packed": 0, "bytes_unpacked": 0, "bytes_appended": 0,
                      "blocks_evicted": 0, "resume_blocks_hit": 0, "resume_blocks_missed": 0,
                      "batch_blocks_fetched": 0, "blocks_prefetched": 0, "prefetches": 0}
        self.log = []              # ("pack"|"unpack", sid, j, slot, t0, t1) in issue order

    # ----------------------------------------------------------- helpers
    def n_in(self, s: Sess, j: int) -> int:
        return min(self.bt, s.T - j * self.bt)

    def _hot(self):
        for sid, s in self.s.items():
            for j, slot in enumerate(s.slots):
                if slot >= 0:
                    yield (s.time, sid, j)

    def _evict(self, need: int, protect: set):
        """Evict LRU blocks until the free list holds `need` blocks."""
        while self.fl.n < need:
            cands = [h for h in self._hot() if h[1] not in protect]
            if not cands:
                raise NoHotBlocks()
            _, sid, j = min(cands)
            s = self.s[sid]
            slot = s.slots[j]
            n = self.n_in(s, j)
            if s.img[j] < n:               # write only what the cold copy lacks
                self.log.append(("pack", sid, j, slot, s.img[j], n))
                self.stats["bytes_packed"] += (n - s.img[j]) * self.tb
                s.img[j] = n
            s.slots[j] = -1
            self.fl.push([slot])
            self.stats["blocks_evicted"] += 1

    def _tick(self) -> int:
        self.clock += 1
        return self.clock

    def _fetch(self, sid: int, js: list):
        s = self.s[sid]
        got = self.fl.pop(len(js))
        for j, slot in zip(js, got):
            s.slots[j] = int(slot)
            n = self.n_in(s, j)
            assert s.img[j] == n, "a block missing from HBM must be whole in the cold tier"
            self.log.append(("unpack", sid, j, int(slot), 0, n))
            self.stats["bytes_unpacked"] += n * self.tb

    def _check_room(self, need: int, protect: set):
        """All-or-nothing: raise before changing anything if eviction cannot
        free `need` blocks."""
        evictable = sum(1 for h in self._hot() if h[1] not in protect)
        if self.fl.n + evictable < need:
            raise NoHotBlocks()

    # ------------------------------------------------------------ ops
    def create(self, sid: int, cap: int):
        self.s[sid] = Sess("active", 0, cap)

    def create_paused(self, sid: int, cap: int, T: int):
        nb = -(-T // self.bt)
        s = Sess("paused", T, cap, [-1] * nb, [0] * nb)
        s.img = [self.n_in(s, j) for j in range(nb)]
        self.s[sid] = s

    def append(self, sid: int, n: int):
        s = self.s[sid]
        assert s.state == "active"
        bt = self.bt
        tail = (s.T - 1) // bt if s.T > 0 else -1
        refetch = [tail] if (s.T % bt and tail >= 0 and s.slots[tail] < 0) else []
        new = -(-(s.T + n) // bt) - len(s.slots)
        self._check_room(len(refetch) + max(0, new), {sid})
        self._evict(len(refetch) + max(0, new), {sid})
        if refetch:
            self._fetch(sid, refetch)
        got = self.fl.pop(max(0, new))
        for slot in got:
            s.slots.append(int(slot))
            s.img.append(0)
        s.T += n
        s.time = self._tick()
        self.stats["bytes_appended"] += n * self.tb

    def pause(self, sid: int):
        s = self.s[sid]
        assert s.state == "active"
        s.state = "paused"

    def resume(self, sid: int):
        s = self.s[sid]
        assert s.state == "paused"
        missing = [j for j, slot in enumerate(s.slots) if slot < 0]
        self._check_room(len(missing), {sid})
        self._evict(len(missing), {sid})
        self.stats["resume_blocks_hit"] += len(s.slots) - len(missing)
        self.stats["resume_blocks_missed"] += len(missing)
        self._fetch(sid, missing)
        s.state = "active"
        s.time = self._tick()

    def _bring_back(self, sids: list, protect: set) -> int:
        """Fetch every missing block of `sids` (each session once, in order of
        first appearance), evicting outside `protect`; stamp them all with one
        time. Returns the number of blocks fetched."""
        uniq = list(dict.fromkeys(sids))
        need = [(sid, [j for j, slot in enumerate(self.s[sid].slots) if slot < 0]) for sid in uniq]
        total = sum(len(m) for _, m in need)
        self._check_room(total, protect)
        self._evict(total, protect)
        for sid, missing in need:
            if missing:
                self._fetch(sid, missing)
        t = self._tick()
        for sid in uniq:
            self.s[sid].time = t
        return total

    def batch(self, sids: list):
        self.stats["batch_blocks_fetched"] += self._bring_back(sids, set(sids))

    def prefetch(self, sids: list, busy: list = ()):
        """One step ahead of decode (Section 3, "Eviction, resume and
        decode"): the next step's sessions get their evicted blocks back now,
        while the current step (the sessions in `busy`) is still decoding, so
        victims may belong to neither. All or nothing; the next step's
        sessions are stamped as used."""
        for sid in sids:
            assert self.s[sid].state == "active"
        self.stats["blocks_prefetched"] += self._bring_back(sids, set(sids) | set(busy))
        self.stats["prefetches"] += 1

    def batch_reserve(self, sids: list):
        """One decode step's fresh token for each session of the batch (its
        values are written by the decode itself): evicted blocks come back,
        a session whose tail block is full gets a new one, and every member
        grows by one token. Victims are outside the batch; pops go member by
        member, missing blocks first."""
        assert len(set(sids)) == len(sids)
        plan = []
        for sid in sids:
            s = self.s[sid]
            assert s.state == "active" and s.T + 1 <= s.cap
            missing = [j for j, slot in enumerate(s.slots) if slot < 0]
            plan.append((sid, missing, 1 if s.T % self.bt == 0 else 0))
        total = sum(len(m) + g for _, m, g in plan)
        self._check_room(total, set(sids))
        self._evict(total, set(sids))
        for sid, missing, grow in plan:
            s = self.s[sid]
            if missing:
                self._fetch(sid, missing)
                self.stats["batch_blocks_fetched"] += len(missing)
            if grow:
                s.slots.append(int(self.fl.pop(1)[0]))
                s.img.append(0)
            s.T += 1
            self.stats["bytes_appended"] += self.tb
        t = self._tick()
        for sid in sids:
            self.s[sid].time = t

    def destroy(self, sid: int):
        s = self.s.pop(sid)
        self.fl.push([slot for slot in s.slots if slot >= 0])

    def shuffle(self, seed: int):
        self.fl.shuffle(seed)

    def row(self, sid: int) -> list:
        return list(self.s[sid].slots)

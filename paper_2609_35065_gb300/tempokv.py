"""TempoKV's control plane as a discrete-event model over the fast-tier ledger.

The hot path of this package moves matched prefix KV from the fast tier into
the GPU's paged cache; this module decides *when* that KV is staged from SSD
into the fast tier and protected, following the paper's design (Sec. 3):

* ``OutputLengthEstimator`` -- remaining output of a running request with n
  generated tokens: the mean of N - n over completed outputs of length N > n,
  with the generation limit bounding the predicted total (Sec. 3.1, TTU).
* ``Runtime`` -- an FCFS engine with at most ``max_active`` sequences; its
  ``ttu`` is a read-only projection of the running and queued-ahead requests on
  one shared timeline with calibrated prefill/decode costs, assuming the
  target is stage-ready and honouring the known retrieval dependencies of the
  requests ahead (Sec. 3.1).
* ``Provider`` -- SSD-to-fast-tier staging in issue order at an aggregate rate,
  over the native ledger (``kvs.Tier``: protection, coalescing, budget, LRU,
  cost integral); ``ttr`` is a metadata-only projection that adds reads only
  for objects neither resident nor covered by queued staging, and takes the
  completion of the last required object (Sec. 3.1, TTR).
* ``Controller`` -- laxity L = TTU - TTR of each uncommitted claim; a claim is
  eligible when L <= 0 or the runtime requests its retrieval; attempts go
  pending-retrieval claims first, then runtime order; a capacity-blocked claim
  does not block others; re-evaluation on every event and on a 50 ms tick;
  commitments are never revoked; a claim whose retrieval is requested but that
  cannot be committed takes the ordinary path (Sec. 3.2).
* ``simulate`` -- requests arriving at fixed intervals (Sec. 5.1), each
  retrieving its matched prefix at the fast-tier-to-GPU rate measured for this
  package's kernels, then prefilling the uncached suffix and decoding; reports
  p95 TTFT, output throughput and the protected-capacity cost
  C = integral P(t) dt / N (Sec. 5, Metrics).

Timing parameters are inputs (``Calibration``); nothing here reads a GPU.
"""
from __future__ import annotations

import heapq
import itertools
from collections import deque
from dataclasses import dataclass, field

import numpy as np

from . import kvs


@dataclass
class Calibration:
    prefill_tok_s: float = 12000.0      # uncached prompt tokens per second
    decode_step_s: float = 0.02         # one decode iteration of the active batch
    retrieval_gbs: float = 211.0        # fast tier -> GPU (GB/s), this package's measured rate
    staging_gibs: float = 11.0          # SSD -> fast tier aggregate rate (GiB/s)
    kv_bytes_per_token: int = 128 * 1024
    chunk_tokens: int = 256
    max_active: int = 4
    gen_limit: int = 128
    tick_s: float = 0.05

    @property
    def object_bytes(self) -> int:
        return self.kv_bytes_per_token * self.chunk_tokens

    def retrieval_s(self, tokens: int) -> float:
        return tokens * self.kv_bytes_per_token / (self.retrieval_gbs * 1e9)

    def prefill_s(self, tokens: int) -> float:
        return tokens / self.prefill_tok_s


@dataclass
class Request:
    rid: int
    arrival: float
    prompt: int
    matched: int                         # tokens of retained prefix KV (whole chunks)
    output: int                          # true output length (unknown to the estimators)
    keys: list = field(default_factory=list)
    admitted: float | None = None
    first_token: float | None = None
    finished: float | None = None
    generated: int = 0


class OutputLengthEstimator:
    """Remaining output of a request with n tokens generated (Sec. 3.1)."""

    def __init__(self, limit: int, history=()):
        self.limit = limit
        self.done = list(history)

    def add(self, n_total: int) -> None:
        self.done.append(n_total)

    def remaining(self, n: int) -> float:
        longer = [N for N in self.done if N > n]
        if not longer:
            return max(self.limit - n, 0)
        return min(float(np.mean(longer)) - n, self.limit - n)


class Provider:
    """SSD -> fast-tier staging in issue order at one aggregate rate, over the ledger."""

    def __init__(self, tier: kvs.Tier, cal: Calibration):
        self.tier, self.cal = tier, cal
        self.rate = cal.staging_gibs * 2 ** 30          # bytes per second
        self.queue = deque()                            # (key, completion time)
        self.done_at = {}                               # key -> projected completion

    def tail(self, now: float) -> float:
        return max(now, self.queue[-1][1]) if self.queue else now

    def enqueue(self, keys, now: float) -> None:
        t = self.tail(now)
        for k in keys:
            t += self.cal.object_bytes / self.rate
            self.queue.append((k, t))
            self.done_at[k] = t

    def ttr(self, keys, now: float) -> float:
        """Metadata-only projection of a commitment made now (Sec. 3.1)."""
        last, new = now, 0
        for k in keys:
            info = self.tier.object(k)
            if info is not None and info["resident"]:
                continue                                # needs protection, not a read
            if k in self.done_at:
                last = max(last, self.done_at[k])       # covered by queued staging
            else:
                new += 1
        if new:
            last = max(last, self.tail(now) + new * self.cal.object_bytes / self.rate)
        return last - now

    def ready_time(self, keys, now: float) -> float:
        """When every object of a committed claim is resident (projected)."""
        return max([now] + [self.done_at[k] for k in keys if k in self.done_at])

    def next_completion(self):
        return self.queue[0][1] if self.queue else None

    def complete_head(self, now: float):
        k, _ = self.queue.popleft()
        del self.done_at[k]
        self.tier.staged(k, now)
        return k


class Runtime:
    """FCFS engine; ``ttu`` is the adapter's shared-timeline projection."""

    def __init__(self, cal: Calibration, est: OutputLengthEstimator):
        self.cal, self.est = cal, est
        self.waiting = deque()
        self.prefilling = []                            # admitted, retrieving/prefilling
        self.running = []                               # Requests being decoded
        self.busy_until = 0.0

    def _decode_until(self, rem, t_from, t_to):
        """Project decoding of the running batch from t_from to t_to."""
        steps = int((t_to - t_from) / self.cal.decode_step_s)
        return [r - steps for r in rem if r - steps > 0]

    def ttu(self, target: Request, now: float, ready_time) -> float:
        """Time until the target's retrieval would begin, assuming it is stage-ready.
        ``ready_time(req)`` gives the projected KV readiness of a request ahead."""
        d = self.cal.decode_step_s
        t = max(now, self.busy_until)
        rem = [max(self.est.remaining(r.generated), 1.0) for r in self.running]
        rem += [max(self.est.remaining(0), 1.0) for _ in self.prefilling]
        for r in self.waiting:
            while len(rem) >= self.cal.max_active:      # wait for a slot
                k = min(rem)
                t += np.ceil(k) * d
                rem = [x - np.ceil(k) for x in rem if x - np.ceil(k) > 0]
            if r is target:
                return t - now
            ready = ready_time(r)
            if ready > t:                               # a known retrieval dependency
                rem = self._decode_until(rem, t, ready)
                t = ready
            t += self.cal.retrieval_s(r.matched) + self.cal.prefill_s(r.prompt - r.matched)
            rem.append(max(self.est.remaining(0), 1.0))
        raise ValueError("target is not waiting")


class Controller:
    """Claims, laxity and commitment (Sec. 3.2)."""

    def __init__(self, tier: kvs.Tier, provider: Provider, runtime: Runtime):
        self.tier, self.provider, self.runtime = tier, provider, runtime
        self.claims = {}            # rid -> dict(req, ttu, stamp, requested, ordinary)
        self.blocked_attempts = 0
        self.commit_times = {}

    def add(self, req: Request, now: float) -> None:
        self.claims[req.rid] = {"req": req, "ttu": None, "stamp": now, "requested": False, "ordinary": False}

    def update_ttus(self, now: float) -> None:
        for c in self.claims.values():
            if self._uncommitted(c) and c["req"] in self.runtime.waiting:
                c["ttu"] = self.runtime.ttu(c["req"], now, self._ready_time)
                c["stamp"] = now

    def _ready_time(self, req: Request) -> float:
        c = self.claims.get(req.rid)
        if c is None:
            return 0.0
        st = self.tier.state(req.rid)
        if st in (kvs.KVS_CLAIM_STAGING, kvs.KVS_CLAIM_ORDINARY):
            return self.provider.ready_time(req.keys, 0.0)
        return 0.0

    def _uncommitted(self, c) -> bool:
        return not c["ordinary"] and self.tier.state(c["req"].rid) in (kvs.KVS_CLAIM_NONE, kvs.KVS_CLAIM_PLANNED)

    def laxity(self, rid: int, now: float) -> float:
        c = self.claims[rid]
        ttu = c["ttu"] - (now - c["stamp"])             # the latest TTU, aged by elapsed time
        return ttu - self.provider.ttr(c["req"].keys, now)

    def evaluate(self, now: float) -> None:
        order = {r.rid: i for i, r in enumerate(self.runtime.waiting)}
        cands = [c for c in self.claims.values() if self._uncommitted(c) and c["ttu"] is not None]
        cands.sort(key=lambda c: (not c["requested"], order.get(c["req"].rid, 1 << 30)))
        for c in cands:
            rid = c["req"].rid
            if not (c["requested"] or self.laxity(rid, now) <= 0):
                continue
            try:
                keys = self.tier.commit(rid, c["req"].keys, now)
            except kvs.KvsError as e:
                if e.code != kvs.KVS_ERR_NOMEM:
                    raise
                self.blocked_attempts += 1              # stays Planned; others still get a try
                continue
            self.commit_times[rid] = now
            self.provider.enqueue(keys, now)

    def request_retrieval(self, req: Request, now: float) -> None:
        c = self.claims[req.rid]
        c["requested"] = True
        self.evaluate(now)
        if self._uncommitted(c):                        # no protection available: ordinary path
            keys = self.tier.ordinary(req.rid, req.keys, now)
            self.provider.enqueue(keys, now)
            c["ordinary"] = True


@dataclass
class Result:
    ttft: list
    p95_ttft: float
    throughput_tok_s: float
    cost_gib_s_per_req: float
    blocked_attempts: int
    ordinary: int
    staged_reads: int
    commit_lead_s: list             # retrieval start minus commitment time, per committed claim
    commit_times: dict              # rid -> time of its commitment
    retrieval_starts: dict          # rid -> time its retrieval began


def simulate(requests, cal: Calibration, capacity_gib: float = 100.0, budget_gib: float = 50.0,
             history=()) -> Result:
    """Runs the requests (sorted by arrival) to completion."""
    cap = int(capacity_gib * 2 ** 30 // cal.object_bytes)
    budget = int(budget_gib * 2 ** 30 // cal.object_bytes)
    tier = kvs.Tier(cap, budget, cal.object_bytes)
    est = OutputLengthEstimator(cal.gen_limit, history)
    rt = Runtime(cal, est)
    prov = Provider(tier, cal)
    ctl = Controller(tier, prov, rt)
    seq = itertools.count()
    events = []

    def push(t, kind, payload=None):
        heapq.heappush(events, (t, next(seq), kind, payload))

    for r in requests:
        push(r.arrival, "arrival", r)
    push(0.0, "tick")
    engine_busy = False
    staging_wakeup = None           # time of the pending "staging" event, if any
    lead = []
    now = 0.0
    remaining = len(requests)

    def schedule_engine(now):
        nonlocal engine_busy
        if engine_busy:
            return
        if rt.waiting and len(rt.running) < cal.max_active:
            head = rt.waiting[0]
            ready = True
            if head.keys:
                c = ctl.claims[head.rid]
                if not c["requested"]:
                    ctl.request_retrieval(head, now)
                st = tier.state(head.rid)
                ready = st == kvs.KVS_CLAIM_STAGE_READY or (
                    st == kvs.KVS_CLAIM_ORDINARY and all(k not in prov.done_at for k in head.keys))
            if ready:
                rt.waiting.popleft()
                rt.prefilling.append(head)
                head.admitted = now
                t_ret = 0.0
                if head.keys:
                    tier.begin_retrieval(head.rid, now, len(head.keys))
                    if head.rid in ctl.commit_times:
                        lead.append(now - ctl.commit_times[head.rid])
                    t_ret = cal.retrieval_s(head.matched)
                    push(now + t_ret, "retrieved", head)
                done = now + t_ret + cal.prefill_s(head.prompt - head.matched)
                engine_busy = True
                rt.busy_until = done
                push(done, "prefilled", head)
                ctl.update_ttus(now)
                return
        if rt.running:
            engine_busy = True
            rt.busy_until = now + cal.decode_step_s
            push(rt.busy_until, "decoded")
            ctl.update_ttus(now)

    while events:
        now, _, kind, payload = heapq.heappop(events)
        nxt = prov.next_completion()
        while nxt is not None and nxt <= now:           # staging completions up to now
            prov.complete_head(nxt)
            nxt = prov.next_completion()
        if kind == "arrival":
            r = payload
            rt.waiting.append(r)
            if r.keys:
                ctl.add(r, now)
            ctl.update_ttus(now)
        elif kind == "retrieved":
            tier.end_retrieval(payload.rid, now)
        elif kind == "prefilled":
            r = payload
            rt.prefilling.remove(r)
            r.first_token = now
            r.generated = 1
            engine_busy = False
            if r.generated >= r.output:
                r.finished = now
                est.add(r.output)
                remaining -= 1
            else:
                rt.running.append(r)
        elif kind == "decoded":
            engine_busy = False
            for r in list(rt.running):
                r.generated += 1
                if r.generated >= r.output:
                    r.finished = now
                    est.add(r.output)
                    rt.running.remove(r)
                    remaining -= 1
        elif kind == "tick":
            if remaining or prov.queue:
                push(now + cal.tick_s, "tick")
        if kind == "staging":
            staging_wakeup = None
        ctl.evaluate(now)
        schedule_engine(now)
        nxt = prov.next_completion()                    # wake up for the next staging completion
        if nxt is not None and staging_wakeup != nxt:
            push(nxt, "staging")
            staging_wakeup = nxt
    end = max(r.finished for r in requests)
    st = tier.stats(max(end, now))
    ttft = [r.first_token - r.arrival for r in requests]
    out_tok = sum(r.output for r in requests)
    first = min(r.arrival for r in requests)
    n_ord = sum(1 for r in requests if r.keys and tier.state(r.rid) == kvs.KVS_CLAIM_RELEASED
                and ctl.claims[r.rid]["ordinary"])
    res = Result(ttft=ttft, p95_ttft=float(np.percentile(ttft, 95)),
                 throughput_tok_s=out_tok / (end - first),
                 cost_gib_s_per_req=st["protected_object_seconds"] * cal.object_bytes / 2 ** 30 / len(requests),
                 blocked_attempts=ctl.blocked_attempts, ordinary=n_ord, staged_reads=st["staged_reads"],
                 commit_lead_s=lead, commit_times=dict(ctl.commit_times),
                 retrieval_starts={r.rid: r.admitted for r in requests if r.keys})
    tier.close()
    return res


def workload(ratio: float, n_docs: int = 12, interval: float = 0.5, seed: int = 0,
             cal: Calibration | None = None, lo: int = 16078, hi: int = 67744):
    """Synthetic stand-in for the paper's documents (Sec. 5.1): prompt lengths drawn
    between the paper's reported bounds, the prefix ratio applied to each document
    and rounded down to whole chunks, a short question appended, outputs up to the
    generation limit with early stops; request i arrives at i * interval."""
    cal = cal or Calibration()
    rng = np.random.default_rng(seed)
    reqs = []
    next_key = itertools.count(1)
    for i in range(n_docs):
        doc = int(rng.integers(lo, hi))
        question = int(rng.integers(16, 64))
        matched = int(doc * ratio) // cal.chunk_tokens * cal.chunk_tokens
        out = int(min(cal.gen_limit, rng.geometric(1 / 60)))
        keys = [next(next_key) for _ in range(matched // cal.chunk_tokens)]
        reqs.append(Request(i, i * interval, doc + question, matched, max(out, 1), keys))
    return reqs

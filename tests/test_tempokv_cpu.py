"""The TempoKV control-plane model (paper_2609_35065_gb300.tempokv) on the CPU:
closed forms for the output-length estimator, the TTR and TTU projections and
the laxity trigger, then invariants of whole simulated runs."""
import numpy as np
import pytest

from paper_2609_35065_gb300 import kvs, tempokv


def test_remaining_output_is_the_conditional_mean_bounded_by_the_limit():
    e = tempokv.OutputLengthEstimator(128, [10, 20, 30, 128])
    assert e.remaining(15) == pytest.approx((20 + 30 + 128) / 3 - 15)
    assert e.remaining(25) == pytest.approx((30 + 128) / 2 - 25)
    assert e.remaining(100) == pytest.approx(28)
    assert e.remaining(128) == 0                       # nothing longer: the limit bounds it
    assert tempokv.OutputLengthEstimator(128, [300]).remaining(10) == 118   # capped at the limit
    assert tempokv.OutputLengthEstimator(64).remaining(4) == 60             # no history yet


def _provider(cap=64, budget=32):
    cal = tempokv.Calibration(staging_gibs=1.0, kv_bytes_per_token=4 << 20)    # 1 GiB objects: 1 s each
    return tempokv.Provider(kvs.Tier(cap, budget, cal.object_bytes), cal), cal


def test_ttr_projection_closed_forms():
    p, cal = _provider()
    u = cal.object_bytes / (cal.staging_gibs * 2 ** 30)
    assert u == pytest.approx(1.0)
    assert p.ttr([1, 2, 3], 0.0) == pytest.approx(3 * u)          # empty queue: new reads only
    p.tier.commit(100, [10, 11, 12], 0.0)
    p.enqueue([10, 11, 12], 0.0)                                  # backlog completes at 1, 2, 3
    assert p.ttr([1, 2], 0.0) == pytest.approx(5 * u)             # behind the backlog
    assert p.ttr([11, 1], 0.0) == pytest.approx(4 * u)            # covered object + one new read
    assert p.ttr([10], 0.0) == pytest.approx(1 * u)               # no new read, still waits
    p.complete_head(1.0)                                          # object 10 is resident at t = 1
    assert p.ttr([10], 1.5) == 0.0                                # resident: protection only
    assert p.ttr([1], 1.5) == pytest.approx(3 * u + u - 1.5)


def test_ttu_projection_closed_forms():
    cal = tempokv.Calibration(max_active=1, decode_step_s=0.02, prefill_tok_s=1000.0,
                              retrieval_gbs=1.0, kv_bytes_per_token=1000)
    est = tempokv.OutputLengthEstimator(128, [100] * 5)          # remaining(n) = 100 - n
    rt = tempokv.Runtime(cal, est)
    running = tempokv.Request(0, 0.0, 10, 0, 100)
    running.generated = 40
    rt.running.append(running)
    target = tempokv.Request(1, 0.0, 3000, 2048, 10, keys=list(range(8)))
    rt.waiting.append(target)
    never = lambda r: 0.0
    assert rt.ttu(target, 0.0, never) == pytest.approx(60 * 0.02)        # the running one finishes
    ahead = tempokv.Request(2, 0.0, 2000, 1024, 10, keys=[99])
    rt.waiting.appendleft(ahead)
    cost_ahead = cal.retrieval_s(1024) + cal.prefill_s(2000 - 1024)
    # the request ahead is admitted after the running one, then decodes 100 tokens (estimate)
    assert rt.ttu(target, 0.0, never) == pytest.approx(60 * 0.02 + cost_ahead + 100 * 0.02)
    # a known retrieval dependency of the request ahead (its KV ready at t = 5 s) delays both
    assert rt.ttu(target, 0.0, lambda r: 5.0 if r is ahead else 0.0) == pytest.approx(5.0 + cost_ahead + 2.0)


def test_commitment_happens_when_laxity_reaches_zero():
    """A predecessor with known remaining work keeps the target waiting; TTU falls by one
    second per second and TTR is constant, so the claim commits at TTU0 - TTR (within a
    control interval) and its KV is ready just as retrieval begins."""
    cal = tempokv.Calibration(max_active=1, decode_step_s=0.02, staging_gibs=11.0)
    pred = tempokv.Request(0, 0.0, 256, 0, 100)                  # 100 decode steps = 2 s
    target = tempokv.Request(1, 0.01, 16384 + 20, 16384, 10, keys=list(range(1, 65)))
    res = tempokv.simulate([pred, target], cal, history=[100] * 5)
    ttr = 64 * cal.object_bytes / (cal.staging_gibs * 2 ** 30)    # 64 objects of 32 MiB: ~0.18 s
    retrieval_start = res.retrieval_starts[1]
    assert res.commit_times[1] == pytest.approx(retrieval_start - ttr, abs=0.05)
    assert retrieval_start == pytest.approx(2.0 + cal.prefill_s(256), abs=0.03)
    assert res.blocked_attempts == 0 and res.ordinary == 0


def test_simulated_runs_are_complete_consistent_and_deterministic():
    cal = tempokv.Calibration()
    reqs = tempokv.workload(0.75, cal=cal, seed=3)
    res = tempokv.simulate(reqs, cal)
    assert all(r.finished is not None for r in reqs)
    for r in reqs:
        assert r.first_token - r.arrival >= cal.retrieval_s(r.matched) + cal.prefill_s(r.prompt - r.matched) - 1e-9
        assert res.retrieval_starts[r.rid] >= res.commit_times.get(r.rid, 0.0)
    assert res.staged_reads == sum(len(r.keys) for r in reqs)      # one read per object
    again = tempokv.simulate(tempokv.workload(0.75, cal=cal, seed=3), cal)
    assert again.ttft == res.ttft and again.cost_gib_s_per_req == res.cost_gib_s_per_req


def test_tight_budget_defers_commitment_and_falls_back_to_ordinary_retrieval():
    cal = tempokv.Calibration()
    reqs = tempokv.workload(1.0, cal=cal, seed=1, interval=0.05)
    res = tempokv.simulate(reqs, cal, capacity_gib=40.0, budget_gib=12.0)
    assert res.blocked_attempts > 0 and res.ordinary > 0
    assert all(r.finished is not None for r in reqs)
    # protection never exceeds the budget, so C is bounded by budget x run length / N
    run = max(r.finished for r in reqs)
    assert res.cost_gib_s_per_req <= 12.0 * run / len(reqs) + 1e-9

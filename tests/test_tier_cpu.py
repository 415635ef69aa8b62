"""The fast tier's object ledger (kvs_tier_*, C++) without a GPU.

Closed-form cases pin the rules of TempoKV Sec. 3.2 / Sec. 5 (protected-capacity
budget, shared objects counted once, coalesced staging, LRU eviction of
unprotected entries, cancellation, the ordinary path, C = integral P dt / N);
random operation sequences then compare the ledger with the independent
Python model in ``oracle/tier_model.py`` after every operation.
"""
import numpy as np
import pytest

from oracle.tier_model import TierModel
from paper_2609_35065_gb300 import kvs

S = kvs.KVS_CLAIM_STAGING
R = kvs.KVS_CLAIM_STAGE_READY


def test_cost_of_one_claim_is_objects_times_protected_time():
    t = kvs.Tier(10, 5, 1 << 20)
    assert sorted(t.commit(1, [7, 8, 9], 2.0)) == [7, 8, 9]
    for k in (7, 8, 9):
        t.staged(k, 3.5)
    t.begin_retrieval(1, 4.0, 3)
    t.end_retrieval(1, 6.0)
    st = t.stats(10.0)
    assert st["protected_object_seconds"] == pytest.approx(3 * (6.0 - 2.0))
    assert st["completed"] == 1 and st["protected_objects"] == 0 and st["resident"] == 3
    # C in GiB.s per request: 3 objects of 1 MiB protected for 4 s, one request
    assert st["protected_object_seconds"] * t.object_bytes / 2 ** 30 / st["completed"] == pytest.approx(12 / 1024)


def test_shared_objects_are_counted_once():
    t = kvs.Tier(10, 6, 1)
    t.commit(1, [1, 2, 3], 0.0)
    assert t.commit(2, [3, 4], 5.0) == [4]            # object 3 is coalesced: no second read
    for k in (1, 2, 3, 4):
        t.staged(k, 5.0)
    t.begin_retrieval(1, 9.0, 3)
    t.end_retrieval(1, 10.0)
    t.begin_retrieval(2, 15.0, 2)
    t.end_retrieval(2, 20.0)
    st = t.stats(30.0)
    # objects 1, 2: [0, 10]; object 3: [0, 20] (held by either claim); object 4: [5, 20]
    assert st["protected_object_seconds"] == pytest.approx(2 * 10 + 20 + 15)
    assert st["staged_reads"] == 4 and st["completed"] == 2


def test_budget_counts_only_bytes_not_already_protected():
    t = kvs.Tier(10, 4, 1)
    t.commit(1, [1, 2, 3], 0.0)
    with pytest.raises(kvs.KvsError) as ei:
        t.commit(2, [3, 4, 5], 1.0)                   # 3 protected + 2 new > 4
    assert ei.value.code == kvs.KVS_ERR_NOMEM and t.state(2) == kvs.KVS_CLAIM_PLANNED
    assert t.commit(3, [3, 4], 1.0) == [4]            # 3 + 1 <= 4: fits
    assert t.stats(1.0)["protected_objects"] == 4
    for k in (1, 2, 3, 4):
        t.staged(k, 2.0)
    t.begin_retrieval(1, 2.0, 3)
    t.end_retrieval(1, 3.0)                           # 1, 2 released; 3, 4 still protected
    assert t.commit(2, [3, 4, 5], 3.0) == [5]         # retried Planned claim now fits
    assert t.state(2) == S


def test_commit_on_resident_objects_is_stage_ready_at_once():
    t = kvs.Tier(6, 3, 1)
    t.commit(1, [1, 2], 0.0)
    t.staged(1, 1.0)
    assert t.state(1) == S
    t.staged(2, 1.5)
    assert t.state(1) == R
    t.begin_retrieval(1, 2.0, 2)
    t.end_retrieval(1, 2.5)
    assert t.commit(2, [2, 1], 3.0) == [] and t.state(2) == R   # resident: protect, no I/O


def test_lru_eviction_takes_the_least_recently_used_unprotected_object():
    t = kvs.Tier(3, 2, 1)
    for cid, k in ((1, 10), (2, 11), (3, 12)):
        t.commit(cid, [k], float(cid))
        t.staged(k, float(cid))
        t.begin_retrieval(cid, float(cid), 1)
        t.end_retrieval(cid, float(cid))
    t.commit(4, [10], 5.0)                            # touch 10 again
    t.begin_retrieval(4, 5.0, 1)
    t.end_retrieval(4, 5.0)
    assert t.commit(5, [13], 6.0) == [13]             # LRU is now 11
    assert t.object(11) is None and t.object(10) is not None and t.object(12) is not None
    assert t.object(13)["slot"] == 1                  # 11's slot
    assert t.stats(6.0)["evictions"] == 1


def test_protected_and_in_use_objects_are_never_evicted():
    t = kvs.Tier(3, 2, 1)
    t.commit(1, [1, 2], 0.0)                          # two protected objects
    t.ordinary(9, [3], 0.0)                           # third slot held by a demand fetch
    with pytest.raises(kvs.KvsError) as ei:
        t.ordinary(10, [4], 1.0)                      # no free or evictable slot left
    assert ei.value.code == kvs.KVS_ERR_NOMEM
    for k in (1, 2, 3):
        assert t.object(k) is not None


def test_cancel_keeps_protection_until_io_and_gpu_access_end():
    t = kvs.Tier(8, 6, 1)
    t.commit(1, [1, 2], 0.0)
    t.cancel(1, 1.0)                                  # staging I/O outstanding
    assert t.stats(1.0)["protected_objects"] == 2 and t.state(1) == S
    t.staged(1, 2.0)
    assert t.stats(2.0)["protected_objects"] == 2
    t.staged(2, 3.0)                                  # last I/O done: protection ends
    assert t.state(1) == kvs.KVS_CLAIM_CANCELLED and t.stats(3.0)["protected_objects"] == 0
    t.commit(2, [1], 4.0)
    t.begin_retrieval(2, 4.0, 1)
    t.cancel(2, 5.0)                                  # GPU access in progress
    assert t.stats(5.0)["protected_objects"] == 1
    t.end_retrieval(2, 6.0)
    assert t.state(2) == kvs.KVS_CLAIM_CANCELLED and t.stats(6.0)["completed"] == 0
    t.commit(3, [5], 7.0)
    with pytest.raises(kvs.KvsError):
        t.cancel(4, 7.0)                              # unknown claim
    t.commit(4, [6], 7.0)
    t.cancel(3, 8.0)
    st = t.stats(9.0)
    # objects 1, 2: [0, 3]; object 1 again: [4, 6]; object 5 (cancelled while staging): [7, 9];
    # object 6: [7, 9]
    assert st["protected_object_seconds"] == pytest.approx(2 * 3 + 2 + 2 + 2)


def test_ordinary_path_reserves_nothing_and_excludes_commitment():
    t = kvs.Tier(6, 1, 1)
    with pytest.raises(kvs.KvsError):
        t.commit(1, [1, 2], 0.0)                      # over budget: Planned
    assert t.ordinary(1, [1, 2], 0.0) == [1, 2]       # the ordinary path takes it
    assert t.state(1) == kvs.KVS_CLAIM_ORDINARY
    with pytest.raises(kvs.KvsError) as ei:
        t.commit(1, [1], 1.0)
    assert ei.value.code == kvs.KVS_ERR_INVALID_ARG
    t.staged(1, 1.0)
    t.staged(2, 1.0)
    t.begin_retrieval(1, 2.0, 2)
    t.end_retrieval(1, 3.0)
    st = t.stats(4.0)
    assert st["protected_object_seconds"] == 0 and st["completed"] == 1
    assert t.object(1)["gpu_refs"] == 0 and t.object(1)["pins"] == 0


def test_invalid_operations():
    t = kvs.Tier(4, 2, 1)
    with pytest.raises(kvs.KvsError):
        t.commit(1, [1, 1], 0.0)                      # duplicate object
    with pytest.raises(kvs.KvsError):
        t.staged(5, 0.0)                              # not staging
    t.commit(2, [1], 1.0)
    with pytest.raises(kvs.KvsError):
        t.begin_retrieval(2, 1.0, 1)                  # not StageReady yet
    with pytest.raises(kvs.KvsError):
        t.stats(0.5)                                  # time went backwards
    with pytest.raises(kvs.KvsError):
        kvs.Tier(4, 4, 1)                             # budget must be below capacity


# ---------------------------------------------------------------------------
# Random sequences: ledger vs model after every operation
# ---------------------------------------------------------------------------
def _compare(t, m, keys, claims):
    for k in keys:
        got = t.object(k)
        want = m.objs.get(k)
        if want is None:
            assert got is None, k
        else:
            assert got is not None, k
            for f in ("slot", "pins", "gpu_refs", "lru"):
                assert got[f] == want[f], (k, f, got, want)
            assert bool(got["staging"]) == want["staging"] and bool(got["resident"]) == want["resident"]
    for c in claims:
        assert t.state(c) == m.state(c), (c, t.state(c), m.state(c))


def _code(e):
    return {kvs.KVS_ERR_NOMEM: "nomem"}.get(e.code, "invalid")


@pytest.mark.parametrize("seed", range(20))
def test_random_sequences_match_the_model(seed):
    rng = np.random.default_rng(seed)
    cap = int(rng.integers(3, 10))
    budget = int(rng.integers(1, cap))
    universe = list(range(100, 100 + int(rng.integers(cap, 3 * cap))))
    t, m = kvs.Tier(cap, budget, 4096), TierModel(cap, budget)
    now, next_claim = 0.0, 1
    claims = []
    for _ in range(300):
        now += float(rng.choice([0.0, 0.25, 1.0]))
        op = rng.choice(["commit", "retry", "staged", "begin", "end", "cancel", "ordinary", "bad"])
        if op in ("commit", "ordinary", "retry"):
            if op == "retry":
                planned = [c for c in claims if m.state(c) == 1]
                if not planned:
                    continue
                cid = int(rng.choice(planned))
                op = "commit" if rng.random() < 0.6 else "ordinary"
            else:
                cid = next_claim
                next_claim += 1
                claims.append(cid)
            keys = [int(x) for x in rng.choice(universe, size=int(rng.integers(1, min(4, len(universe)) + 1)),
                                               replace=False)]
            want, want_stage = getattr(m, op)(cid, keys, now)
            try:
                got_stage = getattr(t, op)(cid, keys, now)
                got = "ok"
            except kvs.KvsError as e:
                got, got_stage = _code(e), []
            assert (got, got_stage) == (want, want_stage), (op, cid, keys)
        elif op == "staged":
            staging = sorted(k for k, o in m.objs.items() if o["staging"])
            if not staging:
                continue
            k = int(rng.choice(staging))
            assert m.staged(k, now) == "ok"
            t.staged(k, now)
        elif op in ("begin", "end", "cancel"):
            if not claims:
                continue
            cid = int(rng.choice(claims))
            want = getattr(m, {"begin": "begin_retrieval", "end": "end_retrieval", "cancel": "cancel"}[op])(cid, now)
            want = want[0] if isinstance(want, tuple) else want
            try:
                if op == "begin":
                    t.begin_retrieval(cid, now, len(m.claims.get(cid, {"keys": []})["keys"]))
                elif op == "end":
                    t.end_retrieval(cid, now)
                else:
                    t.cancel(cid, now)
                got = "ok"
            except kvs.KvsError as e:
                got = _code(e)
            assert got == want, (op, cid)
        else:                                           # an operation that must be refused
            k = 10 ** 6 + int(rng.integers(0, 5))
            with pytest.raises(kvs.KvsError):
                t.staged(k, now)
            assert m.staged(k, now) == "invalid"
        _compare(t, m, universe, claims)
        st, sm = t.stats(now), m.stats(now)
        for f in ("resident", "staging", "protected_objects", "free_slots", "evictions", "staged_reads", "completed"):
            assert st[f] == sm[f], (f, st, sm)
        assert st["protected_object_seconds"] == pytest.approx(sm["protected_object_seconds"], rel=1e-12, abs=1e-9)
        assert st["protected_objects"] <= budget

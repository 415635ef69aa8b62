"""Reference model of the fast tier's object ledger (TempoKV Sec. 3.2, Sec. 4, Sec. 5).

TEST INFRASTRUCTURE ONLY: used by the tests to check the C++ ledger
(``kvs_tier_*``) operation by operation.  Written from the paper's rules with
plain lists and dictionaries, sharing nothing with the C++ code:

* the fast tier has ``capacity`` slots; protected staging and ordinary caching
  share them; a protected-capacity budget below capacity counts protected
  objects and reservations for outstanding staging, each object once (Sec. 3.2,
  "Protected capacity and on-demand retrieval");
* committing a claim protects every object of its manifest; objects not in the
  tier are staged, and an object already being staged is not staged twice; the
  claim must fit the budget with the bytes not already protected by another
  claim, else it stays Planned (Sec. 3.2, "Commitment and replanning",
  "Shared staging and resource lifecycle");
* Planned -> Staging, or StageReady when every object is already resident;
  Staging -> StageReady when the last object arrives; Transferring when the
  retrieval begins; protection ends when the GPU retrieval completes (Released);
  Released ends protection, not residency (Sec. 3.2, last paragraphs);
* a committed claim that is cancelled keeps its protection until its
  outstanding staging and GPU accesses end (Sec. 3.2);
* the ordinary path reserves nothing and excludes commitment (Sec. 3.2);
* unprotected entries are evicted least-recently-used first (Sec. 5 setup);
* C = (integral of P(t) dt) / N, P counting each protected object once (Sec. 5,
  Metrics).

Slot choice is fixed so that two implementations can be compared step by step:
the lowest free slot, else the slot of the least recently used evictable object
(last-use stamps come from one counter, advanced when an object arrives and
when a retrieval touches it).
"""
from __future__ import annotations

PLANNED, STAGING, STAGE_READY, TRANSFERRING, RELEASED, CANCELLED, ORDINARY = 1, 2, 3, 4, 5, 6, 7


class TierModel:
    def __init__(self, capacity: int, budget: int):
        assert 0 <= budget < capacity
        self.capacity, self.budget = capacity, budget
        self.free = list(range(capacity))              # kept sorted
        self.objs = {}          # key -> dict(slot, pins, staging, resident, gpu_refs, lru)
        self.claims = {}        # id -> dict(keys, state, pending, committed, cancel_pending, in_gpu)
        self.clock = 0
        self.t = 0.0
        self.area = 0.0         # integral of P(t) dt, object-seconds
        self.evictions = self.staged_reads = self.completed = 0

    # ---- helpers ---------------------------------------------------------
    def protected(self) -> int:
        return sum(1 for o in self.objs.values() if o["pins"] > 0)

    def _advance(self, now):
        if now < self.t:
            raise ValueError("time went backwards")
        self.area += self.protected() * (now - self.t)
        self.t = now

    @staticmethod
    def _evictable(o):
        return o["resident"] and not o["staging"] and o["pins"] == 0 and o["gpu_refs"] == 0

    def _lru_order(self):
        return sorted((o["lru"], k) for k, o in self.objs.items() if self._evictable(o))

    def _slot(self):
        if self.free:
            return self.free.pop(0)
        _, victim = self._lru_order()[0]
        slot = self.objs.pop(victim)["slot"]
        self.evictions += 1
        return slot

    def _obtainable(self, keys):
        own = sum(1 for k in keys if k in self.objs and self._evictable(self.objs[k]))
        return len(self.free) + len(self._lru_order()) - own

    def _touch(self, k):
        self.clock += 1
        self.objs[k]["lru"] = self.clock

    def _new_obj(self, pins, gpu_refs):
        return {"slot": self._slot(), "pins": pins, "staging": True, "resident": False,
                "gpu_refs": gpu_refs, "lru": 0}

    # ---- operations --------------------------------------------------------
    def commit(self, cid, keys, now):
        """Returns ("ok", keys to stage) or ("nomem", []) or ("invalid", [])."""
        self._advance(now)
        c = self.claims.get(cid)
        if c is not None and c["state"] != PLANNED:
            return "invalid", []
        if len(set(keys)) != len(keys):
            return "invalid", []
        c = self.claims[cid] = {"keys": list(keys), "state": PLANNED, "pending": 0, "committed": False,
                                "cancel_pending": False, "in_gpu": False}
        additional = sum(1 for k in keys if k not in self.objs or self.objs[k]["pins"] == 0)
        if self.protected() + additional > self.budget:
            return "nomem", []
        missing = [k for k in keys if k not in self.objs]
        if len(missing) > self._obtainable(keys):
            return "nomem", []
        for k in keys:
            if k in self.objs:
                self.objs[k]["pins"] += 1
        staged = []
        for k in missing:
            self.objs[k] = self._new_obj(pins=1, gpu_refs=0)
            self.staged_reads += 1
            staged.append(k)
        c["pending"] = sum(1 for k in keys if self.objs[k]["staging"])
        c["committed"] = True
        c["state"] = STAGING if c["pending"] else STAGE_READY
        return "ok", staged

    def staged(self, key, now):
        self._advance(now)
        o = self.objs.get(key)
        if o is None or not o["staging"]:
            return "invalid"
        o["staging"], o["resident"] = False, True
        self._touch(key)
        for cid in sorted(self.claims):
            c = self.claims[cid]
            if c["pending"] == 0 or key not in c["keys"]:
                continue
            c["pending"] -= 1
            if c["pending"]:
                continue
            if c["cancel_pending"] and not c["in_gpu"]:
                if c["committed"]:
                    self._unpin_all(c)
                else:
                    for k in c["keys"]:
                        self.objs[k]["gpu_refs"] -= 1
                c["state"] = CANCELLED
            elif c["state"] == STAGING:
                c["state"] = STAGE_READY
        return "ok"

    def _unpin_all(self, c):
        if c["committed"]:
            for k in c["keys"]:
                self.objs[k]["pins"] -= 1
            c["committed"] = False

    def begin_retrieval(self, cid, now):
        self._advance(now)
        c = self.claims.get(cid)
        if c is None:
            return "invalid", []
        ordinary_ready = (c["state"] == ORDINARY and c["pending"] == 0 and not c["in_gpu"]
                          and not c["cancel_pending"])
        if c["state"] != STAGE_READY and not ordinary_ready:
            return "invalid", []
        slots = []
        for k in c["keys"]:
            if c["committed"]:
                self.objs[k]["gpu_refs"] += 1
            self._touch(k)
            slots.append(self.objs[k]["slot"])
        c["in_gpu"] = True
        if c["committed"]:
            c["state"] = TRANSFERRING
        return "ok", slots

    def end_retrieval(self, cid, now):
        self._advance(now)
        c = self.claims.get(cid)
        if c is None or not c["in_gpu"]:
            return "invalid"
        for k in c["keys"]:
            self.objs[k]["gpu_refs"] -= 1
        c["in_gpu"] = False
        self._unpin_all(c)
        if c["cancel_pending"]:
            c["state"] = CANCELLED
        else:
            c["state"] = RELEASED
            self.completed += 1
        return "ok"

    def cancel(self, cid, now):
        self._advance(now)
        c = self.claims.get(cid)
        if c is None:
            return "invalid"
        if c["state"] in (PLANNED, STAGE_READY):
            self._unpin_all(c)
            c["state"] = CANCELLED
        elif c["state"] in (STAGING, TRANSFERRING):
            c["cancel_pending"] = True
        elif c["state"] == ORDINARY:
            if c["in_gpu"] or c["pending"]:
                c["cancel_pending"] = True
            else:
                for k in c["keys"]:
                    self.objs[k]["gpu_refs"] -= 1
                c["state"] = CANCELLED
        else:
            return "invalid"
        return "ok"

    def ordinary(self, cid, keys, now):
        self._advance(now)
        c = self.claims.get(cid)
        if c is not None and c["state"] != PLANNED:
            return "invalid", []
        if len(set(keys)) != len(keys):
            return "invalid", []
        missing = [k for k in keys if k not in self.objs]
        if len(missing) > self._obtainable(keys):
            return "nomem", []
        c = self.claims[cid] = {"keys": list(keys), "state": ORDINARY, "pending": 0, "committed": False,
                                "cancel_pending": False, "in_gpu": False}
        for k in keys:
            if k in self.objs:
                self.objs[k]["gpu_refs"] += 1
        staged = []
        for k in missing:
            self.objs[k] = self._new_obj(pins=0, gpu_refs=1)
            self.staged_reads += 1
            staged.append(k)
        c["pending"] = sum(1 for k in keys if self.objs[k]["staging"])
        return "ok", staged

    def state(self, cid):
        c = self.claims.get(cid)
        return 0 if c is None else c["state"]

    def stats(self, now):
        self._advance(now)
        return {"resident": sum(1 for o in self.objs.values() if o["resident"]),
                "staging": sum(1 for o in self.objs.values() if o["staging"]),
                "protected_objects": self.protected(), "free_slots": len(self.free),
                "evictions": self.evictions, "staged_reads": self.staged_reads,
                "completed": self.completed, "protected_object_seconds": self.area}

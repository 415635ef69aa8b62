// kvs_tier.cpp -- the fast tier's object ledger: protection, coalesced staging,
// protected-capacity budget, LRU eviction of unprotected entries, claim
// lifecycle and the protected-capacity cost (TempoKV Sec. 3.2, Sec. 4, Sec. 5).
//
// One object = one KV chunk in one slot.  An object is protected while any
// claim pins it; P(t) counts protected objects (a staging reservation of a
// committed claim is a pinned, not yet resident object), each once.  An
// object is evictable while resident, unpinned, not staging and not read by a
// retrieval; the evictable set is ordered by a logical last-use clock.
#include <algorithm>
#include <cstdint>
#include <cstring>
#include <map>
#include <set>
#include <unordered_map>
#include <unordered_set>
#include <vector>

#include <cuda_runtime.h>

#include "kvs.h"
#include "kvs_internal.h"

namespace {

struct Obj {
    int64_t  slot = -1;
    int32_t  pins = 0;
    bool     staging = false;
    bool     resident = false;
    int32_t  gpu_refs = 0;
    uint64_t lru = 0;
};

struct Claim {
    std::vector<uint64_t> keys;
    int      state = KVS_CLAIM_NONE;
    int32_t  pending = 0;          // manifest objects whose staging is outstanding
    bool     committed = false;    // holds pins on its objects
    bool     cancel_pending = false;
    bool     in_gpu = false;       // a retrieval reads its objects
};

int fail(int code, const char* msg) {
    kvs::set_last_error(msg);
    return code;
}

}  // namespace

struct kvs_tier {
    kvs_tier_config cfg{};
    uint8_t* arena = nullptr;
    std::unordered_map<uint64_t, Obj> objs;
    std::map<uint64_t, Claim> claims;
    std::set<int64_t> free_slots;
    std::set<std::pair<uint64_t, uint64_t>> evictable;   // (lru stamp, key)
    uint64_t clock = 0;
    int64_t protected_count = 0, staging_count = 0, resident_count = 0;
    int64_t evictions = 0, staged_reads = 0, completed = 0;
    double last_t = 0, integral = 0;

    bool advance(double now) {
        if (now < last_t) return false;
        integral += (double)protected_count * (now - last_t);
        last_t = now;
        return true;
    }
    static bool is_evictable(const Obj& o) {
        return o.resident && !o.staging && o.pins == 0 && o.gpu_refs == 0;
    }
    // Re-files `key` in the evictable set after any change of its state.
    void refresh(uint64_t key, Obj& o, uint64_t old_stamp) {
        evictable.erase({old_stamp, key});
        if (is_evictable(o)) evictable.insert({o.lru, key});
    }
    void touch(uint64_t key, Obj& o) {
        const uint64_t old = o.lru;
        o.lru = ++clock;
        refresh(key, o, old);
    }
    void pin(uint64_t key, Obj& o) {
        if (o.pins++ == 0) ++protected_count;
        refresh(key, o, o.lru);
    }
    void unpin(uint64_t key, Obj& o) {
        if (--o.pins == 0) --protected_count;
        refresh(key, o, o.lru);
    }
    // A slot for a new object: the lowest free one, else the least recently
    // used evictable object's (that object leaves the tier).
    int64_t take_slot() {
        if (!free_slots.empty()) {
            const int64_t s = *free_slots.begin();
            free_slots.erase(free_slots.begin());
            return s;
        }
        const auto victim = *evictable.begin();
        evictable.erase(evictable.begin());
        auto it = objs.find(victim.second);
        const int64_t s = it->second.slot;
        objs.erase(it);
        --resident_count;
        ++evictions;
        return s;
    }
    // Slots obtainable without touching `keys`' own objects.
    int64_t obtainable(const std::vector<uint64_t>& keys) const {
        int64_t own = 0;
        for (uint64_t k : keys) {
            auto it = objs.find(k);
            if (it != objs.end() && is_evictable(it->second)) ++own;
        }
        return (int64_t)free_slots.size() + (int64_t)evictable.size() - own;
    }
    void finish_claim(Claim& c) {                 // drop the claim's pins
        if (!c.committed) return;
        for (uint64_t k : c.keys) unpin(k, objs.at(k));
        c.committed = false;
    }
};

namespace {

bool distinct(const uint64_t* keys, int32_t n, std::vector<uint64_t>& out) {
    std::unordered_set<uint64_t> seen;
    out.assign(keys, keys + n);
    for (uint64_t k : out)
        if (!seen.insert(k).second) return false;
    return true;
}

}  // namespace

extern "C" {

int kvs_tier_create(const kvs_tier_config* cfg, kvs_tier** out) {
    if (!cfg || !out) return fail(KVS_ERR_INVALID_ARG, "cfg and out must not be NULL");
    if (cfg->capacity_objects <= 0 || cfg->budget_objects < 0 || cfg->budget_objects >= cfg->capacity_objects ||
        cfg->object_bytes <= 0)
        return fail(KVS_ERR_INVALID_ARG, "need 0 <= budget_objects < capacity_objects and object_bytes > 0");
    kvs_tier* t = new kvs_tier;
    t->cfg = *cfg;
    if (cfg->arena) {
        void* p = nullptr;
        if (cudaHostAlloc(&p, (size_t)cfg->capacity_objects * (size_t)cfg->object_bytes, cudaHostAllocDefault)
            != cudaSuccess) {
            cudaGetLastError();
            delete t;
            return fail(KVS_ERR_NOMEM, "cannot allocate the pinned fast-tier arena");
        }
        t->arena = (uint8_t*)p;
    }
    for (int64_t s = 0; s < cfg->capacity_objects; ++s) t->free_slots.insert(t->free_slots.end(), s);
    *out = t;
    return KVS_OK;
}

int kvs_tier_destroy(kvs_tier* t) {
    if (!t) return KVS_OK;
    if (t->arena) cudaFreeHost(t->arena);
    delete t;
    return KVS_OK;
}

int kvs_tier_commit(kvs_tier* t, uint64_t claim, const uint64_t* keys, int32_t n, double now,
                    uint64_t* stage_keys, int32_t* n_stage) {
    if (!t || n < 0 || (n > 0 && (!keys || !stage_keys)) || !n_stage)
        return fail(KVS_ERR_INVALID_ARG, "bad arguments");
    if (!t->advance(now)) return fail(KVS_ERR_INVALID_ARG, "time went backwards");
    *n_stage = 0;
    auto ci = t->claims.find(claim);
    if (ci != t->claims.end() && ci->second.state != KVS_CLAIM_PLANNED)
        return fail(KVS_ERR_INVALID_ARG, "only a new or Planned claim can be committed");
    std::vector<uint64_t> ks;
    if (!distinct(keys, n, ks)) return fail(KVS_ERR_INVALID_ARG, "a manifest names an object twice");
    Claim& c = t->claims[claim];
    c.keys = ks;
    c.state = KVS_CLAIM_PLANNED;
    // Budget: objects not already protected by another claim are the additional footprint.
    int64_t additional = 0, missing = 0;
    for (uint64_t k : ks) {
        auto it = t->objs.find(k);
        if (it == t->objs.end()) { ++additional; ++missing; }
        else if (it->second.pins == 0) ++additional;
    }
    if (t->protected_count + additional > t->cfg.budget_objects)
        return fail(KVS_ERR_NOMEM, "protected-capacity budget exceeded: the claim stays Planned");
    if (missing > t->obtainable(ks))
        return fail(KVS_ERR_NOMEM, "no slot can be freed: the claim stays Planned");
    for (uint64_t k : ks) {                    // protect what is already in the tier ...
        auto it = t->objs.find(k);
        if (it != t->objs.end()) t->pin(k, it->second);
    }
    for (uint64_t k : ks) {                    // ... then stage the rest (coalesced per object)
        if (t->objs.count(k)) continue;
        Obj o;
        o.slot = t->take_slot();
        o.staging = true;
        t->objs[k] = o;
        t->pin(k, t->objs[k]);
        ++t->staging_count;
        ++t->staged_reads;
        stage_keys[(*n_stage)++] = k;
    }
    c.pending = 0;
    for (uint64_t k : ks) c.pending += t->objs.at(k).staging ? 1 : 0;
    c.committed = true;
    c.state = c.pending ? KVS_CLAIM_STAGING : KVS_CLAIM_STAGE_READY;
    return KVS_OK;
}

int kvs_tier_staged(kvs_tier* t, uint64_t key, double now) {
    if (!t) return fail(KVS_ERR_INVALID_ARG, "tier is NULL");
    if (!t->advance(now)) return fail(KVS_ERR_INVALID_ARG, "time went backwards");
    auto it = t->objs.find(key);
    if (it == t->objs.end() || !it->second.staging) return fail(KVS_ERR_INVALID_ARG, "object is not staging");
    Obj& o = it->second;
    o.staging = false;
    o.resident = true;
    --t->staging_count;
    ++t->resident_count;
    t->touch(key, o);
    for (auto& [id, c] : t->claims) {
        if (c.pending == 0 || std::find(c.keys.begin(), c.keys.end(), key) == c.keys.end()) continue;
        if (--c.pending > 0) continue;
        if (c.cancel_pending && !c.in_gpu) {   // cancelled while staging: protection ends now
            if (c.committed) {
                t->finish_claim(c);
            } else {                          // ordinary: drop the holds on its objects
                for (uint64_t k : c.keys) {
                    Obj& h = t->objs.at(k);
                    --h.gpu_refs;
                    t->refresh(k, h, h.lru);
                }
            }
            c.state = KVS_CLAIM_CANCELLED;
        } else if (c.state == KVS_CLAIM_STAGING) {
            c.state = KVS_CLAIM_STAGE_READY;
        }
    }
    return KVS_OK;
}

int kvs_tier_begin_retrieval(kvs_tier* t, uint64_t claim, double now, int64_t* slots_out) {
    if (!t) return fail(KVS_ERR_INVALID_ARG, "tier is NULL");
    if (!t->advance(now)) return fail(KVS_ERR_INVALID_ARG, "time went backwards");
    auto ci = t->claims.find(claim);
    if (ci == t->claims.end()) return fail(KVS_ERR_INVALID_ARG, "unknown claim");
    Claim& c = ci->second;
    const bool ordinary_ready = c.state == KVS_CLAIM_ORDINARY && c.pending == 0 && !c.in_gpu && !c.cancel_pending;
    if (c.state != KVS_CLAIM_STAGE_READY && !ordinary_ready)
        return fail(KVS_ERR_INVALID_ARG, "retrieval needs a StageReady claim (or a fetched ordinary one)");
    for (size_t i = 0; i < c.keys.size(); ++i) {
        Obj& o = t->objs.at(c.keys[i]);
        if (c.committed) ++o.gpu_refs;         // ordinary claims hold their refs already
        t->touch(c.keys[i], o);
        if (slots_out) slots_out[i] = o.slot;
    }
    c.in_gpu = true;
    if (c.committed) c.state = KVS_CLAIM_TRANSFERRING;
    return KVS_OK;
}

int kvs_tier_end_retrieval(kvs_tier* t, uint64_t claim, double now) {
    if (!t) return fail(KVS_ERR_INVALID_ARG, "tier is NULL");
    if (!t->advance(now)) return fail(KVS_ERR_INVALID_ARG, "time went backwards");
    auto ci = t->claims.find(claim);
    if (ci == t->claims.end() || !ci->second.in_gpu) return fail(KVS_ERR_INVALID_ARG, "no retrieval in progress");
    Claim& c = ci->second;
    for (uint64_t k : c.keys) {
        Obj& o = t->objs.at(k);
        --o.gpu_refs;
        t->refresh(k, o, o.lru);
    }
    c.in_gpu = false;
    t->finish_claim(c);
    if (c.cancel_pending) {
        c.state = KVS_CLAIM_CANCELLED;
    } else {
        c.state = KVS_CLAIM_RELEASED;
        ++t->completed;
    }
    return KVS_OK;
}

int kvs_tier_cancel(kvs_tier* t, uint64_t claim, double now) {
    if (!t) return fail(KVS_ERR_INVALID_ARG, "tier is NULL");
    if (!t->advance(now)) return fail(KVS_ERR_INVALID_ARG, "time went backwards");
    auto ci = t->claims.find(claim);
    if (ci == t->claims.end()) return fail(KVS_ERR_INVALID_ARG, "unknown claim");
    Claim& c = ci->second;
    switch (c.state) {
        case KVS_CLAIM_PLANNED:
        case KVS_CLAIM_STAGE_READY:
            t->finish_claim(c);
            c.state = KVS_CLAIM_CANCELLED;
            return KVS_OK;
        case KVS_CLAIM_STAGING:
        case KVS_CLAIM_TRANSFERRING:
            c.cancel_pending = true;              // protection stays until the I/O or GPU access ends
            return KVS_OK;
        case KVS_CLAIM_ORDINARY:
            if (c.in_gpu || c.pending) { c.cancel_pending = true; return KVS_OK; }
            for (uint64_t k : c.keys) {           // fetched, never read: drop the holds
                Obj& o = t->objs.at(k);
                --o.gpu_refs;
                t->refresh(k, o, o.lru);
            }
            c.state = KVS_CLAIM_CANCELLED;
            return KVS_OK;
        default:
            return fail(KVS_ERR_INVALID_ARG, "claim already released or cancelled");
    }
}

int kvs_tier_ordinary(kvs_tier* t, uint64_t claim, const uint64_t* keys, int32_t n, double now,
                      uint64_t* stage_keys, int32_t* n_stage) {
    if (!t || n < 0 || (n > 0 && (!keys || !stage_keys)) || !n_stage)
        return fail(KVS_ERR_INVALID_ARG, "bad arguments");
    if (!t->advance(now)) return fail(KVS_ERR_INVALID_ARG, "time went backwards");
    *n_stage = 0;
    auto ci = t->claims.find(claim);
    if (ci != t->claims.end() && ci->second.state != KVS_CLAIM_PLANNED)
        return fail(KVS_ERR_INVALID_ARG, "the ordinary path excludes a committed claim");
    std::vector<uint64_t> ks;
    if (!distinct(keys, n, ks)) return fail(KVS_ERR_INVALID_ARG, "a manifest names an object twice");
    int64_t missing = 0;
    for (uint64_t k : ks) missing += t->objs.count(k) ? 0 : 1;
    if (missing > t->obtainable(ks)) return fail(KVS_ERR_NOMEM, "no slot can be freed for demand fetches");
    Claim& c = t->claims[claim];
    c.keys = ks;
    for (uint64_t k : ks) {                    // hold what is in the tier for the retrieval
        auto it = t->objs.find(k);
        if (it == t->objs.end()) continue;
        ++it->second.gpu_refs;
        t->refresh(k, it->second, it->second.lru);
    }
    for (uint64_t k : ks) {                    // fetch the rest on demand, unprotected
        if (t->objs.count(k)) continue;
        Obj o;
        o.slot = t->take_slot();
        o.staging = true;
        o.gpu_refs = 1;
        t->objs[k] = o;
        ++t->staging_count;
        ++t->staged_reads;
        stage_keys[(*n_stage)++] = k;
    }
    c.pending = 0;
    for (uint64_t k : ks) c.pending += t->objs.at(k).staging ? 1 : 0;
    c.committed = false;
    c.state = KVS_CLAIM_ORDINARY;
    return KVS_OK;
}

int kvs_tier_claim_state(const kvs_tier* t, uint64_t claim) {
    if (!t) return KVS_CLAIM_NONE;
    auto ci = t->claims.find(claim);
    return ci == t->claims.end() ? KVS_CLAIM_NONE : ci->second.state;
}

int kvs_tier_object(const kvs_tier* t, uint64_t key, kvs_tier_object_info* out) {
    if (!t || !out) return fail(KVS_ERR_INVALID_ARG, "bad arguments");
    auto it = t->objs.find(key);
    if (it == t->objs.end()) {
        *out = kvs_tier_object_info{-1, 0, 0, 0, 0, 0};
        return KVS_ERR_BOUNDS;
    }
    const Obj& o = it->second;
    *out = kvs_tier_object_info{o.slot, o.pins, o.staging ? 1 : 0, o.resident ? 1 : 0, o.gpu_refs, o.lru};
    return KVS_OK;
}

int kvs_tier_stats_get(kvs_tier* t, double now, kvs_tier_stats* out) {
    if (!t || !out) return fail(KVS_ERR_INVALID_ARG, "bad arguments");
    if (!t->advance(now)) return fail(KVS_ERR_INVALID_ARG, "time went backwards");
    out->resident = t->resident_count;
    out->staging = t->staging_count;
    out->protected_objects = t->protected_count;
    out->free_slots = (int64_t)t->free_slots.size();
    out->evictions = t->evictions;
    out->staged_reads = t->staged_reads;
    out->completed = t->completed;
    out->protected_object_seconds = t->integral;
    return KVS_OK;
}

void* kvs_tier_slot(const kvs_tier* t, int64_t slot) {
    if (!t || !t->arena || slot < 0 || slot >= t->cfg.capacity_objects) return nullptr;
    return t->arena + (size_t)slot * (size_t)t->cfg.object_bytes;
}

}  // extern "C"

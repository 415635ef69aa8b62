/* The C ABI used from plain C99, with no GPU work: include/kvs.h must compile as
 * C, libkvs.so must link, argument errors must come back as status codes with a
 * message, and the fast-tier ledger must run one claim through its states with
 * the protected object-seconds of the cost C (TempoKV Sec. 5, Metrics).
 * Prints "ok" and exits 0 on success; exits with the failing check's number. */
#include <stdio.h>
#include <string.h>

#include "kvs.h"

#define CHECK(n, cond)                                                       \
    do {                                                                     \
        if (!(cond)) {                                                       \
            fprintf(stderr, "check %d failed: %s (%s)\n", n, #cond,          \
                    kvs_last_error());                                       \
            return n;                                                        \
        }                                                                    \
    } while (0)

int main(void) {
    CHECK(1, kvs_version() == KVS_VERSION);

    /* a NULL geometry is rejected before any device work */
    kvs_paged_cache cache;
    memset(&cache, 0, sizeof cache);
    CHECK(2, kvs_retrieve(NULL, &cache, NULL, 0, NULL, 0) == KVS_ERR_INVALID_ARG);
    CHECK(3, strlen(kvs_last_error()) > 0);

    /* an empty call with a valid geometry needs no device; the planes are live host
     * buffers of the declared extent (8 blocks x 16 tokens x 4 heads x 64 dims x 2 B) */
    kvs_geometry g = {2, 4, 64, 2, 16, 256};
    static unsigned char plane_mem[4][8 * 16 * 4 * 64 * 2];
    void* planes[4] = {plane_mem[0], plane_mem[1], plane_mem[2], plane_mem[3]};
    cache.kv_planes = planes;
    cache.num_blocks = 8;
    CHECK(4, kvs_retrieve(&g, &cache, NULL, 0, NULL, 0) == KVS_OK);

    /* conflicting variant flags */
    CHECK(5, kvs_retrieve(&g, &cache, NULL, 0, NULL, KVS_F_FORCE_HOSTLINK | KVS_F_FORCE_HBMCOPY)
                 == KVS_ERR_INVALID_ARG);

    /* the ledger: capacity 4, budget 2; one claim of two objects from t = 1 s to 4 s */
    kvs_tier_config cfg = {4, 2, 1 << 20, 0, 0};
    kvs_tier* tier = NULL;
    CHECK(6, kvs_tier_create(&cfg, &tier) == KVS_OK && tier != NULL);
    uint64_t keys[2] = {11, 12}, stage[2] = {0, 0};
    int32_t n_stage = -1;
    CHECK(7, kvs_tier_commit(tier, 1, keys, 2, 1.0, stage, &n_stage) == KVS_OK && n_stage == 2);
    CHECK(8, kvs_tier_claim_state(tier, 1) == KVS_CLAIM_STAGING);
    CHECK(9, kvs_tier_staged(tier, 11, 2.0) == KVS_OK && kvs_tier_staged(tier, 12, 2.5) == KVS_OK);
    CHECK(10, kvs_tier_claim_state(tier, 1) == KVS_CLAIM_STAGE_READY);
    int64_t slots[2] = {-1, -1};
    CHECK(11, kvs_tier_begin_retrieval(tier, 1, 3.0, slots) == KVS_OK && slots[0] >= 0 && slots[1] >= 0);
    CHECK(12, kvs_tier_end_retrieval(tier, 1, 4.0) == KVS_OK);
    kvs_tier_stats st;
    CHECK(13, kvs_tier_stats_get(tier, 5.0, &st) == KVS_OK);
    CHECK(14, st.completed == 1 && st.protected_objects == 0 && st.resident == 2);
    CHECK(15, st.protected_object_seconds > 5.999 && st.protected_object_seconds < 6.001);
    /* a third protected object would exceed the budget of 2 */
    uint64_t three[3] = {21, 22, 23};
    CHECK(16, kvs_tier_commit(tier, 2, three, 3, 5.0, stage, &n_stage) == KVS_ERR_NOMEM);
    CHECK(17, kvs_tier_destroy(tier) == KVS_OK);

    printf("ok\n");
    return 0;
}

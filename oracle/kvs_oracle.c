/*
 * kvs_oracle.c -- CPU oracle for prefix-KV retrieval (chunk -> paged) and
 * store-back (paged -> chunk).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the library's product path may link,
 * load or call this file; only the tests, the smoke check and the benchmark's
 * CPU-baseline leg do.  It shares no header, helper or table with the CUDA
 * path and computes every index from the definition below, one element at a
 * time, with no blocking or reordering.
 *
 * What it computes (TempoKV, Sec. 2.1: a KV object is read-only during reuse
 * and its access order is known before retrieval; Sec. 4: retrieval reuses
 * the runtime's GPU-transfer path into the paged KV cache; Sec. 5.1 Workload:
 * prefix KV is retained in complete 256-token chunks; Sec. 5 setup: BF16 KV):
 *
 *   geometry   L layers, H kv heads, D head dim, e bytes per element,
 *              B tokens per paged block.
 *   chunk j    of one request covers tokens [s_j, s_j + n_j) of that request,
 *              s_0 = first_token, s_{j+1} = s_j + n_j; its bytes are laid out
 *              [L][2][n_j][H][D] (layer-major, K before V, row-major).
 *   plane p    = 2*l + kv, one per (layer, K/V), laid out [NB*B][H][D]:
 *              NB paged blocks of B token slots each.
 *   slot(t)    = block_table[t / B] * B + (t mod B)   (per-request slot map)
 *
 *   retrieve:  plane[2l+kv][slot(s_j+i)][h][d] := chunk_j[l][kv][i][h][d]
 *   store:     chunk_j[l][kv][i][h][d] := plane[2l+kv][slot(s_j+i)][h][d]
 *
 * for every l < L, kv in {0,1}, i < n_j, h < H, d < D.  Every other element
 * is left untouched.  Elements are opaque e-byte values: nothing is ever
 * interpreted as a number, so the result is exact by construction.
 *
 * Planes [p0, p1) only are touched, so a caller can check a very large cache
 * one plane at a time; p0 = 0, p1 = 2L is the whole definition.  Entries of
 * `planes` outside [p0, p1) are never read and may be NULL.
 *
 * Return value: 0 on success; -2 when a token's block index runs past the
 * block table or names a block outside [0, num_blocks) (nothing is written
 * for that element); -1 on a malformed argument.  Range checks are done per
 * element, before each access.
 */
#include <stddef.h>
#include <stdint.h>
#include <string.h>

/* Offset, in elements, of (plane p, slot s, head h, dim d) in a paged plane. */
static int64_t paged_elem(int64_t slot, int64_t h, int64_t d, int64_t H, int64_t D)
{
    return (slot * H + h) * D + d;
}

/* Offset, in elements, of (layer l, kv, token i, head h, dim d) in a chunk of n tokens. */
static int64_t chunk_elem(int64_t l, int64_t kv, int64_t i, int64_t h, int64_t d,
                          int64_t n, int64_t H, int64_t D)
{
    return ((((l * 2 + kv) * n + i) * H + h) * D) + d;
}

/* Physical slot of request token t; -1 when the block table cannot map it. */
static int64_t slot_of(int64_t t, int64_t B, const int32_t *block_table,
                       int64_t block_table_len, int64_t num_blocks)
{
    int64_t logical = t / B;
    if (t < 0 || logical >= block_table_len) return -1;
    int64_t phys = block_table[logical];
    if (phys < 0 || phys >= num_blocks) return -1;
    return phys * B + (t % B);
}

static int copy_request(int to_cache, int L, int H, int D, int e, int B,
                        uint8_t *const *planes, int64_t num_blocks, int p0, int p1,
                        int64_t first_token, int num_chunks,
                        uint8_t *const *chunks, const int32_t *chunk_tokens,
                        const int32_t *block_table, int64_t block_table_len)
{
    if (L <= 0 || H <= 0 || D <= 0 || e <= 0 || B <= 0 || num_chunks < 0 ||
        p0 < 0 || p1 > 2 * L || p0 > p1 || !block_table)
        return -1;
    int status = 0;
    int64_t s = first_token;                 /* s_j: first request token of chunk j */
    for (int j = 0; j < num_chunks; ++j) {
        int64_t n = chunk_tokens[j];
        if (n < 0 || !chunks[j]) return -1;
        for (int64_t l = 0; l < L; ++l)
            for (int64_t kv = 0; kv < 2; ++kv) {
                int64_t p = 2 * l + kv;
                if (p < p0 || p >= p1) continue;
                uint8_t *plane = planes[p];
                if (!plane) return -1;
                for (int64_t i = 0; i < n; ++i) {
                    int64_t slot = slot_of(s + i, B, block_table, block_table_len, num_blocks);
                    for (int64_t h = 0; h < H; ++h)
                        for (int64_t d = 0; d < D; ++d) {
                            if (slot < 0) { status = -2; continue; }
                            uint8_t *cache_el = plane + paged_elem(slot, h, d, H, D) * e;
                            uint8_t *chunk_el = chunks[j] + chunk_elem(l, kv, i, h, d, n, H, D) * e;
                            for (int b = 0; b < e; ++b) {
                                if (to_cache) cache_el[b] = chunk_el[b];
                                else          chunk_el[b] = cache_el[b];
                            }
                        }
                }
            }
        s += n;
    }
    return status;
}

/* Retrieval of one request: chunk buffers -> paged planes [p0, p1). */
int kvs_oracle_retrieve(int L, int H, int D, int e, int B,
                        uint8_t *const *planes, int64_t num_blocks, int p0, int p1,
                        int64_t first_token, int num_chunks,
                        uint8_t *const *chunks, const int32_t *chunk_tokens,
                        const int32_t *block_table, int64_t block_table_len)
{
    return copy_request(1, L, H, D, e, B, planes, num_blocks, p0, p1, first_token,
                        num_chunks, chunks, chunk_tokens, block_table, block_table_len);
}

/* Store-back of one request: paged planes [p0, p1) -> chunk buffers. */
int kvs_oracle_store(int L, int H, int D, int e, int B,
                     uint8_t *const *planes, int64_t num_blocks, int p0, int p1,
                     int64_t first_token, int num_chunks,
                     uint8_t *const *chunks, const int32_t *chunk_tokens,
                     const int32_t *block_table, int64_t block_table_len)
{
    return copy_request(0, L, H, D, e, B, planes, num_blocks, p0, p1, first_token,
                        num_chunks, chunks, chunk_tokens, block_table, block_table_len);
}

/* Fill n elements of e bytes each with the e-byte pattern `value` (sentinel fill). */
void kvs_oracle_fill(uint8_t *dst, int64_t n, int e, const uint8_t *value)
{
    for (int64_t k = 0; k < n; ++k)
        for (int b = 0; b < e; ++b) dst[k * e + b] = value[b];
}

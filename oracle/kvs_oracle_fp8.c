/*
 * kvs_oracle_fp8.c -- CPU oracle for retrieval from, and store-back into,
 * chunks held in the fast tier as 8-bit floats with per-head scales.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the library's product path may link,
 * load or call this file; only the tests, the smoke check and the benchmark's
 * CPU-baseline leg do.  It shares no header, helper, table or constant with
 * the CUDA path.
 *
 * TempoKV keeps KV in BF16 (Sec. 5 setup) and retains it in 256-token chunks
 * (Sec. 5.1, Workload); it does not compress the fast tier.  This file
 * defines a compressed chunk format that halves the bytes each retrieval
 * moves over the host link, so that the GPU path has one exact definition
 * to be checked against:
 *
 *   element format  E4M3 of the OCP 8-bit Floating Point Specification (OFP8),
 *                   Revision 1.0: 1 sign bit, 4 exponent bits (bias 7), 3
 *                   mantissa bits; no infinities; S.1111.111 is NaN; the
 *                   largest finite magnitude is S.1111.110 = 448; exponent
 *                   field 0 encodes subnormals m/8 * 2^-6.
 *   chunk buffer    [scales][codes]: scales = 2L*H float32 (IEEE binary32,
 *                   little-endian), scale of (layer l, K/V kv, head h) at
 *                   index (2l + kv)*H + h, the block padded with zero bytes to
 *                   a multiple of 256 bytes; codes = [L][2][n][H][D] E4M3
 *                   bytes, laid out like a BF16 chunk's elements.
 *   paged planes    BF16 bit patterns, [NB*B][H][D] per plane p = 2l + kv,
 *                   slot(t) = block_table[t / B] * B + t mod B.
 *
 *   retrieve:  plane[2l+kv][slot(s_j+i)][h][d] :=
 *                  bf16( e4m3(code_j[l][kv][i][h][d]) * scale_j[l][kv][h] )
 *              the product rounded to binary32 (round to nearest even), then
 *              to BF16 (round to nearest even); a NaN product gives 0x7FFF.
 *   store:     for each chunk j, layer l, kv and head h:
 *                  amax  = max |x| over the finite elements x of the chunk's
 *                          n tokens and D dims of head h (0 if none),
 *                  scale = amax / 448 in binary32 (1 when amax is 0), stored,
 *                  inv   = 448 / amax in binary32 (1 when amax is 0),
 *                  code  = e4m3(x * inv) with x * inv a binary32 multiply;
 *                          the conversion rounds to nearest even and
 *                          saturates (OFP8 saturation mode): magnitudes at
 *                          or beyond 448, and infinities, give +-448; NaN
 *                          gives the NaN code 0x7F.
 *              (One division per head and one multiply per element: the
 *              format is this build's, not the paper's, and a reciprocal
 *              multiply keeps quantisation cheap next to the bytes it moves.)
 *
 * Every other element is left untouched.  Return values as in kvs_oracle.c:
 * 0, -2 when a token cannot be mapped through the block table, -1 for a
 * malformed argument.  Floating point is plain C binary32 arithmetic: each
 * multiplication and division is one correctly rounded IEEE operation.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <string.h>

/* ---- E4M3 (OFP8 rev 1.0) -------------------------------------------------- */

/* Value of an E4M3 code, from the field definitions (NaN for S.1111.111). */
float kvs_oracle_e4m3_value(uint8_t code)
{
    int s = code >> 7;
    int e = (code >> 3) & 0xF;
    int m = code & 0x7;
    double v;
    if (e == 0xF && m == 0x7) return NAN;
    if (e == 0) v = ldexp((double)m / 8.0, 1 - 7);          /* subnormal: 0.mmm * 2^(1 - bias) */
    else        v = ldexp(1.0 + (double)m / 8.0, e - 7);    /* normal:    1.mmm * 2^(e - bias) */
    return (float)(s ? -v : v);
}

/* Nearest E4M3 code to v: round to nearest, ties to the code with an even
 * mantissa, saturating at +-448.  Non-negative codes 0x00..0x7E are ordered
 * by value, so the search runs over them and the sign is applied after. */
uint8_t kvs_oracle_e4m3_code(float v)
{
    if (isnan(v)) return 0x7F;
    uint8_t sign = signbit(v) ? 0x80 : 0x00;
    double a = fabs((double)v);
    /* largest non-negative finite code whose value is <= a (binary search) */
    int lo = 0, hi = 0x7E;
    while (lo < hi) {
        int mid = (lo + hi + 1) / 2;
        if ((double)kvs_oracle_e4m3_value((uint8_t)mid) <= a) lo = mid;
        else hi = mid - 1;
    }
    int k = lo;
    if (k == 0x7E) return (uint8_t)(sign | 0x7E);        /* at or beyond the largest finite value */
    double below = kvs_oracle_e4m3_value((uint8_t)k);
    double above = kvs_oracle_e4m3_value((uint8_t)(k + 1));
    double midpoint = (below + above) / 2.0;             /* exact: both have few significant bits */
    int pick;
    if (a < midpoint) pick = k;
    else if (a > midpoint) pick = k + 1;
    else pick = (k % 2 == 0) ? k : k + 1;                /* a tie goes to the even mantissa */
    return (uint8_t)(sign | pick);
}

/* ---- BF16 ------------------------------------------------------------------ */

static uint32_t f32_bits(float f)
{
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    return u;
}

static float f32_from_bits(uint32_t u)
{
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

/* BF16 nearest to v (round to nearest, ties to even); 0x7FFF for NaN.  The BF16
 * values are the binary32 values whose low 16 bits are zero: between the one
 * obtained by dropping those bits and the next one up in magnitude, take the
 * nearer, or on a tie the one whose last kept bit is 0. */
uint16_t kvs_oracle_bf16_bits(float v)
{
    if (isnan(v)) return 0x7FFF;
    uint32_t u = f32_bits(v);
    uint32_t down = u & 0xFFFF0000u;
    uint32_t rest = u & 0x0000FFFFu;
    uint32_t up = down + 0x10000u;                       /* next magnitude (may reach infinity) */
    uint32_t r;
    if (rest < 0x8000u) r = down;
    else if (rest > 0x8000u) r = up;
    else r = ((down >> 16) & 1u) ? up : down;
    return (uint16_t)(r >> 16);
}

float kvs_oracle_bf16_value(uint16_t b)
{
    return f32_from_bits((uint32_t)b << 16);
}

/* ---- chunk layout ------------------------------------------------------------ */

/* Bytes of the scale block at the head of every fp8 chunk buffer. */
int64_t kvs_oracle_fp8_scale_bytes(int L, int H)
{
    int64_t raw = (int64_t)2 * L * H * 4;
    return (raw + 255) / 256 * 256;
}

static int64_t chunk_code(int64_t l, int64_t kv, int64_t i, int64_t h, int64_t d,
                          int64_t n, int64_t H, int64_t D)
{
    return ((((l * 2 + kv) * n + i) * H + h) * D) + d;
}

static int64_t paged_elem(int64_t slot, int64_t h, int64_t d, int64_t H, int64_t D)
{
    return (slot * H + h) * D + d;
}

static int64_t slot_of(int64_t t, int64_t B, const int32_t *block_table,
                       int64_t block_table_len, int64_t num_blocks)
{
    int64_t logical = t / B;
    if (t < 0 || logical >= block_table_len) return -1;
    int64_t phys = block_table[logical];
    if (phys < 0 || phys >= num_blocks) return -1;
    return phys * B + (t % B);
}

static float get_scale(const uint8_t *chunk, int64_t l, int64_t kv, int64_t h, int64_t H)
{
    float s;
    memcpy(&s, chunk + ((l * 2 + kv) * H + h) * 4, sizeof s);
    return s;
}

static void put_scale(uint8_t *chunk, int64_t l, int64_t kv, int64_t h, int64_t H, float s)
{
    memcpy(chunk + ((l * 2 + kv) * H + h) * 4, &s, sizeof s);
}

/* Retrieval of one request from fp8 chunks into BF16 planes [p0, p1). */
int kvs_oracle_retrieve_fp8(int L, int H, int D, int B,
                            uint16_t *const *planes, int64_t num_blocks, int p0, int p1,
                            int64_t first_token, int num_chunks,
                            uint8_t *const *chunks, const int32_t *chunk_tokens,
                            const int32_t *block_table, int64_t block_table_len)
{
    if (L <= 0 || H <= 0 || D <= 0 || B <= 0 || num_chunks < 0 ||
        p0 < 0 || p1 > 2 * L || p0 > p1 || !block_table)
        return -1;
    const int64_t hdr = kvs_oracle_fp8_scale_bytes(L, H);
    int status = 0;
    int64_t s = first_token;
    for (int j = 0; j < num_chunks; ++j) {
        int64_t n = chunk_tokens[j];
        if (n < 0 || !chunks[j]) return -1;
        const uint8_t *codes = chunks[j] + hdr;
        for (int64_t l = 0; l < L; ++l)
            for (int64_t kv = 0; kv < 2; ++kv) {
                int64_t p = 2 * l + kv;
                if (p < p0 || p >= p1) continue;
                uint16_t *plane = planes[p];
                if (!plane) return -1;
                for (int64_t i = 0; i < n; ++i) {
                    int64_t slot = slot_of(s + i, B, block_table, block_table_len, num_blocks);
                    for (int64_t h = 0; h < H; ++h) {
                        float scale = get_scale(chunks[j], l, kv, h, H);
                        for (int64_t d = 0; d < D; ++d) {
                            if (slot < 0) { status = -2; continue; }
                            float x = kvs_oracle_e4m3_value(codes[chunk_code(l, kv, i, h, d, n, H, D)]);
                            float y = x * scale;                 /* one binary32 multiply */
                            plane[paged_elem(slot, h, d, H, D)] = kvs_oracle_bf16_bits(y);
                        }
                    }
                }
            }
        s += n;
    }
    return status;
}

/* Store-back of one request from BF16 planes [p0, p1) into fp8 chunks: the
 * scales of the planes in range and their codes are written. */
int kvs_oracle_store_fp8(int L, int H, int D, int B,
                         uint16_t *const *planes, int64_t num_blocks, int p0, int p1,
                         int64_t first_token, int num_chunks,
                         uint8_t *const *chunks, const int32_t *chunk_tokens,
                         const int32_t *block_table, int64_t block_table_len)
{
    if (L <= 0 || H <= 0 || D <= 0 || B <= 0 || num_chunks < 0 ||
        p0 < 0 || p1 > 2 * L || p0 > p1 || !block_table)
        return -1;
    const int64_t hdr = kvs_oracle_fp8_scale_bytes(L, H);
    int status = 0;
    int64_t s = first_token;
    for (int j = 0; j < num_chunks; ++j) {
        int64_t n = chunk_tokens[j];
        if (n < 0 || !chunks[j]) return -1;
        uint8_t *codes = chunks[j] + hdr;
        for (int64_t l = 0; l < L; ++l)
            for (int64_t kv = 0; kv < 2; ++kv) {
                int64_t p = 2 * l + kv;
                if (p < p0 || p >= p1) continue;
                const uint16_t *plane = planes[p];
                if (!plane) return -1;
                for (int64_t h = 0; h < H; ++h) {
                    /* amax over the finite elements of head h in this chunk */
                    float amax = 0.0f;
                    for (int64_t i = 0; i < n; ++i) {
                        int64_t slot = slot_of(s + i, B, block_table, block_table_len, num_blocks);
                        if (slot < 0) { status = -2; continue; }
                        for (int64_t d = 0; d < D; ++d) {
                            float x = kvs_oracle_bf16_value(plane[paged_elem(slot, h, d, H, D)]);
                            if (isfinite(x) && fabsf(x) > amax) amax = fabsf(x);
                        }
                    }
                    float scale = amax > 0.0f ? amax / 448.0f : 1.0f;
                    float inv = amax > 0.0f ? 448.0f / amax : 1.0f;
                    put_scale(chunks[j], l, kv, h, H, scale);
                    for (int64_t i = 0; i < n; ++i) {
                        int64_t slot = slot_of(s + i, B, block_table, block_table_len, num_blocks);
                        if (slot < 0) continue;
                        for (int64_t d = 0; d < D; ++d) {
                            float x = kvs_oracle_bf16_value(plane[paged_elem(slot, h, d, H, D)]);
                            float q = x * inv;                   /* one binary32 multiply */
                            codes[chunk_code(l, kv, i, h, d, n, H, D)] = kvs_oracle_e4m3_code(q);
                        }
                    }
                }
            }
        s += n;
    }
    return status;
}

/* ---- element-wise loops over arrays (for the Python wrapper) --------------- */

void kvs_oracle_e4m3_encode_array(const float *in, uint8_t *out, int64_t n)
{
    for (int64_t k = 0; k < n; ++k) out[k] = kvs_oracle_e4m3_code(in[k]);
}

void kvs_oracle_e4m3_decode_array(const uint8_t *in, float *out, int64_t n)
{
    for (int64_t k = 0; k < n; ++k) out[k] = kvs_oracle_e4m3_value(in[k]);
}

void kvs_oracle_bf16_encode_array(const float *in, uint16_t *out, int64_t n)
{
    for (int64_t k = 0; k < n; ++k) out[k] = kvs_oracle_bf16_bits(in[k]);
}

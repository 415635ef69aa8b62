// kvs_fp8.cu -- retrieval from, and store-back into, fp8 chunks on sm_103a.
//
// A compressed fast-tier format (the paper keeps BF16 KV, Sec. 5 setup): a
// chunk holds E4M3 codes of the OCP 8-bit floating point specification
// (revision 1.0) and one binary32 scale per (layer, K/V, head), so a
// retrieval moves half the bytes of a BF16 chunk over the host link:
//
//   chunk  [scales: 2L*H binary32 at (2l+kv)*H + h, padded to scale_bytes]
//          [codes:  [L][2][n][H][D] E4M3 bytes]
//   plane  BF16 [NB][B][H][D] per (layer, K/V)
//
//   retrieve  plane = bf16_rn(fp32(code) *rn scale); a NaN product gives 0x7FFF
//   store     per (chunk, layer, K/V, head): amax over the finite elements,
//             scale = amax /rn 448 (stored), inv = 448 /rn amax (both 1 when
//             amax is 0), code = e4m3 of x *rn inv, rounded to nearest even
//             and saturated at +-448; NaN gives the code 0x7F
//
// Every element conversion uses the hardware conversions of sm_89+ (E4M3 <->
// f16 pairs, f32 -> bf16 / E4M3 pairs, round to nearest even, the E4M3 one
// saturating) and IEEE round-to-nearest multiplies.  The conversions
// themselves give the canonical NaN patterns the format defines: 0x7FFF for a
// NaN product on retrieval, 0x7F for a NaN input of either sign on store (the
// special-values parity test plants NaN codes, NaN scales and NaN inputs of
// both signs and compares with the oracle).
//
// Retrieval is bound by the host link (or HBM for device chunks): a persistent
// grid of 128-thread CTAs walks 16 KiB pieces of codes; each thread keeps two
// pieces' worth of 16-byte code vectors in registers, so the next piece's
// loads are in flight while the current one is converted and stored.  The H
// scales of a piece's plane are loaded once per piece by H threads (one 4-byte
// load each, beside the codes) and shared through shared memory, instead of
// one scale load per vector; HBM chunks run one CTA per piece instead, and
// KVS_F_FEW_SMS runs a kernel that also stages pieces in shared memory so
// that fewer SMs hold the link beside other kernels.
// Store-back to pinned host runs one 256-thread CTA per (chunk, plane, head):
// the head's BF16 elements are loaded into registers at once, reduced to the
// amax and quantised from registers (heads too large for that take a two-pass
// kernel, one CTA per (chunk, plane)).  Into HBM chunks a persistent CTA per SM
// stages heads in shared memory with per-thread async copies, two heads ahead
// of the one it quantises.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_fp8.h>

#include <algorithm>
#include <cstdint>

#include "kvs.h"
#include "kvs_async.cuh"
#include "kvs_internal.h"

namespace kvs {
namespace {

constexpr int kRtThreads = 128;
constexpr int kRtVec = 8;                            // 16-code vectors per thread per piece
static_assert(kRtThreads * kRtVec * 16 == kFp8PieceCodes, "a piece is one vector set per CTA");
constexpr int kStThreads = 256;

struct Fp8Piece {
    uint64_t codes;      // first code of the piece
    uint64_t out;        // first BF16 element of the piece in the plane
    uint64_t scales;     // scale block row of the piece's plane: H binary32
    uint32_t len;        // codes in the piece (a multiple of 16)
    uint32_t vec0;       // index of the piece's first vector within its run
};

// Piece q -> addresses; false for pieces with nothing to move.  Runs are
// (entry, plane, block) as for BF16 copies; a run holds ntok rows of H*D codes.
__device__ __forceinline__ uint32_t fp8_div(uint32_t n, uint32_t m, uint32_t p) {
    return (uint32_t)(((uint64_t)n * m) >> p);
}

// FAST: the reciprocal divisions (persistent kernels decode a piece per loop
// trip); the one-piece-per-CTA kernel keeps plain divisions and per-vector head indices,
// which holds it at fewer registers.
template <bool FAST = true>
__device__ __forceinline__ bool fp8_piece(const Fp8Job& f, uint32_t q, Fp8Piece& pc) {
    const Job& j = f.job;
    const uint32_t hd = f.heads * f.head_dim;
    const uint32_t per_entry = j.num_planes * j.blocks_per_chunk;
    const uint32_t run = FAST ? fp8_div(q, f.ppr_m, f.ppr_p) : q / j.pieces_per_run;
    const uint32_t k = q - run * j.pieces_per_run;
    const uint32_t e = FAST ? fp8_div(run, f.pe_m, f.pe_p) : run / per_entry;
    const uint32_t rem = run - e * per_entry;
    const uint32_t pr = FAST ? fp8_div(rem, f.bpc_m, f.bpc_p) : rem / j.blocks_per_chunk;
    const uint32_t i = rem - pr * j.blocks_per_chunk;
    const uint32_t p = j.plane_begin + pr;
    const int32_t blk = __ldg(j.blocks + (size_t)(j.entry_base + e) * j.blocks_per_chunk + i);
    const Entry en = j.entries[e];
    const int64_t first = (int64_t)i * j.block_size;
    const int64_t ntok = min((int64_t)j.block_size, (int64_t)en.n_tok - first);
    if (ntok <= 0 || blk < 0) return false;
    if (blk >= j.num_blocks) {
        atomicCAS(j.err, 0, KVS_ERR_BOUNDS);
        return false;
    }
    const uint64_t run_codes = (uint64_t)ntok * hd;
    const uint64_t off = (uint64_t)k * kFp8PieceCodes;
    if (off >= run_codes) return false;
    pc.len = (uint32_t)min((uint64_t)kFp8PieceCodes, run_codes - off);
    pc.vec0 = (uint32_t)(off / 16);
    pc.codes = en.chunk + f.scale_bytes + ((uint64_t)p * (uint64_t)en.n_tok + (uint64_t)first) * hd + off;
    pc.out = j.planes[p] + ((uint64_t)blk * j.block_size) * hd * 2 + off * 2;
    pc.scales = en.chunk + (uint64_t)p * f.heads * 4;
    return true;
}

__device__ __forceinline__ uint4 ld_nc16(uint64_t a) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "l"(a));
    return r;
}

__device__ __forceinline__ void st_cs16(uint64_t a, const uint4& v) {
    asm volatile("st.global.cs.v4.u32 [%0], {%1,%2,%3,%4};"
                 :: "l"(a), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w) : "memory");
}

// Two E4M3 codes (low byte first) times `s` -> two BF16 (low half first).
__device__ __forceinline__ uint32_t e4m3x2_to_bf16x2(uint32_t two, float s) {
    const __half2_raw hr = __nv_cvt_fp8x2_to_halfraw2((__nv_fp8x2_storage_t)(two & 0xFFFFu), __NV_E4M3);
    __half2 h;
    *reinterpret_cast<__half2_raw*>(&h) = hr;
    const float2 v = __half22float2(h);                          // exact
    const float a = __fmul_rn(v.x, s), b = __fmul_rn(v.y, s);
    const __nv_bfloat162 r = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&r);
}

// 16 codes -> 32 bytes of BF16.
__device__ __forceinline__ void dequant16(const uint4& c, float s, uint4& lo, uint4& hi) {
    lo.x = e4m3x2_to_bf16x2(c.x, s);
    lo.y = e4m3x2_to_bf16x2(c.x >> 16, s);
    lo.z = e4m3x2_to_bf16x2(c.y, s);
    lo.w = e4m3x2_to_bf16x2(c.y >> 16, s);
    hi.x = e4m3x2_to_bf16x2(c.z, s);
    hi.y = e4m3x2_to_bf16x2(c.z >> 16, s);
    hi.z = e4m3x2_to_bf16x2(c.w, s);
    hi.w = e4m3x2_to_bf16x2(c.w >> 16, s);
}

// A piece's codes in registers; thread t < H also holds the scale of head t,
// loaded once per piece (not once per vector) beside the codes.
struct RtRegs {
    uint4 c[kRtVec];
    float s;
};

__device__ __forceinline__ void rt_load(const Fp8Job& f, const Fp8Piece& pc, RtRegs& r) {
    const uint32_t nv = pc.len / 16;
#pragma unroll
    for (int u = 0; u < kRtVec; ++u) {
        const uint32_t v = threadIdx.x + u * kRtThreads;
        if (v < nv) r.c[u] = ld_nc16(pc.codes + (uint64_t)v * 16);
    }
    if (threadIdx.x < f.heads) r.s = __ldg(reinterpret_cast<const float*>(pc.scales) + threadIdx.x);
}

// Publishes the piece's scales in shared memory (after every thread has finished
// with the previous piece's), then converts and stores this thread's vectors.
// Head of this thread's vector v of a piece: when pieces start at token rows
// and a row's vpr vectors divide the CTA's thread count T, vector tid + u*T
// is always in head (tid % vpr) / vph, computed once per thread (`h_fixed`).
__device__ __forceinline__ uint32_t fp8_fixed_head(const Fp8Job& f, uint32_t T) {
    const uint32_t vph = f.head_dim / 16, vpr = f.heads * vph;
    return (f.rows_whole && T % vpr == 0) ? (threadIdx.x % vpr) / vph : 0xFFFFFFFFu;
}

__device__ __forceinline__ uint32_t fp8_head(const Fp8Job& f, const Fp8Piece& pc, uint32_t v, uint32_t h_fixed) {
    if (h_fixed != 0xFFFFFFFFu) return h_fixed;
    const uint32_t vph = f.head_dim / 16, vpr = f.heads * vph;
    return ((pc.vec0 + v) % vpr) / vph;
}

__device__ __forceinline__ void rt_store(const Fp8Job& f, const Fp8Piece& pc, const RtRegs& r, float* sm_scale,
                                         uint32_t h_fixed) {
    const uint32_t nv = pc.len / 16;
    __syncthreads();
    if (threadIdx.x < f.heads) sm_scale[threadIdx.x] = r.s;
    __syncthreads();
#pragma unroll
    for (int u = 0; u < kRtVec; ++u) {
        const uint32_t v = threadIdx.x + u * kRtThreads;
        if (v < nv) {
            uint4 lo, hi;
            dequant16(r.c[u], sm_scale[fp8_head(f, pc, v, h_fixed)], lo, hi);
            st_cs16(pc.out + (uint64_t)v * 32, lo);
            st_cs16(pc.out + (uint64_t)v * 32 + 16, hi);
        }
    }
}

__device__ __forceinline__ bool rt_next(const Fp8Job& f, uint32_t n, uint32_t& q, Fp8Piece& pc) {
    while (q < n) {
        const uint32_t cur = q;
        q += gridDim.x;
        if (fp8_piece(f, cur, pc)) return true;
    }
    return false;
}

// Every thread of a CTA walks the same sequence of pieces (the piece index
// depends only on blockIdx), so the barriers in rt_store are reached by all.
__global__ void __launch_bounds__(kRtThreads) kvs_fp8_retrieve_kernel(const Fp8Job f, uint32_t num_pieces) {
    __shared__ float sm_scale[kFp8MaxHeads];
    const uint32_t h_fixed = fp8_fixed_head(f, kRtThreads);
    RtRegs ra, rb;
    Fp8Piece pa, pb;
    uint32_t q = blockIdx.x;
    bool ha = rt_next(f, num_pieces, q, pa);
    if (ha) rt_load(f, pa, ra);
    while (ha) {
        const bool hb = rt_next(f, num_pieces, q, pb);
        if (hb) rt_load(f, pb, rb);
        rt_store(f, pa, ra, sm_scale, h_fixed);
        if (!hb) break;
        ha = rt_next(f, num_pieces, q, pa);
        if (ha) rt_load(f, pa, ra);
        rt_store(f, pb, rb, sm_scale, h_fixed);
    }
}

// Device chunks (HBM source): one CTA per piece, no persistence; the launch
// bound keeps the kernel at 64 registers so eight CTAs -- 128 KiB of code
// loads -- are in flight per SM, and the hardware block scheduler overlaps one
// CTA's stores with the next CTA's loads.
__global__ void __launch_bounds__(kRtThreads, 8) kvs_fp8_retrieve_piece_kernel(const Fp8Job f) {
    __shared__ float sm_scale[kFp8MaxHeads];
    Fp8Piece pc;
    if (!fp8_piece<false>(f, blockIdx.x, pc)) return;  // uniform across the CTA
    RtRegs r;
    rt_load(f, pc, r);
    rt_store(f, pc, r, sm_scale, 0xFFFFFFFFu);
}

// Few-SM flavour of the host-chunk retrieval (KVS_F_FEW_SMS): the scheme of
// the host-link BF16 staged kernel.  A 256-thread CTA keeps seven 16 KiB pieces
// of codes in flight: two in registers and five in shared memory, where each
// thread copies, with cp.async, its own 16-code vectors and the binary32 scale
// of each vector's head into slots that only it reads back (no CTA barrier).
// 100 KiB of shared memory per CTA, two CTAs per SM: 224 KiB of codes in flight
// per SM, where kvs_fp8_retrieve_kernel holds 128 KiB.  Piece i of a CTA lives
// in slot i % 7; pieces come in grid-stride order, so once a slot finds none
// left, neither does any slot after it.
constexpr int kFsThreads = 256;
constexpr int kFsVec = kFp8PieceCodes / 16 / kFsThreads;             // vectors per thread per piece
constexpr int kFsRegPieces = 2;
constexpr int kFsSmemPieces = 5;
constexpr int kFsSlots = kFsRegPieces + kFsSmemPieces;
constexpr uint32_t kFsSlotBytes = kFp8PieceCodes + kFp8PieceCodes / 16 * 4;   // codes + a scale per vector
constexpr uint32_t kFsSmemBytes = kFsSmemPieces * kFsSlotBytes;
static_assert(kFsVec * kFsThreads * 16 == kFp8PieceCodes, "a piece is one vector set per CTA");

__device__ __forceinline__ void fs_cp16(uint32_t dst, uint64_t src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" :: "r"(dst), "l"(src) : "memory");
}

__device__ __forceinline__ void fs_cp4(uint32_t dst, uint64_t src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" :: "r"(dst), "l"(src) : "memory");
}

__device__ __forceinline__ void fs_commit() {
    asm volatile("cp.async.commit_group;" ::: "memory");
}

template <int N>
__device__ __forceinline__ void fs_wait() {
    asm volatile("cp.async.wait_group %0;" :: "n"(N) : "memory");
}

// Scale address of vector v of piece pc (its head's binary32 scale).
__device__ __forceinline__ uint64_t fs_scale_addr(const Fp8Job& f, const Fp8Piece& pc, uint32_t v, uint32_t h_fixed) {
    return pc.scales + (uint64_t)fp8_head(f, pc, v, h_fixed) * 4;
}

struct FsRegs {
    uint4 c[kFsVec];
    float s[kFsVec];
};

__device__ __forceinline__ void fs_load_regs(const Fp8Job& f, const Fp8Piece& pc, FsRegs& r, uint32_t h_fixed) {
    const uint32_t nv = pc.len / 16;
#pragma unroll
    for (int u = 0; u < kFsVec; ++u) {
        const uint32_t v = threadIdx.x + u * kFsThreads;
        if (v < nv) {
            r.c[u] = ld_nc16(pc.codes + (uint64_t)v * 16);
            r.s[u] = __ldg(reinterpret_cast<const float*>(fs_scale_addr(f, pc, v, h_fixed)));
        }
    }
}

__device__ __forceinline__ void fs_store_regs(const Fp8Piece& pc, const FsRegs& r) {
    const uint32_t nv = pc.len / 16;
#pragma unroll
    for (int u = 0; u < kFsVec; ++u) {
        const uint32_t v = threadIdx.x + u * kFsThreads;
        if (v < nv) {
            uint4 lo, hi;
            dequant16(r.c[u], r.s[u], lo, hi);
            st_cs16(pc.out + (uint64_t)v * 32, lo);
            st_cs16(pc.out + (uint64_t)v * 32 + 16, hi);
        }
    }
}

// Slot layout: codes of vector v at v * 16, its scale at kFp8PieceCodes + v * 4.
__device__ __forceinline__ void fs_stage(const Fp8Job& f, const Fp8Piece& pc, uint32_t slot, uint32_t h_fixed) {
    const uint32_t nv = pc.len / 16;
#pragma unroll
    for (int u = 0; u < kFsVec; ++u) {
        const uint32_t v = threadIdx.x + u * kFsThreads;
        if (v < nv) {
            fs_cp16(slot + v * 16, pc.codes + (uint64_t)v * 16);
            fs_cp4(slot + kFp8PieceCodes + v * 4, fs_scale_addr(f, pc, v, h_fixed));
        }
    }
}

__device__ __forceinline__ void fs_unstage(const Fp8Piece& pc, uint32_t slot) {
    const uint32_t nv = pc.len / 16;
#pragma unroll
    for (int u = 0; u < kFsVec; ++u) {
        const uint32_t v = threadIdx.x + u * kFsThreads;
        if (v < nv) {
            uint4 c;
            float sc;
            asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                         : "=r"(c.x), "=r"(c.y), "=r"(c.z), "=r"(c.w) : "r"(slot + v * 16));
            asm volatile("ld.shared.f32 %0, [%1];" : "=f"(sc) : "r"(slot + kFp8PieceCodes + v * 4));
            uint4 lo, hi;
            dequant16(c, sc, lo, hi);
            st_cs16(pc.out + (uint64_t)v * 32, lo);
            st_cs16(pc.out + (uint64_t)v * 32 + 16, hi);
        }
    }
}

__global__ void __launch_bounds__(kFsThreads, 2) kvs_fp8_retrieve_staged_kernel(const Fp8Job f, uint32_t num_pieces) {
    extern __shared__ __align__(128) uint8_t fs_smem[];
    const uint32_t base = smem_u32(fs_smem);
    const uint32_t h_fixed = fp8_fixed_head(f, kFsThreads);
    FsRegs r[kFsRegPieces];
    Fp8Piece pc[kFsSlots];
    bool has[kFsSlots];
    uint32_t q = blockIdx.x;
    // fill slot s with the CTA's next piece; a shared-memory slot always commits
    // one group (empty past the end), so wait_group counts pieces
    auto fill = [&](int s) {
        has[s] = rt_next(f, num_pieces, q, pc[s]);
        if (s < kFsRegPieces) {
            if (has[s]) fs_load_regs(f, pc[s], r[s < kFsRegPieces ? s : 0], h_fixed);
        } else {
            if (has[s]) fs_stage(f, pc[s], base + (s - kFsRegPieces) * kFsSlotBytes, h_fixed);
            fs_commit();
        }
    };
#pragma unroll
    for (int s = 0; s < kFsSlots; ++s) fill(s);
    bool more = true;
    while (more) {
#pragma unroll
        for (int s = 0; s < kFsSlots; ++s) {
            if (more && !has[s]) more = false;
            if (more) {
                if (s < kFsRegPieces) {
                    fs_store_regs(pc[s], r[s < kFsRegPieces ? s : 0]);
                } else {
                    fs_wait<kFsSmemPieces - 1>();    // the younger shared-memory pieces may be in flight
                    fs_unstage(pc[s], base + (s - kFsRegPieces) * kFsSlotBytes);
                }
                fill(s);
            }
        }
    }
    fs_wait<0>();
}

// ---------------------------------------------------------------------------
// Store-back (quantise)
// ---------------------------------------------------------------------------

// Per-halfword running maximum of |x| over the finite BF16 values of a word
// pair.  |x| of a finite BF16 orders like its bits with the sign cleared
// (0x0000..0x7F7F); adding 0x80 to each half moves the finite ones to
// 0x0080..0x7FFF and infinities / NaN (0x7F80..0x7FFF) to 0x8000..0x807F,
// negative as signed 16-bit lanes, so a signed lane maximum that starts from 0
// never takes them (no carry crosses halves: each half stays below 0x10000).
// The running value is offset by 0x80; amax_bits removes the offset.
__device__ __forceinline__ uint32_t amax2(uint32_t m2, uint32_t w) {
    uint32_t r;
    asm("max.s16x2 %0, %1, %2;" : "=r"(r) : "r"(m2), "r"((w & 0x7FFF7FFFu) + 0x00800080u));   // sm_90+
    return r;
}

// Bits of the largest finite |x| (0 when there is none) from a running amax2 value.
__device__ __forceinline__ uint32_t amax_bits(uint32_t m2) {
    return max(max(m2 & 0xFFFFu, m2 >> 16), 0x80u) - 0x80u;
}

__device__ __forceinline__ uint32_t amax_bits8(const uint4& v) {
    return amax_bits(amax2(amax2(amax2(amax2(0u, v.x), v.y), v.z), v.w));
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// Two BF16 (one word) times `inv` -> two E4M3 codes (saturating, nearest even).
__device__ __forceinline__ uint32_t e4m3x2_of(uint32_t w, float inv) {
    return (uint32_t)__nv_cvt_float2_to_fp8x2(make_float2(__fmul_rn(bf16_lo(w), inv), __fmul_rn(bf16_hi(w), inv)),
                                              __NV_SATFINITE, __NV_E4M3);
}

// 8 BF16 (one 16-byte vector) -> 8 codes.
__device__ __forceinline__ uint2 quant8(const uint4& a, float inv) {
    return make_uint2(e4m3x2_of(a.x, inv) | (e4m3x2_of(a.y, inv) << 16),
                      e4m3x2_of(a.z, inv) | (e4m3x2_of(a.w, inv) << 16));
}

// 16 BF16 (two vectors) -> 16 codes.
__device__ __forceinline__ uint4 quant16(const uint4& a, const uint4& b, float inv) {
    const uint2 x = quant8(a, inv), y = quant8(b, inv);
    return make_uint4(x.x, x.y, y.x, y.y);
}

__device__ __forceinline__ void st_cs8(uint64_t a, const uint2& v) {
    asm volatile("st.global.cs.v2.u32 [%0], {%1,%2};" :: "l"(a), "r"(v.x), "r"(v.y) : "memory");
}

// Single pass, one CTA per (entry, plane, head): the head's n x D BF16 elements
// of the chunk (at most kHeadVec * kStThreads * 8, i.e. 64 KiB) are loaded
// into registers at once (kHeadVec 16-byte vectors per thread, all in flight),
// reduced to the head's amax across the CTA, and quantised from registers:
// the planes are read once and the loads of a whole head are in flight together.
// Thread t handles the 16-byte column w = t % (D/8) of tokens t / (D/8) + u *
// step (step = kStThreads / (D/8) tokens), so the column, and with it the
// address arithmetic inside a token row, is fixed per thread.  Needs D/8 to
// divide kStThreads and n, B below 2^16 (checked by the launcher).
constexpr int kHeadVec = 16;
constexpr uint32_t kHeadMaxElems = kHeadVec * kStThreads * 8;

// One segment of the store: FULL when every thread's kHeadVec vectors all lie in
// the chunk (n * D/8 == kHeadVec * kStThreads, e.g. a 256-token chunk of head_dim
// 128), so the loads and stores need no per-vector bounds test.
template <bool FULL>
__device__ __forceinline__ void store_head_segment(const Fp8Job& f, uint32_t e, uint32_t p, uint32_t h,
                                                   uint32_t* warp_max, float* sm_inv) {
    const Job& j = f.job;
    const uint32_t H = f.heads, D = f.head_dim, vpt = D / 8;
    const uint32_t B = j.block_size, step = kStThreads / vpt;
    const uint32_t w = threadIdx.x % vpt, i0 = threadIdx.x / vpt;
    const uint64_t row2 = (uint64_t)H * D * 2;
    const Entry en = j.entries[e];
    const uint32_t n = (uint32_t)en.n_tok;
    const int32_t* blocks = j.blocks + (size_t)(j.entry_base + e) * j.blocks_per_chunk;
    const uint64_t src0 = j.planes[p] + (uint64_t)h * D * 2 + (uint64_t)w * 16;
    uint4 v[kHeadVec];
    uint32_t m2 = 0;
    bool bad = false;
#pragma unroll
    for (int u = 0; u < kHeadVec; ++u) {
        const uint32_t i = i0 + u * step;
        v[u] = make_uint4(0, 0, 0, 0);
        if (FULL || i < n) {
            const uint32_t bi = B == 1 ? i : __umulhi(i, f.block_magic), r = i - bi * B;
            const int32_t blk = __ldg(blocks + bi);
            if (blk < 0 || blk >= j.num_blocks) bad = true;
            else v[u] = ld_nc16(src0 + ((uint64_t)blk * B + r) * row2);
        }
    }
#pragma unroll
    for (int u = 0; u < kHeadVec; ++u)
        m2 = amax2(amax2(amax2(amax2(m2, v[u].x), v[u].y), v[u].z), v[u].w);
    if (bad) atomicCAS(j.err, 0, KVS_ERR_BOUNDS);
    const uint32_t m = __reduce_max_sync(0xFFFFFFFFu, amax_bits(m2));
    if ((threadIdx.x & 31) == 0) warp_max[threadIdx.x >> 5] = m;
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t a = 0;
        for (int k = 0; k < kStThreads / 32; ++k) a = max(a, warp_max[k]);
        const float af = __uint_as_float(a << 16);
        const float sc = af > 0.0f ? __fdiv_rn(af, 448.0f) : 1.0f;
        *sm_inv = af > 0.0f ? __fdiv_rn(448.0f, af) : 1.0f;
        *reinterpret_cast<float*>(en.chunk + ((uint64_t)p * H + h) * 4) = sc;
    }
    __syncthreads();
    const float inv = *sm_inv;
    const uint64_t hd = (uint64_t)H * D;
    const uint64_t codes = en.chunk + f.scale_bytes + (uint64_t)p * n * hd + (uint64_t)h * D + (uint64_t)w * 8 +
                           (uint64_t)i0 * hd;
#pragma unroll
    for (int u = 0; u < kHeadVec; ++u) {
        const uint32_t i = i0 + u * step;
        if (FULL || i < n) st_cs8(codes + (uint64_t)(u * step) * hd, quant8(v[u], inv));
    }
    __syncthreads();                                       // warp_max / sm_inv are reused
}

__global__ void __launch_bounds__(kStThreads) kvs_fp8_store_head_kernel(const Fp8Job f, uint32_t num_segments) {
    __shared__ uint32_t warp_max[kStThreads / 32];
    __shared__ float sm_inv;
    const Job& j = f.job;
    const uint32_t H = f.heads, full_n = kHeadVec * kStThreads / (f.head_dim / 8);
    for (uint32_t seg = blockIdx.x; seg < num_segments; seg += gridDim.x) {
        const uint32_t eh = seg / H, h = seg - eh * H;
        const uint32_t e = eh / j.num_planes;
        const uint32_t p = j.plane_begin + (eh - e * j.num_planes);
        if ((uint32_t)j.entries[e].n_tok == full_n)          // uniform across the CTA
            store_head_segment<true>(f, e, p, h, warp_max, &sm_inv);
        else
            store_head_segment<false>(f, e, p, h, warp_max, &sm_inv);
    }
}

// ---------------------------------------------------------------------------
// Staged store-back for HBM destinations: per-thread async copies
// ---------------------------------------------------------------------------
// A persistent 512-thread CTA per SM walks segments (as above, one (chunk,
// plane, head) each).  Thread t owns the 16-byte column w = t % (D/8) of
// tokens t / (D/8) + u * step, u < kSgVec (step = kSgThreads / (D/8)); its
// loads go through shared memory: it copies its vectors of segment k with
// cp.async into its own slots of stage k % kSgStages, kSgStages - 1 segments
// ahead of the one it quantises, so two heads' loads (128 KiB) are in flight
// per SM while its registers hold only the current head's 8 vectors.  A thread
// reads back only the slots it filled itself, so the stages need no CTA
// barrier (cp.async.wait_group orders them); the amax reduction takes two.
// Slot u of thread t in a stage is at (u * kSgThreads + t) * 16.  The plane
// rows of a full segment depend only on its chunk, so a thread keeps them in
// registers while consecutive segments share the chunk.
constexpr int kSgThreads = 512;
constexpr int kSgVec = 8;
constexpr int kSgStages = 3;
constexpr uint32_t kSgStageBytes = kSgVec * kSgThreads * 16;        // 64 KiB
constexpr uint32_t kSgSmemBytes = kSgStages * kSgStageBytes;
static_assert(kSgStageBytes == kHeadMaxElems * 2, "a stage holds the largest single-pass head");

// A CTA's segments are one contiguous range, walked with a cursor over
// (entry, plane, head): consecutive segments share the chunk (and its plane
// rows) and mostly the plane, and need no division to decode.
struct SgCur {
    uint32_t e, p, h;
};

__device__ __forceinline__ SgCur sg_at(const Fp8Job& f, uint32_t seg) {
    const Job& j = f.job;
    const uint32_t eh = seg / f.heads, h = seg - eh * f.heads;
    const uint32_t e = eh / j.num_planes;
    return {e, j.plane_begin + (eh - e * j.num_planes), h};
}

__device__ __forceinline__ void sg_step(const Fp8Job& f, SgCur& c) {
    if (++c.h == f.heads) {
        c.h = 0;
        if (++c.p == f.job.plane_begin + f.job.num_planes) {
            c.p = f.job.plane_begin;
            ++c.e;
        }
    }
}

__device__ __forceinline__ void cp_async16(uint32_t dst_smem, uint64_t src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" :: "r"(dst_smem), "l"(src) : "memory");
}

__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;" ::: "memory");
}

template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" :: "n"(N) : "memory");
}

__device__ __forceinline__ uint4 lds16(uint32_t a) {
    uint4 r;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "r"(a));
    return r;
}

__device__ __forceinline__ void sts16_zero(uint32_t a) {
    asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};" :: "r"(a), "r"(0u) : "memory");
}

// Two BF16 (one word) times `inv` -> two E4M3 codes: two binary32 multiplies
// rounded to nearest, then one saturating nearest-even pair conversion (the
// high element goes to the high byte).  (A packed f32x2 multiply measured 0.5%
// slower here.)
__device__ __forceinline__ uint32_t e4m3x2_of_pk(uint32_t w, uint64_t inv2) {
    const float inv = __uint_as_float((uint32_t)inv2);
    const float lo = __fmul_rn(__uint_as_float(w << 16), inv), hi = __fmul_rn(__uint_as_float(w & 0xFFFF0000u), inv);
    uint32_t r;
    asm("{\n\t.reg .b16 t;\n\tcvt.rn.satfinite.e4m3x2.f32 t, %1, %2;\n\tcvt.u32.u16 %0, t;\n\t}"
        : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

__device__ __forceinline__ uint2 quant8_pk(const uint4& a, uint64_t inv2) {
    return make_uint2(e4m3x2_of_pk(a.x, inv2) | (e4m3x2_of_pk(a.y, inv2) << 16),
                      e4m3x2_of_pk(a.z, inv2) | (e4m3x2_of_pk(a.w, inv2) << 16));
}

// Plane row (blk * B + token % B) of token i of a chunk, or kNoRow for a bad block.
constexpr uint32_t kNoRow = 0xFFFFFFFFu;

__device__ __forceinline__ uint32_t sg_row(const Fp8Job& f, const int32_t* blocks, uint32_t i) {
    const Job& j = f.job;
    const uint32_t B = j.block_size;
    const uint32_t bi = B == 1 ? i : __umulhi(i, f.block_magic);
    const int32_t blk = __ldg(blocks + bi);
    return (blk < 0 || blk >= j.num_blocks) ? kNoRow : (uint32_t)blk * B + (i - bi * B);
}

// This thread's loads of segment c (n tokens) into its slots of the stage at
// `stage`; a bad block's vectors are zeros (and the call reports the error).
// `rows` / `rows_e`: the cached rows of full segments and the chunk they belong to.
template <bool FULL>
__device__ __forceinline__ void sg_issue(const Fp8Job& f, const SgCur& c, uint32_t n, uint32_t stage,
                                         uint32_t (&rows)[kSgVec], uint32_t& rows_e) {
    const Job& j = f.job;
    const uint32_t D = f.head_dim, vpt = D / 8, step = kSgThreads / vpt;
    const uint32_t w = threadIdx.x % vpt, i0 = threadIdx.x / vpt;
    const uint64_t row2 = (uint64_t)f.heads * D * 2;
    const int32_t* blocks = j.blocks + (size_t)(j.entry_base + c.e) * j.blocks_per_chunk;
    const uint64_t src0 = j.planes[c.p] + (uint64_t)c.h * D * 2 + (uint64_t)w * 16;
    const uint32_t slot0 = stage + threadIdx.x * 16;
    if (FULL && rows_e != c.e) {
#pragma unroll
        for (int u = 0; u < kSgVec; ++u) rows[u] = sg_row(f, blocks, i0 + u * step);
        rows_e = c.e;
    }
    bool bad = false;
#pragma unroll
    for (int u = 0; u < kSgVec; ++u) {
        const uint32_t i = i0 + u * step;
        if (FULL || i < n) {
            const uint32_t row = FULL ? rows[u] : sg_row(f, blocks, i);
            const uint32_t slot = slot0 + u * kSgThreads * 16;
            if (row == kNoRow) {
                bad = true;
                sts16_zero(slot);
            } else {
                cp_async16(slot, src0 + (uint64_t)row * row2);
            }
        }
    }
    if (bad) atomicCAS(j.err, 0, KVS_ERR_BOUNDS);
}

// Running max of |x| over BF16 pairs in one instruction (sm_86+): the result's
// magnitude is the larger magnitude, its sign the XOR of the signs (cleared at
// the end); a NaN input is ignored.  Infinities are not: a head whose maximum
// comes out infinite takes the exact finite amax (amax2) instead.
__device__ __forceinline__ uint32_t absmax2(uint32_t m2, uint32_t w) {
    uint32_t r;
    asm("max.xorsign.abs.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(m2), "r"(w));
    return r;
}

constexpr uint32_t kBf16Inf = 0x7F80u;

// Quantises segment c (n tokens) from this thread's slots of `stage` (its loads
// complete).  One barrier: every warp reads all warps' maxima (from the half of
// warp_max this segment's parity selects) and computes the reciprocal itself;
// a head holding an infinity takes one more barrier for its finite amax.
template <bool FULL>
__device__ __forceinline__ void sg_quantise(const Fp8Job& f, const SgCur& c, uint32_t n, uint32_t stage,
                                            uint32_t* warp_max, uint32_t* warp_max_fin) {
    const Job& j = f.job;
    const uint32_t H = f.heads, D = f.head_dim, vpt = D / 8, step = kSgThreads / vpt;
    const uint32_t t = threadIdx.x, w = t % vpt, i0 = t / vpt;
    const uint32_t slot0 = stage + t * 16;
    uint4 v[kSgVec];
#pragma unroll
    for (int u = 0; u < kSgVec; ++u) {
        v[u] = make_uint4(0, 0, 0, 0);
        if (FULL || i0 + u * step < n) v[u] = lds16(slot0 + u * kSgThreads * 16);
    }
    uint32_t x2 = 0;
#pragma unroll
    for (int u = 0; u < kSgVec; ++u)
        x2 = absmax2(absmax2(absmax2(absmax2(x2, v[u].x), v[u].y), v[u].z), v[u].w);
    x2 &= 0x7FFF7FFFu;                                      // never NaN: at most kBf16Inf per half
    uint32_t m = __reduce_max_sync(0xFFFFFFFFu, max(x2 & 0xFFFFu, x2 >> 16));
    if ((t & 31) == 0) warp_max[t >> 5] = m;
    __syncthreads();
    uint32_t a = __reduce_max_sync(0xFFFFFFFFu, warp_max[(t & 31) % (kSgThreads / 32)]);
    if (a == kBf16Inf) {                                    // uniform across the CTA
        uint32_t m2 = 0;
#pragma unroll
        for (int u = 0; u < kSgVec; ++u)
            m2 = amax2(amax2(amax2(amax2(m2, v[u].x), v[u].y), v[u].z), v[u].w);
        m = __reduce_max_sync(0xFFFFFFFFu, amax_bits(m2));
        if ((t & 31) == 0) warp_max_fin[t >> 5] = m;
        __syncthreads();
        a = __reduce_max_sync(0xFFFFFFFFu, warp_max_fin[(t & 31) % (kSgThreads / 32)]);
    }
    const float af = __uint_as_float(a << 16);
    const float inv = af > 0.0f ? __fdiv_rn(448.0f, af) : 1.0f;
    const uint64_t chunk = j.entries[c.e].chunk;
    if (t == 0) *reinterpret_cast<float*>(chunk + ((uint64_t)c.p * H + c.h) * 4) = af > 0.0f ? __fdiv_rn(af, 448.0f) : 1.0f;
    const uint64_t inv2 = ((uint64_t)__float_as_uint(inv) << 32) | __float_as_uint(inv);
    const uint64_t hd = (uint64_t)H * D;
    const uint64_t codes = chunk + f.scale_bytes + (uint64_t)c.p * n * hd + (uint64_t)c.h * D + (uint64_t)w * 8 +
                           (uint64_t)i0 * hd;
#pragma unroll
    for (int u = 0; u < kSgVec; ++u)
        if (FULL || i0 + u * step < n) st_cs8(codes + (uint64_t)(u * step) * hd, quant8_pk(v[u], inv2));
}

// CTA b takes segments [b * N / G, (b + 1) * N / G).  warp_max has two halves,
// alternating by segment: a warp writes a half again only two segments later,
// after the next segment's barrier, which every warp reaches only once it has
// read this segment's half.  warp_max_fin (heads holding an infinity) is
// written after a segment's first barrier and read before its next one.
static_assert(kSgThreads / 32 <= 32, "one lane per warp maximum");
__global__ void __launch_bounds__(kSgThreads, 1) kvs_fp8_store_staged_kernel(const Fp8Job f, uint32_t num_segments) {
    extern __shared__ __align__(128) uint8_t sg_stage[];
    __shared__ uint32_t warp_max[2][kSgThreads / 32];
    __shared__ uint32_t warp_max_fin[kSgThreads / 32];
    const uint32_t base = smem_u32(sg_stage);
    const uint32_t full_n = kSgVec * (kSgThreads / (f.head_dim / 8));
    const uint32_t lo = (uint32_t)((uint64_t)blockIdx.x * num_segments / gridDim.x);
    const uint32_t hi = (uint32_t)((uint64_t)(blockIdx.x + 1) * num_segments / gridDim.x);
    if (lo >= hi) return;                                   // uniform across the CTA
    const Entry* entries = f.job.entries;
    uint32_t rows[kSgVec];
    uint32_t rows_e = 0xFFFFFFFFu;
    SgCur ic = sg_at(f, lo), qc = ic;                       // issue / quantise cursors
    uint32_t issued = 0;
    // one commit group per segment slot, empty past the end, so wait_group counts segments
    auto issue = [&]() {
        if (lo + issued < hi) {
            const uint32_t n = (uint32_t)entries[ic.e].n_tok;
            const uint32_t stage = base + (issued % kSgStages) * kSgStageBytes;
            if (n == full_n) sg_issue<true>(f, ic, n, stage, rows, rows_e);
            else sg_issue<false>(f, ic, n, stage, rows, rows_e);
            sg_step(f, ic);
            ++issued;
        }
        cp_async_commit();
    };
    for (int s = 0; s + 1 < kSgStages; ++s) issue();
    for (uint32_t k = 0; lo + k < hi; ++k) {
        issue();
        cp_async_wait<kSgStages - 1>();
        const uint32_t n = (uint32_t)entries[qc.e].n_tok;
        const uint32_t stage = base + (k % kSgStages) * kSgStageBytes;
        if (n == full_n) sg_quantise<true>(f, qc, n, stage, warp_max[k & 1], warp_max_fin);
        else sg_quantise<false>(f, qc, n, stage, warp_max[k & 1], warp_max_fin);
        sg_step(f, qc);
    }
    cp_async_wait<0>();
}

constexpr int kStUnroll = 4;                         // vectors per thread in flight per step

// One CTA per (entry, plane) segment: the chunk's n tokens of that plane.
__global__ void __launch_bounds__(kStThreads) kvs_fp8_store_kernel(const Fp8Job f, uint32_t num_segments) {
    __shared__ uint32_t amax[kFp8MaxHeads];
    __shared__ float scale[kFp8MaxHeads];                    // holds 448 / amax per head
    const Job& j = f.job;
    const uint32_t H = f.heads, vph = f.head_dim / 16, vpr = H * vph;
    const uint64_t row2 = (uint64_t)H * f.head_dim * 2;          // BF16 bytes per token row
    for (uint32_t seg = blockIdx.x; seg < num_segments; seg += gridDim.x) {
        const uint32_t e = seg / j.num_planes;
        const uint32_t p = j.plane_begin + (seg - e * j.num_planes);
        const Entry en = j.entries[e];
        const uint32_t n = (uint32_t)en.n_tok;
        const int32_t* blocks = j.blocks + (size_t)(j.entry_base + e) * j.blocks_per_chunk;
        const uint64_t plane = j.planes[p];
        const uint64_t codes = en.chunk + f.scale_bytes + (uint64_t)p * n * vpr * 16;
        const uint32_t nvec = n * vpr;
        // source address of vector v (16 BF16 = 32 bytes), or 0 for a bad block
        auto src_of = [&](uint32_t v, uint32_t& h) -> uint64_t {
            const uint32_t i = v / vpr, w = v - i * vpr;
            h = w / vph;
            const int32_t blk = __ldg(blocks + i / j.block_size);
            if (blk < 0 || blk >= j.num_blocks) return 0;
            return plane + ((uint64_t)blk * j.block_size + i % j.block_size) * row2 + (uint64_t)w * 32;
        };
        for (uint32_t h = threadIdx.x; h < H; h += blockDim.x) amax[h] = 0;
        __syncthreads();
        // pass 1: per-head amax over the finite elements of this chunk's plane p
        uint32_t cur_h = 0xFFFFFFFFu, m = 0;
        bool bad = false;
        for (uint32_t v0 = threadIdx.x; v0 < nvec; v0 += blockDim.x * kStUnroll) {
            uint4 a[kStUnroll], b[kStUnroll];
            uint32_t hh[kStUnroll];
            bool ok[kStUnroll];
#pragma unroll
            for (int u = 0; u < kStUnroll; ++u) {
                const uint32_t v = v0 + u * blockDim.x;
                ok[u] = false;
                if (v < nvec) {
                    const uint64_t src = src_of(v, hh[u]);
                    if (src) {
                        a[u] = ld_nc16(src);
                        b[u] = ld_nc16(src + 16);
                        ok[u] = true;
                    } else {
                        bad = true;
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < kStUnroll; ++u) {
                if (!ok[u]) continue;
                const uint32_t lm = max(amax_bits8(a[u]), amax_bits8(b[u]));
                if (hh[u] != cur_h) {
                    if (cur_h != 0xFFFFFFFFu) atomicMax(&amax[cur_h], m);
                    cur_h = hh[u];
                    m = 0;
                }
                m = max(m, lm);
            }
        }
        if (cur_h != 0xFFFFFFFFu) atomicMax(&amax[cur_h], m);
        if (bad) atomicCAS(j.err, 0, KVS_ERR_BOUNDS);
        __syncthreads();
        for (uint32_t h = threadIdx.x; h < H; h += blockDim.x) {
            const float a = __uint_as_float(amax[h] << 16);
            const float s = a > 0.0f ? __fdiv_rn(a, 448.0f) : 1.0f;
            scale[h] = a > 0.0f ? __fdiv_rn(448.0f, a) : 1.0f;        // the inverse, for pass 2
            *reinterpret_cast<float*>(en.chunk + ((uint64_t)p * H + h) * 4) = s;
        }
        __syncthreads();
        // pass 2: quantise
        for (uint32_t v0 = threadIdx.x; v0 < nvec; v0 += blockDim.x * kStUnroll) {
            uint4 a[kStUnroll], b[kStUnroll];
            uint32_t hh[kStUnroll];
            bool ok[kStUnroll];
#pragma unroll
            for (int u = 0; u < kStUnroll; ++u) {
                const uint32_t v = v0 + u * blockDim.x;
                ok[u] = false;
                if (v < nvec) {
                    const uint64_t src = src_of(v, hh[u]);
                    if (src) {
                        a[u] = ld_nc16(src);
                        b[u] = ld_nc16(src + 16);
                        ok[u] = true;
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < kStUnroll; ++u)
                if (ok[u]) st_cs16(codes + (uint64_t)(v0 + u * blockDim.x) * 16, quant16(a[u], b[u], scale[hh[u]]));
        }
        __syncthreads();                                   // amax / scale are reused by the next segment
    }
}

constexpr int kMaxDev = 64;
int g_sms[kMaxDev];                      // SM count per device
bool g_sg_attr[kMaxDev];                 // dynamic shared memory limit of the staged store raised
bool g_fs_attr[kMaxDev];                 // ... of the few-SM retrieval

int sm_count() {
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= kMaxDev) dev = 0;
    if (g_sms[dev] == 0) {
        int n = 0;
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        g_sms[dev] = n > 0 ? n : 1;
    }
    return g_sms[dev];
}

}  // namespace

cudaError_t launch_fp8_retrieve(const Fp8Job& fj, int grid, cudaStream_t s) {
    const uint64_t n = fj.job.num_pieces;
    if (n == 0) return cudaSuccess;
    if (grid == kFp8PerPiece) {
        kvs_fp8_retrieve_piece_kernel<<<(uint32_t)n, kRtThreads, 0, s>>>(fj);
        return cudaGetLastError();
    }
    int per_sm = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kvs_fp8_retrieve_kernel, kRtThreads, 0);
    const int full = sm_count() * std::max(per_sm, 1);
    if (grid <= 0 || grid > full) grid = full;
    if ((uint64_t)grid > n) grid = (int)n;
    kvs_fp8_retrieve_kernel<<<grid, kRtThreads, 0, s>>>(fj, (uint32_t)n);
    return cudaGetLastError();
}

cudaError_t launch_fp8_retrieve_staged(const Fp8Job& fj, int grid, cudaStream_t s) {
    const uint64_t n = fj.job.num_pieces;
    if (n == 0) return cudaSuccess;
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= kMaxDev) dev = 0;
    if (!g_fs_attr[dev]) {
        cudaError_t e = cudaFuncSetAttribute(kvs_fp8_retrieve_staged_kernel,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kFsSmemBytes);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(kvs_fp8_retrieve_staged_kernel, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
        if (e != cudaSuccess) return e;
        g_fs_attr[dev] = true;
    }
    const int full = sm_count() * 2;
    if (grid <= 0 || grid > full) grid = full;
    if ((uint64_t)grid > n) grid = (int)n;
    kvs_fp8_retrieve_staged_kernel<<<grid, kFsThreads, kFsSmemBytes, s>>>(fj, (uint32_t)n);
    return cudaGetLastError();
}

cudaError_t launch_fp8_store(const Fp8Job& fj, int grid, cudaStream_t s, uint32_t chunk_tokens, bool staged) {
    const uint32_t vpt = fj.head_dim / 8;
    if ((uint64_t)chunk_tokens * fj.head_dim <= kHeadMaxElems && kStThreads % vpt == 0 && chunk_tokens < 65536 &&
        fj.job.block_size < 65536) {
        const uint64_t segs = (uint64_t)fj.job.num_entries * fj.job.num_planes * fj.heads;
        if (segs == 0) return cudaSuccess;
        // the staged kernel needs D/8 to divide its CTA and plane rows below 2^32 - 1
        if (staged && kSgThreads % vpt == 0 && (uint64_t)fj.job.num_blocks * fj.job.block_size < 0xFFFFFFFFull) {
            int dev = 0;
            cudaGetDevice(&dev);
            if (dev < 0 || dev >= kMaxDev) dev = 0;
            if (!g_sg_attr[dev]) {
                const cudaError_t e = cudaFuncSetAttribute(kvs_fp8_store_staged_kernel,
                                                           cudaFuncAttributeMaxDynamicSharedMemorySize, kSgSmemBytes);
                if (e != cudaSuccess) return e;
                g_sg_attr[dev] = true;
            }
            if (grid <= 0 || grid > sm_count()) grid = sm_count();
            if ((uint64_t)grid > segs) grid = (int)segs;
            kvs_fp8_store_staged_kernel<<<grid, kSgThreads, kSgSmemBytes, s>>>(fj, (uint32_t)segs);
            return cudaGetLastError();
        }
        if (grid <= 0 || (uint64_t)grid > segs) grid = (int)std::min<uint64_t>(segs, 1u << 30);
        kvs_fp8_store_head_kernel<<<grid, kStThreads, 0, s>>>(fj, (uint32_t)segs);
        return cudaGetLastError();
    }
    const uint64_t segs = (uint64_t)fj.job.num_entries * fj.job.num_planes;
    if (segs == 0) return cudaSuccess;
    if (grid <= 0 || (uint64_t)grid > segs) grid = (int)segs;
    kvs_fp8_store_kernel<<<grid, kStThreads, 0, s>>>(fj, (uint32_t)segs);
    return cudaGetLastError();
}

}  // namespace kvs

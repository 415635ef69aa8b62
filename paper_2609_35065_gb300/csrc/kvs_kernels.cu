// kvs_kernels.cu -- copy kernels for prefix-KV retrieval / store-back on sm_103a.
//
// The work is pure data movement (TempoKV reuses the runtime's transfer path
// into the paged cache, Sec. 4): every run is one contiguous B*R-byte copy
// between a chunk buffer [L][2][n][H][D] and one paged block of one
// (layer, K/V) plane [NB][B][H][D].  Two flavours:
//
//  * LDG: the threads of a CTA move one 32 KiB piece with 16-byte vector
//    loads (non-coherent, no L1 allocation) issued ahead of 16-byte streaming
//    stores.  Uncapped 16-byte work runs one 512-thread, 28-register CTA per
//    piece (kvs_ldg_piece_kernel, four CTAs per SM); capped grids, narrower
//    vectors and the validation compare run a 256-thread grid-stride kernel.
//  * LINK: the LDG scheme double-buffered in registers (the next piece's loads
//    are issued before the current piece is stored), for host-resident
//    chunks whose loads/stores cross the long-latency host link.
//  * TMA: 1-D bulk async copies through shared memory (cp.async.bulk
//    global->shared completing on an mbarrier, then a shared->global bulk
//    store).  Uncapped work runs one 32-thread CTA per piece (six per SM);
//    a capped grid runs one thread per CTA driving a ring of stages.  Every
//    wait is bounded by the global timer and reports KVS_ERR_TIMEOUT instead
//    of hanging.
#include <algorithm>
#include <cstdint>

#include "kvs.h"
#include "kvs_async.cuh"
#include "kvs_internal.h"

namespace kvs {
namespace {

// ---------------------------------------------------------------------------
// Division by a launch-invariant divisor d, for dividends below 2^31: with
// p = 31 + ceil(log2 d) and m = ceil(2^p / d), floor(n / d) = (n * m) >> p
// (round-up reciprocal method; the error term n*(m*d - 2^p)/(d*2^p) stays
// below 1/d).  m < 2^32 for every d >= 1.
// ---------------------------------------------------------------------------
struct FastDiv {
    uint32_t d, m, p;
};

FastDiv make_fastdiv(uint32_t d) {
    uint32_t l = 0;
    while ((1ull << l) < d) ++l;
    FastDiv f;
    f.d = d;
    f.p = 31 + l;
    f.m = (uint32_t)(((1ull << f.p) + d - 1) / d);
    return f;
}

__device__ __forceinline__ uint32_t fdiv(uint32_t n, const FastDiv& f) {
    return (uint32_t)(((uint64_t)n * f.m) >> f.p);
}

struct Decoder {
    Job job;
    FastDiv ppr, bpc, planes;
};

struct Piece {
    uint64_t chunk_addr;
    uint64_t plane_addr;
    uint32_t len;
};

// Piece q -> addresses.  Returns false for pieces with nothing to move
// (past the end of a short chunk, a skipped block, a bounds violation).
__device__ __forceinline__ bool decode_piece(const Decoder& dc, uint32_t q, Piece& pc) {
    const Job& j = dc.job;
    const uint32_t g = fdiv(q, dc.ppr);
    const uint32_t k = q - g * dc.ppr.d;
    const uint32_t ep = fdiv(g, dc.bpc);
    const uint32_t i = g - ep * dc.bpc.d;
    const uint32_t e = fdiv(ep, dc.planes);
    const uint32_t p = j.plane_begin + (ep - e * dc.planes.d);
    // The two descriptor loads are independent, so both are in flight at once.
    const int32_t blk = __ldg(j.blocks + (size_t)(j.entry_base + e) * j.blocks_per_chunk + i);
    const Entry en = j.entries[e];
    const int64_t first = (int64_t)i * j.block_size;
    const int64_t ntok = min((int64_t)j.block_size, (int64_t)en.n_tok - first);
    if (ntok <= 0) return false;
    if (blk < 0) return false;
    if (blk >= j.num_blocks) {
        atomicCAS(j.err, 0, KVS_ERR_BOUNDS);
        return false;
    }
    const uint64_t run_bytes = (uint64_t)ntok * j.row_bytes;
    const uint64_t off = (uint64_t)k * j.piece_bytes;
    if (off >= run_bytes) return false;
    pc.len = (uint32_t)min((uint64_t)j.piece_bytes, run_bytes - off);
    pc.chunk_addr = en.chunk + ((uint64_t)p * (uint64_t)en.n_tok + (uint64_t)first) * j.row_bytes + off;
    pc.plane_addr = j.planes[p] + (uint64_t)blk * j.block_size * j.row_bytes + off;
    return true;
}

// ---------------------------------------------------------------------------
// Vector loads / stores.
// ---------------------------------------------------------------------------
template <int V> struct Vec;
template <> struct Vec<16> { using T = uint4; };
template <> struct Vec<8>  { using T = uint2; };
template <> struct Vec<4>  { using T = uint32_t; };
template <> struct Vec<2>  { using T = uint16_t; };
template <> struct Vec<1>  { using T = uint8_t; };

template <int V>
__device__ __forceinline__ typename Vec<V>::T ld_stream(const typename Vec<V>::T* p) {
    if constexpr (V == 16) {
        uint4 r;
        asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                     : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "l"(p));
        return r;
    } else {
        return __ldg(p);
    }
}

template <int V>
__device__ __forceinline__ void st_stream(typename Vec<V>::T* p, const typename Vec<V>::T& v) {
    if constexpr (V == 16) {
        asm volatile("st.global.cs.v4.u32 [%0], {%1,%2,%3,%4};"
                     :: "l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w) : "memory");
    } else {
        *p = v;
    }
}

template <int V>
__device__ __forceinline__ bool vec_equal(const typename Vec<V>::T& a, const typename Vec<V>::T& b) {
    if constexpr (V == 16) {
        return a.x == b.x && a.y == b.y && a.z == b.z && a.w == b.w;
    } else if constexpr (V == 8) {
        return a.x == b.x && a.y == b.y;
    } else {
        return a == b;
    }
}

// All threads of the CTA copy `len` bytes (a multiple of V) from src to dst:
// U independent loads per thread are in flight before their stores.
template <int V, int U>
__device__ __forceinline__ void copy_piece(uint64_t src, uint64_t dst, uint32_t len) {
    using T = typename Vec<V>::T;
    const T* s = reinterpret_cast<const T*>(src);
    T* d = reinterpret_cast<T*>(dst);
    const uint32_t n = len / V;
    const uint32_t stride = blockDim.x;
    for (uint32_t base = threadIdx.x; base < n; base += stride * U) {
        T r[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const uint32_t k = base + u * stride;
            if (k < n) r[u] = ld_stream<V>(s + k);
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const uint32_t k = base + u * stride;
            if (k < n) st_stream<V>(d + k, r[u]);
        }
    }
}

template <int V, int U>
__device__ __forceinline__ bool equal_piece(uint64_t a_addr, uint64_t b_addr, uint32_t len) {
    using T = typename Vec<V>::T;
    const T* a = reinterpret_cast<const T*>(a_addr);
    const T* b = reinterpret_cast<const T*>(b_addr);
    const uint32_t n = len / V;
    bool same = true;
    for (uint32_t k = threadIdx.x; k < n; k += blockDim.x)
        same &= vec_equal<V>(ld_stream<V>(a + k), ld_stream<V>(b + k));
    return same;
}

constexpr int kLdgThreads = 256;
constexpr int kLdgUnroll = 8;

template <int V, int MODE>
__global__ void __launch_bounds__(kLdgThreads) kvs_ldg_kernel(const Decoder dc, uint32_t num_pieces) {
    const Job& j = dc.job;
    for (uint32_t q = blockIdx.x; q < num_pieces; q += gridDim.x) {
        Piece pc;
        if (!decode_piece(dc, q, pc)) continue;          // uniform across the CTA
        if constexpr (MODE == MODE_RETRIEVE) {
            copy_piece<V, kLdgUnroll>(pc.chunk_addr, pc.plane_addr, pc.len);
        } else if constexpr (MODE == MODE_STORE) {
            copy_piece<V, kLdgUnroll>(pc.plane_addr, pc.chunk_addr, pc.len);
        } else {
            if (!equal_piece<V, kLdgUnroll>(pc.chunk_addr, pc.plane_addr, pc.len))
                atomicCAS(j.err, 0, KVS_ERR_ALIAS);
        }
    }
}

// Whole-GPU flavour for 16-byte aligned work: exactly one CTA per piece, 512
// threads x 4 vectors.  The launch bound caps the kernel at 32 registers, so
// four CTAs (2048 threads, 128 KiB of loads in flight) fit on an SM, twice the
// residency of kvs_ldg_kernel<16>.
constexpr int kPieceThreads = 512;
constexpr int kPieceUnroll = kPieceBytes / 16 / kPieceThreads;

template <int MODE>
__global__ void __launch_bounds__(kPieceThreads, 4) kvs_ldg_piece_kernel(const Decoder dc) {
    static_assert(kPieceUnroll * kPieceThreads * 16 == kPieceBytes, "one piece per CTA");
    Piece pc;
    if (!decode_piece(dc, blockIdx.x, pc)) return;       // uniform across the CTA
    const uint4* s = reinterpret_cast<const uint4*>(MODE == MODE_RETRIEVE ? pc.chunk_addr : pc.plane_addr);
    uint4* d = reinterpret_cast<uint4*>(MODE == MODE_RETRIEVE ? pc.plane_addr : pc.chunk_addr);
    const uint32_t n = pc.len / 16;
    uint4 r[kPieceUnroll];
    if (n == kPieceThreads * kPieceUnroll) {
#pragma unroll
        for (int u = 0; u < kPieceUnroll; ++u) r[u] = ld_stream<16>(s + threadIdx.x + u * kPieceThreads);
#pragma unroll
        for (int u = 0; u < kPieceUnroll; ++u) st_stream<16>(d + threadIdx.x + u * kPieceThreads, r[u]);
    } else {                                             // a short run: the tail of a partial chunk
#pragma unroll
        for (int u = 0; u < kPieceUnroll; ++u) {
            const uint32_t k = threadIdx.x + u * kPieceThreads;
            if (k < n) r[u] = ld_stream<16>(s + k);
        }
#pragma unroll
        for (int u = 0; u < kPieceUnroll; ++u) {
            const uint32_t k = threadIdx.x + u * kPieceThreads;
            if (k < n) st_stream<16>(d + k, r[u]);
        }
    }
}

// Host-link flavour: each thread keeps two pieces' worth of 16-byte vectors in
// registers, so the loads of the next piece are in flight while the current
// one is stored.  A CTA then always has 32-64 KiB outstanding over the
// long-latency host link, and a small grid saturates it.
__device__ __forceinline__ bool next_piece_ldg(const Decoder& dc, uint32_t num_pieces, uint32_t& q, Piece& pc) {
    while (q < num_pieces) {
        const uint32_t cur = q;
        q += gridDim.x;
        if (decode_piece(dc, cur, pc)) return true;
    }
    return false;
}

__device__ __forceinline__ void load_piece16(uint64_t src, uint32_t len, uint4 (&r)[kLdgUnroll]) {
    const uint4* s = reinterpret_cast<const uint4*>(src);
    const uint32_t n = len / 16;
#pragma unroll
    for (int u = 0; u < kLdgUnroll; ++u) {
        const uint32_t k = threadIdx.x + u * kLdgThreads;
        if (k < n) r[u] = ld_stream<16>(s + k);
    }
}

__device__ __forceinline__ void store_piece16(uint64_t dst, uint32_t len, const uint4 (&r)[kLdgUnroll]) {
    uint4* d = reinterpret_cast<uint4*>(dst);
    const uint32_t n = len / 16;
#pragma unroll
    for (int u = 0; u < kLdgUnroll; ++u) {
        const uint32_t k = threadIdx.x + u * kLdgThreads;
        if (k < n) st_stream<16>(d + k, r[u]);
    }
}

template <int MODE>
__global__ void __launch_bounds__(kLdgThreads) kvs_link_kernel(const Decoder dc, uint32_t num_pieces) {
    static_assert(kPieceBytes == kLdgUnroll * kLdgThreads * 16, "one piece per register set");
    constexpr bool to_plane = (MODE == MODE_RETRIEVE);
    uint4 ra[kLdgUnroll], rb[kLdgUnroll];
    Piece pa, pb;
    uint32_t q = blockIdx.x;
    bool ha = next_piece_ldg(dc, num_pieces, q, pa);
    if (ha) load_piece16(to_plane ? pa.chunk_addr : pa.plane_addr, pa.len, ra);
    while (ha) {
        const bool hb = next_piece_ldg(dc, num_pieces, q, pb);
        if (hb) load_piece16(to_plane ? pb.chunk_addr : pb.plane_addr, pb.len, rb);
        store_piece16(to_plane ? pa.plane_addr : pa.chunk_addr, pa.len, ra);
        if (!hb) break;
        ha = next_piece_ldg(dc, num_pieces, q, pa);
        if (ha) load_piece16(to_plane ? pa.chunk_addr : pa.plane_addr, pa.len, ra);
        store_piece16(to_plane ? pb.plane_addr : pb.chunk_addr, pb.len, rb);
    }
}

// Few-SM flavour of the host-link retrieval (KVS_F_FEW_SMS).  Beside a kernel
// whose CTAs fill whole SMs (a GEMM), every SM that holds a copy CTA is lost to
// it, so what matters is the bytes in flight per SM.  Each thread keeps one
// piece in registers, as the link kernel does, and three more in shared
// memory, copied there with cp.async into slots that only it reads back (no
// CTA barrier; cp.async.wait_group orders them): 128 KiB per CTA and two CTAs
// per SM, 256 KiB per SM against the link kernel's 192.  Piece i of a CTA
// lives in slot i % 4 -- slot 0 the registers, slots 1-3 shared memory -- and
// its successor i + 4 is issued into the slot as soon as piece i is stored.
// Pieces come in grid-stride order, so once a slot finds none left, neither
// does any slot after it.
constexpr int kStagedSmemPieces = 3;
constexpr int kStagedSlots = 1 + kStagedSmemPieces;
constexpr uint32_t kStagedSmemBytes = kStagedSmemPieces * kPieceBytes;

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

// This thread's vectors of a piece into its slots of shared-memory stage `stage`.
__device__ __forceinline__ void stage_piece16(uint64_t src, uint32_t len, uint32_t stage) {
    const uint32_t n = len / 16;
#pragma unroll
    for (int u = 0; u < kLdgUnroll; ++u) {
        const uint32_t k = threadIdx.x + u * kLdgThreads;
        if (k < n) cp_async16(stage + k * 16, src + (uint64_t)k * 16);
    }
}

// ... and from its slots to `dst` (the thread's own cp.async copies are complete).
__device__ __forceinline__ void unstage_piece16(uint64_t dst, uint32_t len, uint32_t stage) {
    const uint32_t n = len / 16;
    uint4 v[kLdgUnroll];
#pragma unroll
    for (int u = 0; u < kLdgUnroll; ++u) {
        const uint32_t k = threadIdx.x + u * kLdgThreads;
        if (k < n)
            asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                         : "=r"(v[u].x), "=r"(v[u].y), "=r"(v[u].z), "=r"(v[u].w) : "r"(stage + k * 16));
    }
    store_piece16(dst, len, v);
}

__global__ void __launch_bounds__(kLdgThreads, 2) kvs_link_staged_kernel(const Decoder dc, uint32_t num_pieces) {
    extern __shared__ __align__(128) uint8_t link_stage[];
    const uint32_t base = smem_u32(link_stage);
    uint4 r[kLdgUnroll];
    Piece pc[kStagedSlots];
    bool has[kStagedSlots];
    uint32_t q = blockIdx.x;
    // fill slot s with the CTA's next piece; a shared-memory slot always commits
    // one group (empty past the end), so wait_group counts pieces
    auto fill = [&](int s) {
        has[s] = next_piece_ldg(dc, num_pieces, q, pc[s]);
        if (s == 0) {
            if (has[s]) load_piece16(pc[s].chunk_addr, pc[s].len, r);
        } else {
            if (has[s]) stage_piece16(pc[s].chunk_addr, pc[s].len, base + (s - 1) * kPieceBytes);
            cp_async_commit();
        }
    };
#pragma unroll
    for (int s = 0; s < kStagedSlots; ++s) fill(s);
    bool more = true;
    while (more) {
#pragma unroll
        for (int s = 0; s < kStagedSlots; ++s) {
            if (more && !has[s]) more = false;
            if (more) {
                if (s == 0) {
                    store_piece16(pc[s].plane_addr, pc[s].len, r);
                } else {
                    // the kStagedSmemPieces - 1 younger shared-memory pieces may still be in flight
                    cp_async_wait<kStagedSmemPieces - 1>();
                    unstage_piece16(pc[s].plane_addr, pc[s].len, base + (s - 1) * kPieceBytes);
                }
                fill(s);
            }
        }
    }
    cp_async_wait<0>();
}

// L2-prefetch flavour of the host-link retrieval.  Over the host link a piece's
// loads take ~15 us beside a busy GPU, so the plain flavour needs ~3 MiB of
// loads in flight, held in registers: 16 or more SMs' worth of CTAs.  Here the
// CTA's thread 0 keeps the CTA's next `ahead` pieces in flight as bulk L2
// prefetches (cp.async.bulk.prefetch.L2, which holds no registers or shared
// memory), so the bytes in flight wait in L2; the CTA's own loads then find
// their piece in L2 and the grid can be small.  Prefetches of a piece that
// are still in flight, or evicted, only cost time: the loads fetch the bytes
// themselves either way.
__device__ __forceinline__ void prefetch_l2(uint64_t addr, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" :: "l"(addr), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool next_piece_pf(const Decoder& dc, uint32_t num_pieces, uint32_t stride_ahead,
                                              uint32_t& q, Piece& pc) {
    while (q < num_pieces) {
        const uint32_t cur = q;
        q += gridDim.x;
        if (threadIdx.x == 0) {
            const uint32_t f = cur + stride_ahead;            // < 2^32: both terms are below 2^31
            Piece pf;
            if (f < num_pieces && decode_piece(dc, f, pf)) prefetch_l2(pf.chunk_addr, pf.len);
        }
        if (decode_piece(dc, cur, pc)) return true;
    }
    return false;
}

__global__ void __launch_bounds__(kLdgThreads) kvs_link_pf_kernel(const Decoder dc, uint32_t num_pieces,
                                                                  uint32_t ahead) {
    const uint32_t stride_ahead = ahead * gridDim.x;
    if (threadIdx.x == 0)
        for (uint32_t k = 0; k < ahead; ++k) {
            const uint32_t f = blockIdx.x + k * gridDim.x;
            Piece pf;
            if (f < num_pieces && decode_piece(dc, f, pf)) prefetch_l2(pf.chunk_addr, pf.len);
        }
    uint4 ra[kLdgUnroll], rb[kLdgUnroll];
    Piece pa, pb;
    uint32_t q = blockIdx.x;
    bool ha = next_piece_pf(dc, num_pieces, stride_ahead, q, pa);
    if (ha) load_piece16(pa.chunk_addr, pa.len, ra);
    while (ha) {
        const bool hb = next_piece_pf(dc, num_pieces, stride_ahead, q, pb);
        if (hb) load_piece16(pb.chunk_addr, pb.len, rb);
        store_piece16(pa.plane_addr, pa.len, ra);
        if (!hb) break;
        ha = next_piece_pf(dc, num_pieces, stride_ahead, q, pa);
        if (ha) load_piece16(pa.chunk_addr, pa.len, ra);
        store_piece16(pb.plane_addr, pb.len, rb);
    }
}

// Plane-major decode for the signalling kernel: q -> (plane, entry, block, piece).
__device__ __forceinline__ bool decode_piece_plane_major(const Decoder& dc, const FastDiv& entries, uint32_t q,
                                                         uint32_t& p_rel, Piece& pc) {
    const Job& j = dc.job;
    const uint32_t g = fdiv(q, dc.ppr);
    const uint32_t k = q - g * dc.ppr.d;
    const uint32_t g2 = fdiv(g, dc.bpc);
    const uint32_t i = g - g2 * dc.bpc.d;
    p_rel = fdiv(g2, entries);
    const uint32_t e = g2 - p_rel * entries.d;
    const uint32_t p = j.plane_begin + p_rel;
    const int32_t blk = __ldg(j.blocks + (size_t)(j.entry_base + e) * j.blocks_per_chunk + i);
    const Entry en = j.entries[e];
    const int64_t first = (int64_t)i * j.block_size;
    const int64_t ntok = min((int64_t)j.block_size, (int64_t)en.n_tok - first);
    if (ntok <= 0 || blk < 0) return false;
    if (blk >= j.num_blocks) {
        atomicCAS(j.err, 0, KVS_ERR_BOUNDS);
        return false;
    }
    const uint64_t run_bytes = (uint64_t)ntok * j.row_bytes;
    const uint64_t off = (uint64_t)k * j.piece_bytes;
    if (off >= run_bytes) return false;
    pc.len = (uint32_t)min((uint64_t)j.piece_bytes, run_bytes - off);
    pc.chunk_addr = en.chunk + ((uint64_t)p * (uint64_t)en.n_tok + (uint64_t)first) * j.row_bytes + off;
    pc.plane_addr = j.planes[p] + (uint64_t)blk * j.block_size * j.row_bytes + off;
    return true;
}

// Counts piece q as done; the CTA completing its group publishes the flag.
__device__ __forceinline__ void piece_done(const Signal& sg, uint32_t p_rel, uint32_t group_pieces_full,
                                           uint32_t last_group_pieces) {
    __threadfence();                               // this thread's stores of the piece
    __syncthreads();
    if (threadIdx.x == 0) {
        const uint32_t grp = p_rel / sg.planes_per_group;
        const uint32_t total = (grp + 1 == sg.groups) ? last_group_pieces : group_pieces_full;
        if (atomicAdd(&sg.counters[grp], 1u) + 1u == total) {
            __threadfence();
            atomicExch(&sg.flags[grp], sg.gen);
        }
    }
}

template <int MODE>
__global__ void __launch_bounds__(kLdgThreads) kvs_link_signal_kernel(const Decoder dc, const FastDiv entries,
                                                                      const Signal sg, uint32_t num_pieces) {
    constexpr bool to_plane = (MODE == MODE_RETRIEVE);
    const Job& j = dc.job;
    const uint32_t per_plane = j.num_entries * j.blocks_per_chunk * j.pieces_per_run;
    const uint32_t group_full = sg.planes_per_group * per_plane;
    const uint32_t last_group = (j.num_planes - (sg.groups - 1) * sg.planes_per_group) * per_plane;
    uint4 ra[kLdgUnroll], rb[kLdgUnroll];
    Piece pa, pb;
    uint32_t qa = blockIdx.x, qb, pra = 0, prb = 0;
    bool ha = qa < num_pieces, va = false, vb = false;
    if (ha && (va = decode_piece_plane_major(dc, entries, qa, pra, pa)))
        load_piece16(to_plane ? pa.chunk_addr : pa.plane_addr, pa.len, ra);
    while (ha) {
        qb = qa + gridDim.x;
        const bool hb = qb < num_pieces;
        vb = hb && decode_piece_plane_major(dc, entries, qb, prb, pb);
        if (vb) load_piece16(to_plane ? pb.chunk_addr : pb.plane_addr, pb.len, rb);
        if (va) store_piece16(to_plane ? pa.plane_addr : pa.chunk_addr, pa.len, ra);
        piece_done(sg, fdiv(fdiv(fdiv(qa, dc.ppr), dc.bpc), entries), group_full, last_group);
        if (!hb) break;
        qa = qb + gridDim.x;
        ha = qa < num_pieces;
        va = ha && decode_piece_plane_major(dc, entries, qa, pra, pa);
        if (va) load_piece16(to_plane ? pa.chunk_addr : pa.plane_addr, pa.len, ra);
        if (vb) store_piece16(to_plane ? pb.plane_addr : pb.chunk_addr, pb.len, rb);
        piece_done(sg, fdiv(fdiv(fdiv(qb, dc.ppr), dc.bpc), entries), group_full, last_group);
    }
    // The last CTA to finish writes every flag (all groups are complete by then).
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        if (atomicAdd(sg.ctas_done, 1u) + 1u == gridDim.x)
            for (uint32_t g = 0; g < sg.groups; ++g) atomicExch(&sg.flags[g], sg.gen);
    }
}

__global__ void __launch_bounds__(kLdgThreads) kvs_flat_copy_kernel(uint64_t dst, uint64_t src, uint64_t bytes) {
    const uint64_t pieces = (bytes + kPieceBytes - 1) / kPieceBytes;
    for (uint64_t q = blockIdx.x; q < pieces; q += gridDim.x) {
        const uint64_t off = q * kPieceBytes;
        const uint32_t len = (uint32_t)min((uint64_t)kPieceBytes, bytes - off);
        copy_piece<16, kLdgUnroll>(src + off, dst + off, len);
    }
}

// ---------------------------------------------------------------------------
// TMA flavour: bulk async copies through a ring of shared-memory stages.
// ---------------------------------------------------------------------------
constexpr int kTmaStages = 6;
// One elected thread runs the whole pipeline: piece k of this CTA lives in
// stage k % S; S-1 loads are kept in flight; before a stage is refilled the
// bulk store that read it (one iteration earlier) must have finished reading.
template <int S>
__global__ void __launch_bounds__(32, 1) kvs_tma_kernel(const Decoder dc, uint32_t num_pieces) {
    extern __shared__ __align__(128) uint8_t stage_mem[];
    __shared__ __align__(8) uint64_t bars[S];
    if (threadIdx.x != 0) return;
    const Job& j = dc.job;
    const uint32_t piece_bytes = j.piece_bytes;
    const bool to_plane = (j.mode == MODE_RETRIEVE);

    for (int s = 0; s < S; ++s) mbar_init(smem_u32(&bars[s]), 1);
    mbar_init_fence();

    uint32_t cursor = blockIdx.x;
    auto next_piece = [&](Piece& out) -> bool {
        while (cursor < num_pieces) {
            const uint32_t q = cursor;
            cursor += gridDim.x;
            if (decode_piece(dc, q, out)) return true;
        }
        return false;
    };
    Piece pend[S] = {};
    auto issue_load = [&](int s) {
        const uint32_t bar = smem_u32(&bars[s]);
        mbar_expect_tx(bar, pend[s].len);
        bulk_load(smem_u32(stage_mem + (size_t)s * piece_bytes),
                  to_plane ? pend[s].chunk_addr : pend[s].plane_addr, pend[s].len, bar);
    };

    uint32_t loaded = 0;
    for (int s = 0; s < S - 1; ++s) {
        if (!next_piece(pend[s])) break;
        issue_load(s);
        ++loaded;
    }
    for (uint32_t k = 0; k < loaded; ++k) {
        const int s = (int)(k % S);
        if (!mbar_wait(smem_u32(&bars[s]), (k / S) & 1u, kWaitLimitNs)) {
            atomicCAS(j.err, 0, KVS_ERR_TIMEOUT);
            // Let the loads still in flight land (bounded) before leaving.
            for (uint32_t r = k; r < loaded; ++r)
                mbar_wait(smem_u32(&bars[r % S]), (r / S) & 1u, kWaitLimitNs);
            break;
        }
        bulk_store(to_plane ? pend[s].plane_addr : pend[s].chunk_addr,
                   smem_u32(stage_mem + (size_t)s * piece_bytes), pend[s].len);
        bulk_commit();
        Piece nx;
        if (next_piece(nx)) {
            const int s2 = (int)((k + S - 1) % S);
            bulk_wait_read<1>();
            pend[s2] = nx;
            issue_load(s2);
            ++loaded;
        }
    }
    bulk_wait_all();
}

// Whole-GPU TMA flavour: exactly one 32-thread CTA per piece; its elected
// thread moves the piece through 32 KiB of shared memory with one bulk load
// (completing on an mbarrier, bounded wait) and one bulk store, and leaves once
// the store has read the stage.  Shared memory allows six such CTAs per SM,
// 192 KiB of loads in flight, with almost no registers.
template <int MODE>
__global__ void __launch_bounds__(32) kvs_tma_piece_kernel(const Decoder dc) {
    extern __shared__ __align__(128) uint8_t stage[];
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x != 0) return;
    Piece pc;
    if (!decode_piece(dc, blockIdx.x, pc)) return;
    const uint32_t b = smem_u32(&bar);
    mbar_init(b, 1);
    mbar_init_fence();
    mbar_expect_tx(b, pc.len);
    bulk_load(smem_u32(stage), MODE == MODE_RETRIEVE ? pc.chunk_addr : pc.plane_addr, pc.len, b);
    if (!mbar_wait(b, 0, kWaitLimitNs)) {
        atomicCAS(dc.job.err, 0, KVS_ERR_TIMEOUT);
        mbar_wait(b, 0, kWaitLimitNs);             // let the load land before the stage goes away
        return;
    }
    bulk_store(MODE == MODE_RETRIEVE ? pc.plane_addr : pc.chunk_addr, smem_u32(stage), pc.len);
    bulk_commit();
    bulk_wait_read<0>();
}

// Waits on a barrier phase that nothing completes; the bounded wait must give up.
__global__ void kvs_stall_kernel(int32_t* err, uint64_t limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x != 0) return;
    mbar_init(smem_u32(&bar), 1);
    mbar_init_fence();
    if (!mbar_wait(smem_u32(&bar), 0, limit_ns)) atomicCAS(err, 0, KVS_ERR_TIMEOUT);
}

Decoder make_decoder(const Job& job) {
    Decoder dc;
    dc.job = job;
    dc.ppr = make_fastdiv(job.pieces_per_run);
    dc.bpc = make_fastdiv(job.blocks_per_chunk);
    dc.planes = make_fastdiv(job.num_planes);
    return dc;
}

// Per-device facts, looked up once per device (a process may drive several GPUs).
constexpr int kMaxDevices = 64;
int g_sms[kMaxDevices];
size_t g_tma_smem[kMaxDevices];          // dynamic shared memory the TMA kernel may use
bool g_tma_piece_cfg[kMaxDevices];       // carveout preference of the per-piece TMA kernel set

int current_device() {
    int dev = 0;
    cudaGetDevice(&dev);
    return (dev >= 0 && dev < kMaxDevices) ? dev : 0;
}

int num_sms() {
    const int dev = current_device();
    if (g_sms[dev] == 0) {
        int n = 0;
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        g_sms[dev] = n > 0 ? n : 1;
    }
    return g_sms[dev];
}

int clamp_grid(int grid, int per_sm, uint64_t pieces) {
    int full = num_sms() * per_sm;
    if (grid <= 0 || grid > full) grid = full;
    if ((uint64_t)grid > pieces) grid = (int)pieces;
    return grid < 1 ? 1 : grid;
}

// With no cap, one CTA per piece: the hardware block scheduler keeps every SM
// busy and overlaps one CTA's stores with the next CTA's loads.  Measured on a
// 2 GiB HBM copy this reaches 7.1 TB/s (read + write) against 6.5-6.7 TB/s for
// persistent grid-stride grids of any shape.
template <int V>
cudaError_t launch_ldg_v(const Job& job, int grid, cudaStream_t s) {
    const Decoder dc = make_decoder(job);
    const uint32_t n = (uint32_t)job.num_pieces;
    if (V == 16 && grid <= 0 && job.mode != MODE_COMPARE) {
        if (job.mode == MODE_RETRIEVE)
            kvs_ldg_piece_kernel<MODE_RETRIEVE><<<n, kPieceThreads, 0, s>>>(dc);
        else
            kvs_ldg_piece_kernel<MODE_STORE><<<n, kPieceThreads, 0, s>>>(dc);
        return cudaGetLastError();
    }
    grid = grid > 0 ? clamp_grid(grid, ldg_ctas_per_sm(), job.num_pieces) : (int)job.num_pieces;
    if (job.mode == MODE_RETRIEVE)
        kvs_ldg_kernel<V, MODE_RETRIEVE><<<grid, kLdgThreads, 0, s>>>(dc, n);
    else if (job.mode == MODE_STORE)
        kvs_ldg_kernel<V, MODE_STORE><<<grid, kLdgThreads, 0, s>>>(dc, n);
    else
        kvs_ldg_kernel<V, MODE_COMPARE><<<grid, kLdgThreads, 0, s>>>(dc, n);
    return cudaGetLastError();
}

}  // namespace

int link_ctas_per_sm() {
    static int n = 0;
    if (n == 0) {
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kvs_link_kernel<MODE_RETRIEVE>, kLdgThreads, 0);
        if (n <= 0) n = 1;
    }
    return n;
}

cudaError_t launch_link_prefetch(const Job& job, int grid, cudaStream_t s) {
    if (job.num_pieces == 0) return cudaSuccess;
    grid = clamp_grid(grid, link_ctas_per_sm(), job.num_pieces);
    // about 4 MiB of prefetches in flight over the whole grid
    const uint32_t ahead = (uint32_t)std::min(64, std::max(2, (int)((4u << 20) / kPieceBytes) / grid));
    kvs_link_pf_kernel<<<grid, kLdgThreads, 0, s>>>(make_decoder(job), (uint32_t)job.num_pieces, ahead);
    return cudaGetLastError();
}

// Raises the kernel's dynamic shared-memory limit on the current device (once
// per device) and returns its resident CTAs per SM.
int g_staged_per_sm[kMaxDevices];

int link_staged_ctas_per_sm() {
    const int dev = current_device();
    if (g_staged_per_sm[dev] == 0) {
        cudaFuncSetAttribute(kvs_link_staged_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kStagedSmemBytes);
        cudaFuncSetAttribute(kvs_link_staged_kernel, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
        int n = 0;
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kvs_link_staged_kernel, kLdgThreads, kStagedSmemBytes);
        g_staged_per_sm[dev] = n > 0 ? n : 1;
    }
    return g_staged_per_sm[dev];
}

cudaError_t launch_link_staged(const Job& job, int grid, cudaStream_t s) {
    if (job.num_pieces == 0) return cudaSuccess;
    if (job.mode != MODE_RETRIEVE) return cudaErrorInvalidValue;
    grid = clamp_grid(grid, link_staged_ctas_per_sm(), job.num_pieces);
    kvs_link_staged_kernel<<<grid, kLdgThreads, kStagedSmemBytes, s>>>(make_decoder(job), (uint32_t)job.num_pieces);
    return cudaGetLastError();
}

cudaError_t launch_link(const Job& job, int grid, cudaStream_t s) {
    if (job.num_pieces == 0) return cudaSuccess;
    grid = clamp_grid(grid, link_ctas_per_sm(), job.num_pieces);
    const Decoder dc = make_decoder(job);
    const uint32_t n = (uint32_t)job.num_pieces;
    if (job.mode == MODE_RETRIEVE)
        kvs_link_kernel<MODE_RETRIEVE><<<grid, kLdgThreads, 0, s>>>(dc, n);
    else
        kvs_link_kernel<MODE_STORE><<<grid, kLdgThreads, 0, s>>>(dc, n);
    return cudaGetLastError();
}

int ldg_ctas_per_sm() {
    static int n = 0;
    if (n == 0) {
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kvs_ldg_kernel<16, MODE_RETRIEVE>, kLdgThreads, 0);
        if (n <= 0) n = 1;
        if (n > 4) n = 4;
    }
    return n;
}

int tma_ctas_per_sm() { return 1; }

cudaError_t launch_ldg(const Job& job, int vec_bytes, int grid, cudaStream_t s) {
    if (job.num_pieces == 0) return cudaSuccess;
    switch (vec_bytes) {
        case 16: return launch_ldg_v<16>(job, grid, s);
        case 8:  return launch_ldg_v<8>(job, grid, s);
        case 4:  return launch_ldg_v<4>(job, grid, s);
        case 2:  return launch_ldg_v<2>(job, grid, s);
        default: return launch_ldg_v<1>(job, grid, s);
    }
}

cudaError_t launch_tma(const Job& job, int grid, cudaStream_t s) {
    if (job.num_pieces == 0) return cudaSuccess;
    const int dev = current_device();
    if (grid <= 0 && job.mode != MODE_COMPARE) {
        // The carveout preference asks for the largest shared-memory split, so
        // that six 33 KiB CTAs (stage + reserved) fit on an SM.
        if (!g_tma_piece_cfg[dev]) {
            for (auto fn : {kvs_tma_piece_kernel<MODE_RETRIEVE>, kvs_tma_piece_kernel<MODE_STORE>}) {
                cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributePreferredSharedMemoryCarveout,
                                                     (int)cudaSharedmemCarveoutMaxShared);
                if (e != cudaSuccess) return e;
            }
            g_tma_piece_cfg[dev] = true;
        }
        const Decoder dc = make_decoder(job);
        const uint32_t n = (uint32_t)job.num_pieces;
        if (job.mode == MODE_RETRIEVE)
            kvs_tma_piece_kernel<MODE_RETRIEVE><<<n, 32, job.piece_bytes, s>>>(dc);
        else
            kvs_tma_piece_kernel<MODE_STORE><<<n, 32, job.piece_bytes, s>>>(dc);
        return cudaGetLastError();
    }
    const size_t smem = (size_t)kTmaStages * job.piece_bytes;
    if (g_tma_smem[dev] < smem) {             // the attribute is set per device
        cudaError_t e = cudaFuncSetAttribute(kvs_tma_kernel<kTmaStages>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        g_tma_smem[dev] = smem;
    }
    grid = clamp_grid(grid, tma_ctas_per_sm(), job.num_pieces);
    kvs_tma_kernel<kTmaStages><<<grid, 32, smem, s>>>(make_decoder(job), (uint32_t)job.num_pieces);
    return cudaGetLastError();
}

cudaError_t launch_stall(int32_t* err, uint64_t limit_ns, cudaStream_t s) {
    kvs_stall_kernel<<<1, 32, 0, s>>>(err, limit_ns);
    return cudaGetLastError();
}

cudaError_t launch_link_signal(const Job& job, const Signal& sig, int grid, cudaStream_t s) {
    grid = clamp_grid(grid, link_ctas_per_sm(), std::max<uint64_t>(job.num_pieces, 1));
    const Decoder dc = make_decoder(job);
    const FastDiv entries = make_fastdiv(job.num_entries);
    const uint32_t n = (uint32_t)job.num_pieces;
    if (job.mode == MODE_RETRIEVE)
        kvs_link_signal_kernel<MODE_RETRIEVE><<<grid, kLdgThreads, 0, s>>>(dc, entries, sig, n);
    else
        kvs_link_signal_kernel<MODE_STORE><<<grid, kLdgThreads, 0, s>>>(dc, entries, sig, n);
    return cudaGetLastError();
}

cudaError_t launch_flat_copy(void* dst, const void* src, uint64_t bytes, int grid, cudaStream_t s) {
    const uint64_t pieces = (bytes + kPieceBytes - 1) / kPieceBytes;
    if (pieces == 0) return cudaSuccess;
    grid = grid > 0 ? clamp_grid(grid, ldg_ctas_per_sm(), pieces) : (int)std::min<uint64_t>(pieces, 1u << 30);
    kvs_flat_copy_kernel<<<grid, kLdgThreads, 0, s>>>((uint64_t)dst, (uint64_t)src, bytes);
    return cudaGetLastError();
}

}  // namespace kvs

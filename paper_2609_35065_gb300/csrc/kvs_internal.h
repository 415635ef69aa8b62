// kvs_internal.h -- descriptors shared by the planner (kvs_api.cpp) and the
// copy kernels (kvs_kernels.cu).  Not part of the public ABI.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace kvs {

// One (request, chunk) pair of a call.  The chunk buffer is [L][2][n_tok][H][D].
// Entry k's blocks are Job::blocks[k * blocks_per_chunk ...], so a kernel can
// load a block id without waiting for the entry itself.
struct Entry {
    uint64_t chunk;     // device-visible address of the chunk buffer
    int32_t  n_tok;     // tokens held by the chunk (its token stride)
    int32_t  pad;
};
static_assert(sizeof(Entry) == 16, "Entry is uploaded as raw bytes");

enum Mode : int32_t {
    MODE_RETRIEVE = 0,  // chunk -> plane
    MODE_STORE    = 1,  // plane -> chunk
    MODE_COMPARE  = 2,  // flag KVS_ERR_ALIAS where chunk bytes differ from plane bytes
};

// Work of one launch.  A "run" is the contiguous copy of one (entry, plane p,
// block i of the chunk): up to B token rows, B*R bytes, contiguous on both
// sides.  Runs are cut into "pieces" of at most piece_bytes for the kernels.
// Run index g = (entry * num_planes + p) * blocks_per_chunk + i.
struct Job {
    const Entry*    entries;
    const int32_t*  blocks;          // physical block of (entry k, i) at k * blocks_per_chunk + i;
                                     // < 0 means "skip"
    const uint64_t* planes;          // 2L plane base addresses
    int32_t*        err;             // device error word (first error wins)
    uint64_t        row_bytes;       // R = H * D * e
    uint64_t        num_pieces;      // num_entries * num_planes * blocks_per_chunk * pieces_per_run
    int64_t         num_blocks;      // NB, for the device-side bounds check
    uint32_t        num_entries;
    uint32_t        entry_base;      // index of entries[0] among all entries of the call
    uint32_t        num_planes;      // planes copied by this launch ...
    uint32_t        plane_begin;     // ... starting at this plane (2 * first layer)
    uint32_t        blocks_per_chunk;
    uint32_t        pieces_per_run;
    uint32_t        piece_bytes;     // multiple of 16
    uint32_t        block_size;      // B
    int32_t         mode;            // Mode
};

// Piece size used by both kernel flavours.
constexpr uint32_t kPieceBytes = 32768;

// Launchers (kvs_kernels.cu).  `grid` <= 0 means "fill the GPU".
cudaError_t launch_ldg(const Job& job, int vec_bytes, int grid, cudaStream_t s);
cudaError_t launch_tma(const Job& job, int grid, cudaStream_t s);
// Double-buffered 16-byte flavour for host-resident chunks (retrieve or store).
cudaError_t launch_link(const Job& job, int grid, cudaStream_t s);
// Retrieval of host chunks holding more bytes in flight per SM (one piece in
// registers and three in shared memory per 256 threads, two CTAs per SM), for
// GPUs that run other kernels meanwhile (KVS_F_FEW_SMS).
cudaError_t launch_link_staged(const Job& job, int grid, cudaStream_t s);
// The same for retrieval, with each CTA's upcoming pieces prefetched into L2.
cudaError_t launch_link_prefetch(const Job& job, int grid, cudaStream_t s);
// Contiguous copy of `bytes` (multiple of 16, 16-byte aligned) for bandwidth probes.
cudaError_t launch_flat_copy(void* dst, const void* src, uint64_t bytes, int grid, cudaStream_t s);
// Layer-wise copy of host chunks in one launch: pieces go in plane-major
// order, and the CTA that completes the last piece of layer group g writes
// flags[g] = gen (after making the group's stores visible); the last CTA to
// finish writes every flag, so all are written whatever the counts.  Consumers
// wait on the flags with stream memory operations, not with kernels.
struct Signal {
    uint32_t* counters;        // per group: pieces done (zeroed before the launch)
    uint32_t* flags;           // per group: generation of the last completed copy
    uint32_t* ctas_done;       // CTAs finished (zeroed before the launch)
    uint32_t  gen;
    uint32_t  groups;
    uint32_t  planes_per_group;
};
cudaError_t launch_link_signal(const Job& job, const Signal& sig, int grid, cudaStream_t s);

// fp8 chunks: [scales: 2L*H binary32, zero-padded to scale_bytes][codes [L][2][n][H][D] E4M3].
// The Job's planes are BF16 ([NB][B][H][D], row_bytes = 2*H*D); entries point at chunk
// buffers (scale block first); blocks_per_chunk / block_size / planes as for BF16 copies.
struct Fp8Job {
    Job      job;                // mode MODE_RETRIEVE (dequantise) or MODE_STORE (quantise)
    uint32_t heads;              // H
    uint32_t head_dim;           // D, a multiple of 16
    uint32_t scale_bytes;        // bytes of the scale block, a multiple of 256
    uint32_t block_magic;        // floor(2^32 / B) + 1: floor(i / B) = umulhi(i, magic) for i, B < 2^16
    // Piece decode by round-up reciprocals: floor(n / d) = (n * m) >> p for n < 2^31
    // (p = 31 + ceil(log2 d), m = ceil(2^p / d)), d = pieces per run, runs per
    // entry (num_planes * blocks_per_chunk) and blocks per chunk.
    uint32_t ppr_m, ppr_p, pe_m, pe_p, bpc_m, bpc_p;
    uint32_t rows_whole;         // 1 when every piece starts at a token row (H*D/16 divides 1024)
};
constexpr uint32_t kFp8MaxHeads = 128;
// Retrieval: a persistent grid of `grid` CTAs (<= 0: fill the GPU) over pieces of at
// most 16 KiB of codes, double-buffered; grid == kFp8PerPiece: one CTA per piece
// (HBM sources).  The number of pieces is in job.num_pieces.
constexpr int kFp8PerPiece = -1;
cudaError_t launch_fp8_retrieve(const Fp8Job& fj, int grid, cudaStream_t s);
// Retrieval of host chunks with more codes in flight per SM (two pieces in
// registers and five in shared memory per 256 threads, two CTAs per SM), for
// GPUs that run other kernels meanwhile (KVS_F_FEW_SMS); `grid` <= 0: 2 per SM.
cudaError_t launch_fp8_retrieve_staged(const Fp8Job& fj, int grid, cudaStream_t s);
// Store-back: one CTA per (entry, plane, head) in a single pass when a head's
// chunk_tokens x head_dim elements fit the CTA's registers, else one CTA per
// (entry, plane) in two passes; a grid-stride loop over them with `grid` > 0.
// `staged` (HBM destinations): the single pass runs as a persistent CTA per SM
// (at most `grid` > 0) that stages heads in shared memory with bulk copies.
cudaError_t launch_fp8_store(const Fp8Job& fj, int grid, cudaStream_t s, uint32_t chunk_tokens, bool staged);
// Codes per retrieval piece (16 KiB).
constexpr uint32_t kFp8PieceCodes = 16384;

// One CTA waits (bounded by limit_ns) on an mbarrier phase that nothing
// completes, then records KVS_ERR_TIMEOUT: exercises the bounded-wait path.
cudaError_t launch_stall(int32_t* err, uint64_t limit_ns, cudaStream_t s);
// Sets the calling thread's message returned by kvs_last_error() (kvs_api.cpp).
void set_last_error(const char* msg);
// CTA cap kvs_retrieve / kvs_store give host-link kernels on the current device
// (the measured one after kvs_query_bw, else the built-in default); allocates
// nothing (kvs_api.cpp).
int hostlink_grid(bool retrieve);
// Forgets the per-device address of the allocation-free entry point's static
// scratch (kvs_noalloc.cu); kvs_shutdown calls it.
void noalloc_forget_devices();
// CTAs per SM the flavour runs with (occupancy); used to size persistent grids.
int ldg_ctas_per_sm();
int link_ctas_per_sm();
int tma_ctas_per_sm();

}  // namespace kvs

/*
 * kvs.h -- C ABI for prefix-KV retrieval into a paged GPU KV cache (GB300, sm_103a).
 *
 * TempoKV separates SSD-to-fast-tier staging from fast-tier-to-GPU retrieval
 * (Sec. 2.2) and reuses the runtime's GPU-transfer path once matched KV is
 * stage-ready (Sec. 3, Sec. 4).  This library is that transfer path:
 *
 *   kvs_retrieve  copies the matched prefix of each request from its chunk
 *                 buffers in the fast tier into the runtime's paged KV cache;
 *   kvs_store     copies newly computed KV from the paged cache back into
 *                 chunk buffers (KV is retained in complete 256-token chunks,
 *                 Sec. 5.1, Workload);
 *   kvs_query_bw  measures the host link and HBM on this GPU and picks, per
 *                 direction, how host-resident chunks are moved.
 *
 * The arguments follow the paper's statement of a retrieval: the matched
 * prefix tokens of each request, where its KV objects sit in the fast tier
 * (their ordered manifest, Sec. 3, and their access order, known before
 * retrieval begins, Sec. 2.1), the destination block table, and the KV
 * geometry (layers, KV heads, head dim; BF16 in the paper, Sec. 5 setup).
 *
 * Layouts (all row-major, contiguous):
 *   chunk  of n tokens:  [L][2][n][H][D]   K before V, one buffer per chunk
 *   paged plane p=2l+kv: [num_blocks][B][H][D]   one device buffer per
 *                        (layer, K/V); the caller passes 2L plane pointers,
 *                        so split or fused K/V caches both fit.
 *   request token t of a request lives in slot  block_table[t / B] * B + t % B.
 *
 * Ownership: the caller owns every buffer it passes (chunks, planes, tables).
 * The library owns only small internal buffers (descriptor upload slots, an
 * error word, a staging ring for the copy-engine variant, probe buffers),
 * kept per device until kvs_shutdown() or process exit.
 *
 * Asynchrony: kvs_retrieve / kvs_store enqueue work on the caller's CUDA
 * stream and return; every host array they are given is consumed before they
 * return (it may be freed or reused at once).  Chunk buffers and planes must
 * stay valid and unmodified until the stream reaches the enqueued work.
 * The return code reports validation and enqueue status; device-side faults
 * are reported by kvs_check_errors() or by a KVS_F_VALIDATE call.
 *
 * Threading: calls may come from several host threads; the library
 * serialises its own planning.  The work runs on the device that is current
 * on the calling thread.
 */
#ifndef KVS_H
#define KVS_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ------------------------------------------------------ */
#define KVS_OK               0
#define KVS_ERR_INVALID_ARG (-1)  /* null pointer, bad geometry, token counts that do not
                                     tile the matched range, misplaced partial chunk      */
#define KVS_ERR_BOUNDS      (-2)  /* block table shorter than the range, or a block id
                                     outside [0, num_blocks)                                */
#define KVS_ERR_ALIAS       (-3)  /* one physical block named twice by one request, or
                                     (KVS_F_VALIDATE) shared blocks with differing bytes,
                                     or written memory overlapping written or read memory */
#define KVS_ERR_CUDA        (-4)  /* a CUDA runtime call failed; see kvs_last_error()     */
#define KVS_ERR_TIMEOUT     (-5)  /* a bounded device-side wait expired                    */
#define KVS_ERR_NOMEM       (-6)  /* an internal buffer could not be allocated            */
#define KVS_ERR_UNSUPPORTED (-7)  /* a forced variant cannot serve these arguments        */

/* ---- residency of a chunk buffer (the fast-tier stand-in) --------------- */
#define KVS_SRC_HOST_PINNED 1     /* page-locked host memory mapped into the GPU's address
                                     space (cudaHostAlloc / cudaHostRegister), reached over
                                     the host link                                          */
#define KVS_SRC_DEVICE      2     /* device memory of the current GPU (an HBM staging copy) */

/* ---- flags (bitwise OR) --------------------------------------------------- */
#define KVS_F_VALIDATE       (1u << 0) /* synchronise the stream after the copy and return
                                          the device error word; also verify that blocks
                                          shared by several requests receive equal bytes,
                                          that chunk pointers are what their residency
                                          says, and (on the host, before any copy) that
                                          the memory the call writes overlaps neither
                                          itself nor the memory it reads              */
#define KVS_F_FORCE_HOSTLINK (1u << 1) /* host chunks: SMs load/store host memory directly  */
#define KVS_F_FORCE_HBMCOPY  (1u << 2) /* host chunks: copy engine to/from an HBM staging
                                          ring, SMs scatter/gather in HBM                    */
#define KVS_F_FORCE_LDG      (1u << 3) /* kernel flavour: vector loads/stores by all threads */
#define KVS_F_FORCE_TMA      (1u << 4) /* kernel flavour: bulk async copies (TMA) staged
                                          through shared memory; 16-byte aligned data only  */
#define KVS_F_NO_DEDUP       (1u << 5) /* write shared physical blocks once per request      */
#define KVS_F_LAYER_LAUNCHES (1u << 6) /* layer-wise calls: one launch per layer group
                                          (the default; accepted for explicitness)         */
#define KVS_F_LAYER_SIGNAL   (1u << 7) /* layer-wise calls: one resident launch that
                                          signals each group (see kvs_retrieve_layers)     */
#define KVS_F_FORCE_DMA      (1u << 8) /* host chunks: the copy engine moves each (chunk,
                                          block) straight between the chunk and all 2L
                                          planes with one 2D copy; no SM runs a kernel for
                                          them.  Needs equally spaced planes (plane p at
                                          plane 0 + p * pitch, as in one [2L][...] cache
                                          allocation); KVS_ERR_UNSUPPORTED otherwise      */
#define KVS_F_PREFETCH_L2    (1u << 9) /* retrieval of host chunks on the host-link kernel:
                                          each CTA keeps its upcoming pieces in flight as
                                          bulk L2 prefetches, so the bytes in flight wait
                                          in L2 rather than in registers and a small
                                          KVS_F_MAX_CTAS grid can hold the link rate      */
#define KVS_F_FEW_SMS        (1u << 10) /* retrieval of host chunks on a GPU that runs
                                          other kernels meanwhile (a model's compute):
                                          the host-link variant with a kernel that holds
                                          more bytes in flight per SM (BF16: one 32 KiB
                                          piece in registers and three in shared memory
                                          per 256 threads; fp8: two 16 KiB pieces of
                                          codes in registers and five in shared memory;
                                          two CTAs per SM), on its own measured cap
                                          (kvs_bw_report.few_sm_ctas), so the link rate
                                          needs fewer SMs.  BF16: 16-byte aligned
                                          chunks, planes and rows (else the plain
                                          host-link kernels run); not with
                                          KVS_F_FORCE_HBMCOPY / _DMA, KVS_F_PREFETCH_L2
                                          or KVS_F_LAYER_SIGNAL; store calls ignore it  */
#define KVS_F_MAX_CTAS(n)    ((((uint32_t)(n)) & 0xFFFFu) << 16) /* cap on CTAs, 0 = auto */
#define KVS_F_GET_MAX_CTAS(f) (((f) >> 16) & 0xFFFFu)

/* Variant identifiers reported by kvs_query_bw. */
#define KVS_VARIANT_HOSTLINK 1
#define KVS_VARIANT_HBMCOPY  2
#define KVS_VARIANT_DMA      3
#define KVS_KERNEL_LDG       1
#define KVS_KERNEL_TMA       2

/* KV geometry.  elem_bytes is 2 for BF16 KV (1, 2, 4 and 8 are accepted; elements
 * are copied as opaque bytes).  chunk_tokens must be a multiple of block_size. */
typedef struct kvs_geometry {
    int32_t num_layers;     /* L */
    int32_t num_kv_heads;   /* H */
    int32_t head_dim;       /* D */
    int32_t elem_bytes;     /* e */
    int32_t block_size;     /* B: tokens per paged block (vLLM block)  */
    int32_t chunk_tokens;   /* C: tokens per full chunk (LMCache: 256) */
} kvs_geometry;

/* One chunk buffer, [L][2][num_tokens][H][D].  Every chunk of a request holds
 * chunk_tokens tokens except the last, which may hold fewer (1..C). */
typedef struct kvs_chunk {
    void*   base;           /* host (KVS_SRC_HOST_PINNED) or device (KVS_SRC_DEVICE) address */
    int32_t num_tokens;
    int32_t residency;      /* KVS_SRC_* */
} kvs_chunk;

/* One request's matched range [first_token, first_token + num_tokens) and the
 * chunks that hold it, in token order.  first_token must be a multiple of
 * chunk_tokens (a prefix starts at 0).  block_table is a HOST array mapping
 * logical block k of the request to a physical block id in [0, num_blocks);
 * it must cover ceil((first_token + num_tokens) / B) blocks. */
typedef struct kvs_request {
    int64_t          first_token;
    int64_t          num_tokens;
    const kvs_chunk* chunks;
    int32_t          num_chunks;
    int32_t          block_table_len;
    const int32_t*   block_table;
} kvs_request;

/* The paged KV cache: a HOST array of 2L device pointers ordered
 * K0, V0, K1, V1, ..., each to a [num_blocks][B][H][D] plane. */
typedef struct kvs_paged_cache {
    void* const* kv_planes;
    int64_t      num_blocks;
} kvs_paged_cache;

/*
 * Retrieval (fast tier -> GPU): for every request r, chunk j, layer l, K/V kv,
 * token i of the chunk, head h and dim d,
 *     plane[2l+kv][slot(s_j + i)][h][d] = chunk_j[l][kv][i][h][d],
 * with s_j the first request token of chunk j.  Nothing else is written.
 * When a call holds both device- and host-resident chunks, the two classes
 * are copied concurrently (the device part on a library stream that joins
 * the caller's stream before the call's work is complete).
 * A physical block named by several requests (a shared prefix) must carry the
 * same KV in each; it is written once, from the request that covers the most
 * of its tokens (the lowest index among equals), unless KVS_F_NO_DEDUP.
 * Returns KVS_OK or a KVS_ERR_* code (nothing is enqueued on error).
 */
int kvs_retrieve(const kvs_geometry* geom, const kvs_paged_cache* cache,
                 const kvs_request* requests, int32_t num_requests,
                 void* cuda_stream, uint32_t flags);

/*
 * Store-back (GPU -> chunks): the same correspondence read the other way,
 *     chunk_j[l][kv][i][h][d] = plane[2l+kv][slot(s_j + i)][h][d];
 * the chunks are the destinations.  The cache is only read.  Destination
 * chunks must not overlap each other or any plane.
 */
int kvs_store(const kvs_geometry* geom, const kvs_paged_cache* cache,
              const kvs_request* requests, int32_t num_requests,
              void* cuda_stream, uint32_t flags);

/*
 * Layer-wise retrieval.  The paper's time-to-use ends when retrieval begins,
 * not when the model consumes the KV (Sec. 3.1): the model can start on the
 * first layers while later layers are still in flight.  This call does the
 * same copy as kvs_retrieve, planned and uploaded once, as ceil(L /
 * layers_per_step) launch groups in layer order on cuda_stream; after group k
 * (layers [k * layers_per_step, (k + 1) * layers_per_step)) is enqueued,
 * layer_events[k] is recorded on cuda_stream, so another stream can
 * cudaStreamWaitEvent on it and use those layers while later groups copy.
 * layer_events may be NULL, and so may any of its entries; the events are the
 * caller's (cudaEvent_t cast to void*).  Host-resident chunks always take the
 * host-link kernel here (KVS_F_FORCE_HBMCOPY returns KVS_ERR_UNSUPPORTED).
 * By default each group is its own launch followed by its event on
 * cuda_stream: between groups the SMs go back to whatever else runs (the
 * model's compute), so the copy keeps just ahead of its consumer without a
 * tuned CTA cap.  With KVS_F_LAYER_SIGNAL, when every chunk is host-resident
 * and 16-byte aligned and events are given, the copy is instead ONE launch
 * that stays resident and publishes each group's completion in device flags;
 * a library stream waits on those flags (driver stream memory operations) and
 * records layer_events[k] as group k lands (otherwise the call falls back to
 * per-group launches).  A resident launch holds its SMs for the whole copy,
 * so it suits a small KVS_F_MAX_CTAS cap.  KVS_F_LAYER_LAUNCHES together with
 * KVS_F_LAYER_SIGNAL is KVS_ERR_INVALID_ARG.  Either way cuda_stream reaches
 * the end of the whole copy after it.
 */
int kvs_retrieve_layers(const kvs_geometry* geom, const kvs_paged_cache* cache,
                        const kvs_request* requests, int32_t num_requests,
                        int32_t layers_per_step, void* const* layer_events,
                        void* cuda_stream, uint32_t flags);

/* Layer-wise store-back: kvs_store in layer groups, so that newly computed KV
 * leaves the GPU while later layers are still being computed.  Before group k
 * (layers [k * layers_per_step, (k + 1) * layers_per_step)) is copied,
 * cuda_stream waits on ready_events[k] (cudaStreamWaitEvent: the caller
 * records it on its compute stream once those layers' KV is in the cache,
 * before this call); after group k, layer_events[k] is recorded.  Either array
 * may be NULL, and so may any of its entries (no wait / no record).  Groups are
 * always separate launches here.  KVS_F_FORCE_HBMCOPY returns
 * KVS_ERR_UNSUPPORTED; KVS_F_LAYER_SIGNAL together with ready_events is
 * KVS_ERR_INVALID_ARG (a resident launch cannot wait between groups). */
int kvs_store_layers(const kvs_geometry* geom, const kvs_paged_cache* cache,
                     const kvs_request* requests, int32_t num_requests,
                     int32_t layers_per_step, void* const* ready_events,
                     void* const* layer_events, void* cuda_stream, uint32_t flags);

/*
 * fp8 chunks.  The paper keeps KV in BF16 (Sec. 5 setup) and retains it in
 * 256-token chunks (Sec. 5.1, Workload); these two calls add a compressed
 * chunk format for the fast tier, which halves the bytes a retrieval moves
 * over the host link.  A chunk of n tokens is one buffer:
 *
 *   [scales] 2L*H IEEE binary32 values, the scale of (layer l, K/V kv, head h)
 *            at index (2l + kv)*H + h, zero-padded to KVS_FP8_SCALE_BYTES(L, H)
 *            bytes (a multiple of 256);
 *   [codes]  [L][2][n][H][D] bytes in the E4M3 format of the OCP 8-bit
 *            Floating Point Specification (OFP8), revision 1.0.
 *
 * The paged planes stay BF16 (geom->elem_bytes must be 2).  head_dim must be
 * a multiple of 16, H at most 128, chunks and planes 16-byte aligned
 * (KVS_ERR_UNSUPPORTED otherwise).  Arguments, layouts of the planes and
 * block tables, residencies, asynchrony and errors are as for kvs_retrieve /
 * kvs_store; the accepted flags are KVS_F_VALIDATE, KVS_F_MAX_CTAS,
 * KVS_F_FEW_SMS (retrieval: host chunks on a kernel holding more codes in
 * flight per SM, on kvs_bw_report.few_sm_ctas; stores ignore it) and
 * KVS_F_FORCE_HOSTLINK / KVS_F_FORCE_LDG, which name what always runs: host
 * chunks are read or written over the host link by SM loads and stores.
 *
 * kvs_retrieve_fp8: plane[2l+kv][slot(s_j+i)][h][d] =
 *     bf16(e4m3(code[l][kv][i][h][d]) * scale[l][kv][h]): the product is one
 *     binary32 multiply rounded to nearest even, then rounded to BF16 (nearest
 *     even); a NaN product (a NaN code, or a NaN scale) gives 0x7FFF.  A
 *     physical block named by two requests of one call is refused
 *     (KVS_ERR_ALIAS): quantised copies of one block differ with the scales of
 *     the chunks that hold them.
 * kvs_store_fp8: for every chunk, layer, K/V and head, amax = the largest |x|
 *     over the finite BF16 elements of the chunk's tokens (0 if none), scale =
 *     amax / 448 and inv = 448 / amax (binary32 divisions, nearest even; both
 *     1 when amax is 0), code = E4M3 of x * inv (one binary32 multiply,
 *     nearest even), rounded to nearest even and saturated to +-448 (OFP8
 *     saturation mode; infinities too); NaN elements give the code 0x7F.  The scales and codes of every destination
 *     chunk are written; the cache is only read.
 */
#define KVS_FP8_SCALE_BYTES(L, H) ((((int64_t)2 * (L) * (H) * 4) + 255) / 256 * 256)
int kvs_retrieve_fp8(const kvs_geometry* geom, const kvs_paged_cache* cache,
                     const kvs_request* requests, int32_t num_requests,
                     void* cuda_stream, uint32_t flags);
int kvs_store_fp8(const kvs_geometry* geom, const kvs_paged_cache* cache,
                  const kvs_request* requests, int32_t num_requests,
                  void* cuda_stream, uint32_t flags);

/* Layer-wise forms of the two fp8 calls, with the semantics of kvs_retrieve_layers
 * / kvs_store_layers (the model can start on layer group k once layer_events[k]
 * fires; group k of a store waits on ready_events[k]): one launch per layer
 * group and source class, on cuda_stream.  Layer by layer, host-chunk stores
 * run on the host-link store cap (see kvs_bw_report.store_ctas; KVS_F_MAX_CTAS
 * overrides it), so that each group's launch leaves most SMs to the compute
 * producing the next layers.  KVS_F_LAYER_SIGNAL is not accepted. */
int kvs_retrieve_fp8_layers(const kvs_geometry* geom, const kvs_paged_cache* cache,
                            const kvs_request* requests, int32_t num_requests,
                            int32_t layers_per_step, void* const* layer_events,
                            void* cuda_stream, uint32_t flags);
int kvs_store_fp8_layers(const kvs_geometry* geom, const kvs_paged_cache* cache,
                         const kvs_request* requests, int32_t num_requests,
                         int32_t layers_per_step, void* const* ready_events,
                         void* const* layer_events, void* cuda_stream, uint32_t flags);

/* Bandwidths measured by kvs_query_bw, in GB/s (1e9 bytes per second). */
typedef struct kvs_bw_report {
    double  hbm_copy_gbs;          /* device->device copy kernel, read + write bytes      */
    double  h2d_copy_engine_gbs;   /* cudaMemcpyAsync pinned host -> device                */
    double  d2h_copy_engine_gbs;   /* cudaMemcpyAsync device -> pinned host                */
    double  zero_copy_read_gbs;    /* copy kernel reading pinned host, writing HBM         */
    double  zero_copy_write_gbs;   /* copy kernel reading HBM, writing pinned host         */
    double  retrieve_gbs[2];       /* host-chunk retrieval probe: [HOSTLINK, HBMCOPY]      */
    double  store_gbs[2];          /* host-chunk store probe:     [HOSTLINK, HBMCOPY]      */
    double  device_kernel_gbs[2];  /* device-chunk retrieval probe, payload bytes: [LDG, TMA] */
    int32_t chosen_retrieve_host;  /* KVS_VARIANT_* used for host chunks by kvs_retrieve   */
    int32_t chosen_store_host;     /* KVS_VARIANT_* used for host chunks by kvs_store      */
    int32_t chosen_kernel_device;  /* KVS_KERNEL_* used for device-resident chunks         */
    int32_t num_sms;
    int32_t hostlink_ctas;         /* CTAs given to host-link retrieval kernels (0 = all):
                                      4 x the smallest probed grid within 1% of the best
                                      rate, so that kernels on other streams keep most SMs
                                      (before any kvs_query_bw: one per 3 SMs)            */
    int32_t store_ctas;            /* the same for host-link store kernels                 */
    int64_t probe_bytes;           /* bytes moved per probe                                */
    double  retrieve_dma_gbs;      /* host-chunk retrieval probe, DMA variant              */
    double  store_dma_gbs;         /* host-chunk store probe, DMA variant                  */
    int32_t few_sm_ctas;           /* CTA cap of KVS_F_FEW_SMS retrievals: 1.25 x the
                                      smallest probed grid within 3% of the kernel's best
                                      rate (before any kvs_query_bw: one per 8 SMs, at
                                      least 8)                                             */
    int32_t reserved;
    double  few_sm_gbs;            /* best KVS_F_FEW_SMS retrieval probe rate              */
} kvs_bw_report;

/*
 * Measures the bandwidths above on the current device with probes of
 * probe_bytes bytes (0 = 1 GiB), synchronously, using cuda_stream, and makes
 * the measured fastest variants (and the host-link CTA caps) the defaults of
 * later kvs_retrieve / kvs_store calls on this device.  Allocates (and frees before returning) probe
 * buffers: 2 * probe_bytes of device memory and probe_bytes of pinned host
 * memory.  `out` may be NULL.
 */
int kvs_query_bw(kvs_bw_report* out, void* cuda_stream, int64_t probe_bytes);

/* Reads the defaults currently in force on this device (after kvs_query_bw,
 * or the built-in ones) into `out`; bandwidth fields are 0 if never measured. */
int kvs_get_choice(kvs_bw_report* out);

/*
 * Variant choice measured on the caller's own call.  kvs_query_bw probes a
 * fixed 1 GiB pattern; how fast the copy engine moves host memory can depend
 * on the buffer (its size and how it was allocated) and on what else the GPU
 * runs, which only the real call shows.  kvs_tune performs the given call
 * (direction KVS_DIR_RETRIEVE or KVS_DIR_STORE) `reps` + 1 times with each
 * variant that can serve its host-resident chunks -- HOSTLINK, HBMCOPY and,
 * with equally spaced planes, DMA -- times each on cuda_stream (best of
 * `reps`, after one untimed run), and makes the fastest the default of later
 * kvs_retrieve / kvs_store calls in that direction on this device.  Every
 * candidate produces the same result, so the call's copy is done when
 * kvs_tune returns (the stream is synchronised).  KVS_F_MAX_CTAS(n) caps the
 * HOSTLINK candidate's grid (and becomes the host-link cap of that direction
 * if it wins); KVS_F_VALIDATE is honoured on the untimed runs; FORCE, layer,
 * KVS_F_FEW_SMS and KVS_F_PREFETCH_L2 flags are KVS_ERR_INVALID_ARG.  When the call holds device-resident chunks, those
 * chunks alone are then timed with the LDG and the TMA kernel (TMA only for
 * 16-byte aligned data), each chunk as a request of its own, and the faster
 * kernel becomes the default for device chunks.  A call with no chunk of a
 * class leaves that class's default unchanged.  `out` (may be NULL) receives
 * the rates in GB/s of each class's bytes (0 for a candidate that cannot
 * serve the call) and the choices.
 */
#define KVS_DIR_RETRIEVE 0
#define KVS_DIR_STORE    1
typedef struct kvs_tune_report {
    double  gbs[3];            /* [HOSTLINK, HBMCOPY, DMA]                              */
    int64_t host_bytes;        /* bytes of host-resident chunks in the call             */
    int32_t chosen;            /* KVS_VARIANT_* now the default for this direction      */
    int32_t direction;         /* KVS_DIR_*                                             */
    double  device_gbs[2];     /* device-resident chunks alone: [LDG, TMA] (0: not run)  */
    int64_t device_bytes;      /* bytes of device-resident chunks in the call           */
    int32_t chosen_kernel_device; /* KVS_KERNEL_* now the default for device chunks     */
    int32_t reserved;
} kvs_tune_report;
int kvs_tune(const kvs_geometry* geom, const kvs_paged_cache* cache,
             const kvs_request* requests, int32_t num_requests,
             void* cuda_stream, uint32_t flags, int32_t direction, int32_t reps,
             kvs_tune_report* out);

/*
 * Synchronises cuda_stream, then reads and clears this device's error word.
 * Returns KVS_OK, or the first KVS_ERR_* a kernel recorded since the last check.
 */
int kvs_check_errors(void* cuda_stream);

/*
 * Pipelined form of kvs_check_errors for loops that keep the GPU busy: enqueues
 * on cuda_stream a copy of this device's error word into *host_word followed by
 * a reset of the word, and returns at once without synchronising.  host_word
 * must be page-locked host memory owned by the caller and stay valid until the
 * stream has passed the copy (record an event after this call and wait on it);
 * it then holds 0 or the first KVS_ERR_* recorded by kernels that the stream ran
 * before the copy.  Kernels of other streams of the same device that record an
 * error between the copy and the reset are not reported; use one status stream
 * per device.  Returns KVS_ERR_INVALID_ARG for a NULL host_word, KVS_ERR_CUDA if
 * the copy cannot be enqueued.
 */
int kvs_enqueue_error_read(void* cuda_stream, int32_t* host_word);

/* Message describing the last error on the calling thread ("" if none). */
const char* kvs_last_error(void);

/* Frees every library-owned buffer on every device (device must be idle). */
int kvs_shutdown(void);

/*
 * Self-test of the bounded device-side wait used by the TMA kernel: one CTA
 * waits on a barrier phase that nothing completes, gives up after limit_ns
 * (at most 2e9) and records KVS_ERR_TIMEOUT in the error word; the call then
 * synchronises cuda_stream and returns (and clears) that code.  A correct
 * build returns KVS_ERR_TIMEOUT and leaves the context usable.
 */
int kvs_selftest_wait_timeout(void* cuda_stream, int64_t limit_ns);

/* Number of kernels this library has launched in this process (all devices). */
int64_t kvs_stat_launches(void);

/*
 * Retrieval that allocates nothing.  The paper has no counterpart: this entry
 * point exists for callers that cannot let a library allocate GPU memory --
 * serving runtimes that reserve almost all free HBM for their own KV block
 * pool at start-up and sub-allocate it themselves (a cudaMalloc during serving
 * could fail or break their accounting), and latency-critical paths where
 * cudaMalloc / cudaFree would synchronise the device.
 *
 * Same arguments and result as kvs_retrieve, with these differences:
 *  - no cudaMalloc, cudaFree, cudaHostAlloc or other allocating call is made;
 *    the kernel's scratch (descriptor tables and error word) lives in a static
 *    device array of KVS_NOALLOC_SCRATCH_BYTES compiled into the library,
 *    which every GPU that loads the library holds until the process exits.
 *    A call whose tables do not fit (about 10 KB for 16 requests of 2048
 *    tokens at 32 layers; roughly 16 + 4 * chunk_tokens / block_size bytes
 *    per chunk, twice the block part with KVS_F_VALIDATE) returns
 *    KVS_ERR_UNSUPPORTED with a message saying so;
 *  - the first call on a device looks up the device address of that array
 *    (once per device, with that device current); make that first call
 *    before any stream capture.  kvs_shutdown() forgets the address, so
 *    after a cudaDeviceReset call kvs_shutdown() before the next call;
 *  - every call shares the one array and overwrites it: calls whose work can
 *    overlap on the GPU (different streams, or other host threads) race and
 *    must be ordered by the caller; calls in order on one stream are safe;
 *    the error word is cleared at the start of each call;
 *  - every chunk pointer is checked as kvs_retrieve's KVS_F_VALIDATE checks
 *    it (mapped page-locked host memory, or device memory), on every call;
 *  - host chunks are always read directly over the host link, by the same
 *    double-buffered kernel and CTA cap as kvs_retrieve (KVS_F_MAX_CTAS
 *    overrides the cap); device chunks take the vector-load kernel; the two
 *    classes run one after the other on cuda_stream (KVS_F_FORCE_HBMCOPY,
 *    KVS_F_FORCE_TMA and KVS_F_NO_DEDUP are refused with
 *    KVS_ERR_UNSUPPORTED);
 *  - device-side errors are only reported with KVS_F_VALIDATE.
 */
#define KVS_NOALLOC_SCRATCH_BYTES (1u << 20)
int kvs_retrieve_noalloc(const kvs_geometry* geom, const kvs_paged_cache* cache,
                         const kvs_request* requests, int32_t num_requests,
                         void* cuda_stream, uint32_t flags);

/* ======================================================================
 * Fast tier: the objects retrieval reads from, and their protection.
 *
 * TempoKV's storage-side provider (Sec. 3.2, Sec. 4) keeps reusable KV
 * objects in a fast tier shared by protected staging and ordinary caching:
 *  - a protected-capacity budget below the tier's capacity counts protected
 *    objects and reservations for outstanding staging, each shared object
 *    once, without partitioning memory statically;
 *  - committing a claim protects each object of its manifest, staging the
 *    ones not resident (staging of one object is coalesced across claims);
 *    a claim whose additional footprint does not fit the budget stays Planned;
 *  - a claim is StageReady once every object is resident and protected, and
 *    Transferring from the start of its GPU retrieval; protection ends when
 *    that retrieval completes (Released), unprotected objects stay resident
 *    as evictable cache entries (LRU);
 *  - cancelling a committed claim keeps its protection until its outstanding
 *    staging and GPU accesses end;
 *  - the ordinary (demand) path reserves nothing and, once selected for a
 *    claim, excludes its commitment;
 *  - the protected-capacity cost is C = (integral of P(t) dt) / N (Sec. 5).
 * One object = one KV chunk of object_bytes.  Every call takes the caller's
 * clock `now` (seconds, non-decreasing) so that P(t) is integrated exactly.
 * The tier is a host-side ledger; with arena != 0 it also owns a pinned,
 * device-mapped host arena of capacity_objects slots that kvs_retrieve can
 * read (the fast-tier stand-in).  Not thread-safe: one tier per thread.
 * ====================================================================== */
typedef struct kvs_tier kvs_tier;

typedef struct kvs_tier_config {
    int64_t capacity_objects;   /* slots in the fast tier                         */
    int64_t budget_objects;     /* protected-capacity budget, < capacity_objects  */
    int64_t object_bytes;       /* bytes of one object (one chunk)                */
    int32_t arena;              /* 1: allocate the pinned arena, 0: ledger only   */
    int32_t reserved;
} kvs_tier_config;

/* claim states */
#define KVS_CLAIM_NONE         0
#define KVS_CLAIM_PLANNED      1
#define KVS_CLAIM_STAGING      2
#define KVS_CLAIM_STAGE_READY  3
#define KVS_CLAIM_TRANSFERRING 4
#define KVS_CLAIM_RELEASED     5
#define KVS_CLAIM_CANCELLED    6
#define KVS_CLAIM_ORDINARY     7   /* ordinary retrieval selected (never protected) */

typedef struct kvs_tier_object_info {
    int64_t slot;               /* -1 when the object holds no slot               */
    int32_t pins;               /* claims protecting it                           */
    int32_t staging;            /* 1 while its staging I/O is outstanding         */
    int32_t resident;           /* 1 once its bytes are in the slot               */
    int32_t gpu_refs;           /* retrievals in progress that read it            */
    uint64_t lru;               /* last-use stamp (logical clock)                 */
} kvs_tier_object_info;

typedef struct kvs_tier_stats {
    int64_t resident, staging, protected_objects, free_slots, evictions;
    int64_t staged_reads;       /* staging I/Os issued (coalesced ones count once) */
    int64_t completed;          /* claims Released (N of the cost C)              */
    double  protected_object_seconds;   /* integral of P(t) dt, in objects x s   */
} kvs_tier_stats;

int kvs_tier_create(const kvs_tier_config* cfg, kvs_tier** out);
int kvs_tier_destroy(kvs_tier* tier);

/* Commit `claim` (a new id, or a Planned one being retried) with the ordered
 * manifest keys[0..n).  On KVS_OK the claim is Staging or StageReady and
 * stage_keys[0..*n_stage) receive the objects whose staging I/O the caller
 * must now perform (fill the slot, see kvs_tier_slot, then kvs_tier_staged);
 * stage_keys needs room for n keys.  KVS_ERR_NOMEM: the footprint does not fit
 * the budget (or no slot can be freed); the claim is Planned and nothing else
 * changed.  KVS_ERR_INVALID_ARG: duplicate keys, a claim past Planned, or one
 * on the ordinary path. */
int kvs_tier_commit(kvs_tier* tier, uint64_t claim, const uint64_t* keys, int32_t n,
                    double now, uint64_t* stage_keys, int32_t* n_stage);
/* Staging I/O of `key` completed: the object is resident; claims waiting only
 * on it become StageReady. */
int kvs_tier_staged(kvs_tier* tier, uint64_t key, double now);
/* Retrieval of a StageReady claim begins (Transferring); slots_out[i] gets the
 * slot of keys[i] of its manifest. */
int kvs_tier_begin_retrieval(kvs_tier* tier, uint64_t claim, double now, int64_t* slots_out);
/* The claim's GPU retrieval completed: protection on its behalf ends (Released). */
int kvs_tier_end_retrieval(kvs_tier* tier, uint64_t claim, double now);
/* Cancel a claim: Planned ones at once; committed ones keep their protection
 * until their outstanding staging and GPU accesses end. */
int kvs_tier_cancel(kvs_tier* tier, uint64_t claim, double now);
/* Select the ordinary (demand) path for a claim that is not committed: its
 * objects are held for the retrieval without protection; stage_keys receive
 * the non-resident ones to fetch on demand (into evictable slots).  Finish with
 * kvs_tier_staged for each, then kvs_tier_begin_retrieval / end_retrieval. */
int kvs_tier_ordinary(kvs_tier* tier, uint64_t claim, const uint64_t* keys, int32_t n,
                      double now, uint64_t* stage_keys, int32_t* n_stage);

int kvs_tier_claim_state(const kvs_tier* tier, uint64_t claim);          /* KVS_CLAIM_* */
int kvs_tier_object(const kvs_tier* tier, uint64_t key, kvs_tier_object_info* out); /* KVS_ERR_BOUNDS if unknown */
int kvs_tier_stats_get(kvs_tier* tier, double now, kvs_tier_stats* out);
/* Host address of a slot in the arena (NULL without an arena or out of range);
 * arena slots are pinned and device-mapped: pass them to kvs_retrieve as
 * KVS_SRC_HOST_PINNED chunks. */
void* kvs_tier_slot(const kvs_tier* tier, int64_t slot);

/* ABI version of this header: major * 10000 + minor * 100 + patch. */
int kvs_version(void);
#define KVS_VERSION 10900

#ifdef __cplusplus
}
#endif

#endif /* KVS_H */

// kvs_noalloc.cu -- kvs_retrieve_noalloc: retrieval for callers that cannot
// allocate GPU memory.
//
// kvs_retrieve keeps its descriptor tables and error word in buffers the
// library allocates on first use.  Some callers cannot let a library allocate:
// serving runtimes that reserve almost all free HBM for their own KV block pool
// at start-up and sub-allocate it themselves (a cudaMalloc in the middle of
// serving can fail, or make their accounting wrong), and latency-critical
// paths where cudaMalloc / cudaFree would synchronise the device.  This entry
// point allocates nothing: its scratch is the file-scope array below, part of
// the library image, which every GPU that loads the library holds until the
// process exits.  Host-side planning uses static storage as well.
//
// The same copy kernels as kvs_retrieve move the bytes; only where their
// scratch lives differs.  Host chunks are read directly over the host link by
// the double-buffered link kernel on kvs_retrieve's CTA cap (no copy-engine
// staging ring, which would need an allocation); device chunks take the vector
// LDG kernel.  The two classes run one after the other on the caller's stream
// (kvs_retrieve runs them side by side on two streams).
#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "kvs.h"
#include "kvs_internal.h"

namespace kvs {
namespace {

// Scratch layout: [error word, 256 B][plane table][entries][blocks][demoted blocks].
static __device__ __align__(256) unsigned char g_scratch[KVS_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
constexpr uint32_t kMaxBlockRefs = KVS_NOALLOC_SCRATCH_BYTES / 4;     // bounds every host table

std::mutex g_na_mu;
void* g_dev_addr[kMaxDevices];                  // device address of g_scratch, per device
bool g_dev_ready[kMaxDevices];

// Host staging, copied into g_scratch by one cudaMemcpyAsync per call.  The
// source is pageable memory: the CUDA runtime documents that an asynchronous
// copy from pageable host memory to device memory returns only once the source
// has been copied to a staging buffer, so the next call may refill g_stage at
// once while the previous upload is still queued on the stream.

unsigned char g_stage[KVS_NOALLOC_SCRATCH_BYTES];
uint64_t g_keys[kMaxBlockRefs];                  // (physical block << 32) | block-ref index
int32_t  g_ref_req[kMaxBlockRefs];               // request of each block-ref
int32_t  g_ref_ntok[kMaxBlockRefs];              // tokens the block-ref writes
int32_t  g_err_host;

int na_fail(int code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    set_last_error(buf);                 // reported by kvs_last_error()
    return code;
}

#define NA_CUDA(call)                                                                       \
    do {                                                                                    \
        cudaError_t e_ = (call);                                                            \
        if (e_ != cudaSuccess)                                                              \
            return na_fail(KVS_ERR_CUDA, "%s failed: %s", #call, cudaGetErrorString(e_));   \
    } while (0)

size_t up256(size_t x) { return (x + 255) & ~(size_t)255; }

// Set-up, once per device, with that device current: the kernel needs the
// device address of g_scratch; in host code the name g_scratch is only a
// host-side stand-in.
int scratch_address(void** out) {
    int dev = 0;
    NA_CUDA(cudaGetDevice(&dev));
    if (dev < 0 || dev >= kMaxDevices) return na_fail(KVS_ERR_UNSUPPORTED, "device %d out of range", dev);
    if (!g_dev_ready[dev]) {
        void* p = nullptr;
        NA_CUDA(cudaGetSymbolAddress(&p, g_scratch));
        g_dev_addr[dev] = p;
        g_dev_ready[dev] = true;
    }
    *out = g_dev_addr[dev];
    return KVS_OK;
}

// Device-visible address of a chunk, checked against its residency the way
// kvs_retrieve checks it: a host chunk must be page-locked host memory mapped
// into the GPU (its device pointer is used), a device chunk device memory.
// Anything else is refused before any work is enqueued.
int chunk_address(const kvs_chunk& c, int32_t r, int32_t j, uint64_t* out) {
    cudaPointerAttributes at{};
    if (cudaPointerGetAttributes(&at, c.base) != cudaSuccess) {
        cudaGetLastError();
        return na_fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: unknown pointer", r, j);
    }
    if (c.residency == KVS_SRC_DEVICE) {
        if (!(at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged))
            return na_fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: not device memory", r, j);
        *out = (uint64_t)c.base;
    } else {
        if (at.type != cudaMemoryTypeHost || !at.devicePointer)
            return na_fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: not mapped page-locked host memory", r, j);
        *out = (uint64_t)at.devicePointer;
    }
    return KVS_OK;
}

int retrieve_noalloc(const kvs_geometry* g, const kvs_paged_cache* cache, const kvs_request* reqs,
                     int32_t nreq, cudaStream_t s, uint32_t flags) {
    const uint32_t allowed = KVS_F_VALIDATE | KVS_F_FORCE_HOSTLINK | KVS_F_FORCE_LDG | 0xFFFF0000u;
    if (flags & ~allowed)
        return na_fail(KVS_ERR_UNSUPPORTED, "kvs_retrieve_noalloc takes only KVS_F_VALIDATE, "
                       "KVS_F_FORCE_HOSTLINK, KVS_F_FORCE_LDG and KVS_F_MAX_CTAS");
    if (!g) return na_fail(KVS_ERR_INVALID_ARG, "geometry is NULL");
    if (g->num_layers <= 0 || g->num_kv_heads <= 0 || g->head_dim <= 0)
        return na_fail(KVS_ERR_INVALID_ARG, "layers, kv heads and head dim must be positive");
    const int e_b = g->elem_bytes;
    if (!(e_b == 1 || e_b == 2 || e_b == 4 || e_b == 8))
        return na_fail(KVS_ERR_INVALID_ARG, "elem_bytes must be 1, 2, 4 or 8 (got %d)", e_b);
    if (g->block_size <= 0 || g->chunk_tokens <= 0 || g->chunk_tokens % g->block_size)
        return na_fail(KVS_ERR_INVALID_ARG, "chunk_tokens (%d) must be a positive multiple of block_size (%d)",
                       g->chunk_tokens, g->block_size);
    if ((int64_t)g->num_layers * 2 > 65536) return na_fail(KVS_ERR_INVALID_ARG, "too many layers");
    if (!cache || !cache->kv_planes) return na_fail(KVS_ERR_INVALID_ARG, "cache or its plane array is NULL");
    if (cache->num_blocks <= 0 || cache->num_blocks > INT32_MAX)
        return na_fail(KVS_ERR_INVALID_ARG, "num_blocks must be in [1, 2^31)");
    if (nreq < 0 || (nreq > 0 && !reqs)) return na_fail(KVS_ERR_INVALID_ARG, "bad request array");

    const int L = g->num_layers, B = g->block_size, C = g->chunk_tokens, P = 2 * L;
    const uint64_t R = (uint64_t)g->num_kv_heads * g->head_dim * e_b;
    const uint32_t bpc = (uint32_t)((C + B - 1) / B);
    uint64_t addr_or = R;
    for (int p = 0; p < P; ++p) {
        if (!cache->kv_planes[p]) return na_fail(KVS_ERR_INVALID_ARG, "plane %d is NULL", p);
        addr_or |= (uint64_t)cache->kv_planes[p];
    }
    uint64_t nent = 0, ndev = 0;
    for (int32_t r = 0; r < nreq; ++r) {
        const kvs_request& q = reqs[r];
        if (q.first_token < 0 || q.first_token % C)
            return na_fail(KVS_ERR_INVALID_ARG, "request %d: first_token %lld is not a non-negative multiple of %d",
                           r, (long long)q.first_token, C);
        if (q.num_tokens < 0 || q.num_chunks < 0 || (q.num_chunks > 0 && !q.chunks))
            return na_fail(KVS_ERR_INVALID_ARG, "request %d: bad token or chunk count", r);
        if (q.first_token + q.num_tokens > INT32_MAX)
            return na_fail(KVS_ERR_INVALID_ARG, "request %d: token range too large", r);
        int64_t sum = 0;
        for (int32_t j = 0; j < q.num_chunks; ++j) {
            const kvs_chunk& c = q.chunks[j];
            if (!c.base) return na_fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: base is NULL", r, j);
            if (c.residency != KVS_SRC_HOST_PINNED && c.residency != KVS_SRC_DEVICE)
                return na_fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: unknown residency %d", r, j, c.residency);
            if (c.num_tokens <= 0 || c.num_tokens > C)
                return na_fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: num_tokens %d not in [1, %d]",
                               r, j, c.num_tokens, C);
            if (j + 1 < q.num_chunks && c.num_tokens != C)
                return na_fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: only the last chunk may be partial", r, j);
            sum += c.num_tokens;
            if (c.residency == KVS_SRC_DEVICE) ++ndev;
        }
        if (sum != q.num_tokens)
            return na_fail(KVS_ERR_INVALID_ARG, "request %d: chunks hold %lld tokens, num_tokens is %lld",
                           r, (long long)sum, (long long)q.num_tokens);
        if (q.num_tokens > 0) {
            const int64_t need = (q.first_token + q.num_tokens + B - 1) / B;
            if (!q.block_table) return na_fail(KVS_ERR_INVALID_ARG, "request %d: block_table is NULL", r);
            if (q.block_table_len < need)
                return na_fail(KVS_ERR_BOUNDS, "request %d: block table has %d entries, %lld needed",
                               r, q.block_table_len, (long long)need);
            for (int64_t k = q.first_token / B; k < need; ++k) {
                const int32_t b = q.block_table[k];
                if (b < 0 || b >= cache->num_blocks)
                    return na_fail(KVS_ERR_BOUNDS, "request %d: block_table[%lld] = %d outside [0, %lld)",
                                   r, (long long)k, b, (long long)cache->num_blocks);
            }
        }
        nent += (uint64_t)q.num_chunks;
    }
    if (nent == 0) return KVS_OK;

    // Scratch needed by this call: refuse anything beyond the static array.
    const bool validate = flags & KVS_F_VALIDATE;
    const uint64_t nrefs = nent * bpc;
    const size_t off_pl = 256;
    const size_t off_en = off_pl + up256((size_t)P * 8);
    const size_t off_bl = off_en + up256((size_t)nent * sizeof(Entry));
    const size_t off_bc = off_bl + up256((size_t)nrefs * 4);
    const size_t need = off_bc + (validate ? up256((size_t)nrefs * 4) : 0);
    if (need > KVS_NOALLOC_SCRATCH_BYTES || nrefs > kMaxBlockRefs)
        return na_fail(KVS_ERR_UNSUPPORTED,
                       "this call needs %zu bytes of descriptor scratch; kvs_retrieve_noalloc holds at most %u "
                       "(KVS_NOALLOC_SCRATCH_BYTES): split the call or use kvs_retrieve",
                       need, (unsigned)KVS_NOALLOC_SCRATCH_BYTES);
    const uint64_t ppr = ((uint64_t)B * R + kPieceBytes - 1) / kPieceBytes;
    if (nrefs * P * ppr >= (1ull << 31))
        return na_fail(KVS_ERR_INVALID_ARG, "call too large: split it (more than 2^31 pieces)");

    // Pack the tables: device-resident entries first, then host-resident ones,
    // so that each class is one contiguous range of entries (one launch each).
    // Block refs: one per (entry, block of its chunk); a ref of a physical
    // block also named by another request is dropped unless it covers the
    // most tokens of that block (the lowest request on ties).
    unsigned char* st = g_stage;
    memset(st, 0, off_bc);
    uint64_t* planes = (uint64_t*)(st + off_pl);
    Entry* entries = (Entry*)(st + off_en);
    int32_t* blocks = (int32_t*)(st + off_bl);
    int32_t* demoted = (int32_t*)(st + off_bc);
    for (int p = 0; p < P; ++p) planes[p] = (uint64_t)cache->kv_planes[p];
    uint32_t e_dev = 0, e_host = (uint32_t)ndev, nk = 0;
    for (int32_t r = 0; r < nreq; ++r) {
        const kvs_request& q = reqs[r];
        int64_t s0 = q.first_token;
        for (int32_t j = 0; j < q.num_chunks; ++j) {
            const kvs_chunk& c = q.chunks[j];
            const uint32_t e = (c.residency == KVS_SRC_DEVICE) ? e_dev++ : e_host++;
            uint64_t addr = 0;
            int rc = chunk_address(c, r, j, &addr);
            if (rc) return rc;
            addr_or |= addr;
            entries[e].chunk = addr;
            entries[e].n_tok = c.num_tokens;
            entries[e].pad = 0;
            for (uint32_t i = 0; i < bpc; ++i) {
                const uint32_t ref = e * bpc + i;
                blocks[ref] = -1;
                if ((int64_t)i * B >= c.num_tokens) continue;
                const int32_t blk = q.block_table[(s0 + (int64_t)i * B) / B];
                blocks[ref] = blk;
                g_keys[nk++] = ((uint64_t)(uint32_t)blk << 32) | ref;
                g_ref_req[ref] = r;
                g_ref_ntok[ref] = std::min<int32_t>(B, c.num_tokens - (int32_t)i * B);
            }
            s0 += c.num_tokens;
        }
    }
    if (validate)
        for (uint64_t k = 0; k < nrefs; ++k) demoted[k] = -1;
    // Sorted by (block, ref), the refs of one block are adjacent; within a
    // block, refs of one request are adjacent too only if the request names
    // the block twice, which is refused (checked against every earlier ref of
    // the block by request).
    std::sort(g_keys, g_keys + nk);                         // in place: no allocation
    bool any_demoted = false;
    for (uint32_t a = 0; a < nk;) {
        uint32_t b = a + 1;
        const uint32_t blk = (uint32_t)(g_keys[a] >> 32);
        while (b < nk && (uint32_t)(g_keys[b] >> 32) == blk) ++b;
        if (b - a > 1) {
            uint32_t keep = (uint32_t)g_keys[a];
            for (uint32_t k = a + 1; k < b; ++k) {
                const uint32_t ref = (uint32_t)g_keys[k];
                for (uint32_t m = a; m < k; ++m)
                    if (g_ref_req[(uint32_t)g_keys[m]] == g_ref_req[ref])
                        return na_fail(KVS_ERR_ALIAS, "request %d names physical block %u twice",
                                       g_ref_req[ref], blk);
                const uint32_t kr = keep;
                if (g_ref_ntok[ref] > g_ref_ntok[kr] ||
                    (g_ref_ntok[ref] == g_ref_ntok[kr] && g_ref_req[ref] < g_ref_req[kr]))
                    keep = ref;
            }
            for (uint32_t k = a; k < b; ++k) {
                const uint32_t ref = (uint32_t)g_keys[k];
                if (ref == keep) continue;
                blocks[ref] = -1;
                if (validate) demoted[ref] = (int32_t)blk;
                any_demoted = true;
            }
        }
        a = b;
    }

    void* dscratch = nullptr;
    int rc = scratch_address(&dscratch);
    if (rc) return rc;
    unsigned char* d = (unsigned char*)dscratch;
    const size_t upload = validate && any_demoted ? need : off_bc;
    NA_CUDA(cudaMemsetAsync(d, 0, sizeof(int32_t), s));             // error word starts at zero
    NA_CUDA(cudaMemcpyAsync(d + off_pl, st + off_pl, upload - off_pl, cudaMemcpyHostToDevice, s));

    int vec = 16;
    while (vec > 1 && (addr_or & (uint64_t)(vec - 1))) vec >>= 1;
    Job j{};
    j.entries = (const Entry*)(d + off_en);
    j.blocks = (const int32_t*)(d + off_bl);
    j.planes = (const uint64_t*)(d + off_pl);
    j.err = (int32_t*)d;
    j.row_bytes = R;
    j.num_blocks = cache->num_blocks;
    j.num_planes = (uint32_t)P;
    j.plane_begin = 0;
    j.blocks_per_chunk = bpc;
    j.piece_bytes = kPieceBytes;
    j.block_size = (uint32_t)B;
    j.pieces_per_run = (uint32_t)ppr;
    j.mode = MODE_RETRIEVE;
    const int cap = (int)KVS_F_GET_MAX_CTAS(flags);
    // host-resident entries: the link kernel on kvs_retrieve's cap (16-byte data)
    const uint32_t nhost = e_host - (uint32_t)ndev;
    if (nhost) {
        Job jh = j;
        jh.entries = j.entries + ndev;
        jh.entry_base = (uint32_t)ndev;
        jh.num_entries = nhost;
        jh.num_pieces = (uint64_t)nhost * P * bpc * ppr;
        if (vec == 16)
            NA_CUDA(launch_link(jh, cap ? cap : hostlink_grid(true), s));
        else
            NA_CUDA(launch_ldg(jh, vec, cap, s));
    }
    if (ndev) {
        Job jd = j;
        jd.entry_base = 0;
        jd.num_entries = (uint32_t)ndev;
        jd.num_pieces = ndev * P * bpc * ppr;
        NA_CUDA(launch_ldg(jd, vec, cap, s));
    }
    if (validate && any_demoted) {
        Job jc = j;
        jc.blocks = (const int32_t*)(d + off_bc);
        jc.entry_base = 0;
        jc.num_entries = (uint32_t)nent;
        jc.num_pieces = nent * P * bpc * ppr;
        jc.mode = MODE_COMPARE;
        NA_CUDA(launch_ldg(jc, vec, cap, s));
    }
    if (validate) {
        NA_CUDA(cudaMemcpyAsync(&g_err_host, d, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
        NA_CUDA(cudaStreamSynchronize(s));
        if (g_err_host != 0) return na_fail(g_err_host, "device reported error %d", g_err_host);
    }
    return KVS_OK;
}

}  // namespace

void noalloc_forget_devices() {
    std::lock_guard<std::mutex> lk(g_na_mu);
    for (int d = 0; d < kMaxDevices; ++d) {
        g_dev_ready[d] = false;
        g_dev_addr[d] = nullptr;
    }
}

}  // namespace kvs

extern "C" int kvs_retrieve_noalloc(const kvs_geometry* geom, const kvs_paged_cache* cache,
                                    const kvs_request* requests, int32_t num_requests,
                                    void* cuda_stream, uint32_t flags) {
    std::lock_guard<std::mutex> lk(kvs::g_na_mu);
    kvs::set_last_error("");
    return kvs::retrieve_noalloc(geom, cache, requests, num_requests, (cudaStream_t)cuda_stream, flags);
}

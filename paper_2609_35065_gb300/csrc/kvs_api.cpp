// kvs_api.cpp -- C ABI, argument validation, planning and variant choice for
// prefix-KV retrieval / store-back (declared in include/kvs.h).
//
// A call is planned on the host: every (request, chunk) pair becomes one
// Entry, every block of a chunk one physical block id, and the 2L plane
// pointers one table.  The three arrays go to the device in one upload (a
// pinned slot copied on a library stream that the caller's stream waits on),
// then one launch per source class
// (per layer group, for layer-wise calls) moves the bytes:
//   device-resident chunks  -> LDG or TMA kernel, HBM to HBM (on a library
//                              stream joined back when host chunks run too);
//   host-resident chunks    -> HOSTLINK: a double-buffered vector kernel loads/stores
//                              host memory over the host link directly, or
//                              HBMCOPY: the copy engine moves whole chunks
//                              through a ring of HBM staging slots and the
//                              device kernel scatters/gathers from there, or
//                              DMA: the copy engine scatters/gathers directly,
//                              one 2D copy per (chunk, block) across all planes
//                              (equally spaced planes only; no SMs used).
#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include <cuda.h>

#include "kvs.h"
#include "kvs_internal.h"

namespace kvs {
namespace {

thread_local std::string t_error;

int fail(int code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    t_error = buf;
    return code;
}

#define KVS_CUDA(call)                                                                  \
    do {                                                                                \
        cudaError_t e_ = (call);                                                        \
        if (e_ != cudaSuccess)                                                          \
            return fail(KVS_ERR_CUDA, "%s failed: %s", #call, cudaGetErrorString(e_));  \
    } while (0)

constexpr int kUploadSlots = 4;
constexpr int kSignalSlots = 4;
constexpr int kRingSlots = 4;
constexpr uint64_t kRingMinSlotBytes = 64ull << 20;

struct UploadSlot {
    void*       host = nullptr;   // pinned
    void*       dev = nullptr;
    size_t      cap = 0;
    cudaEvent_t done = nullptr;   // recorded after the last kernel that reads `dev`
    cudaEvent_t uploaded = nullptr;   // recorded after the host->device copy
    bool        used = false;
};

// Flags of one layer-wise signalling call: [ctas_done][counters x cap][flags x cap].
struct SignalSlot {
    uint32_t*   mem = nullptr;
    uint32_t    cap = 0;          // groups
    uint32_t    gen = 0;
    cudaEvent_t done = nullptr;   // recorded after the kernel that uses `mem`
    bool        used = false;
};

using WaitValueFn = CUresult (*)(CUstream, CUdeviceptr, cuuint32_t, unsigned int);

struct DevState {
    bool         ready = false;
    int          device = -1;
    int          sms = 0;
    int32_t*     err = nullptr;          // device error word
    int32_t*     err_host = nullptr;     // pinned read-back
    UploadSlot   up[kUploadSlots];
    int          next_up = 0;
    // descriptor copies run here, so that a call's upload overlaps the kernels
    // the caller's stream is still running
    cudaStream_t upload_stream = nullptr;
    // HBM staging ring of the HBMCOPY variant
    uint8_t*     ring = nullptr;
    uint64_t     ring_slot_bytes = 0;
    cudaStream_t copy_stream = nullptr;
    cudaEvent_t  ring_filled[kRingSlots] = {};
    cudaEvent_t  ring_free[kRingSlots] = {};
    cudaEvent_t  ev_fork = nullptr, ev_join = nullptr;
    // device-resident chunks run on this stream, beside the host-resident ones
    cudaStream_t aux_stream = nullptr;
    cudaEvent_t  ev_aux_fork = nullptr, ev_aux_join = nullptr;
    // layer-wise signalling: flags written by the copy kernel, waited on by this
    // stream (stream memory operations), which then records the caller's events
    cudaStream_t signal_stream = nullptr;
    SignalSlot   sig[kSignalSlots];
    int          next_sig = 0;
    WaitValueFn  wait_value = nullptr;
    // per-block ownership for de-duplication: stamp[b] == gen -> owner[b] valid
    std::vector<uint32_t> stamp;
    std::vector<int64_t>  owner;
    uint32_t     gen = 0;
    // defaults (kvs_query_bw may change them)
    int          retrieve_host = KVS_VARIANT_HOSTLINK;
    int          store_host = KVS_VARIANT_HOSTLINK;
    int          kernel_device = KVS_KERNEL_LDG;
    size_t       max_pitch = 0;              // largest pitch a 2D copy accepts
    int          hostlink_ctas = 0;          // CTA cap of host-link kernels, 0 = whole GPU
    int          store_ctas = 0;
    int          few_sm_ctas = 0;            // CTA cap of KVS_F_FEW_SMS retrievals
    kvs_bw_report report{};
};

std::mutex g_mu;
std::vector<DevState> g_dev;
int64_t g_launches = 0;

int get_state(DevState** out) {
    int dev = 0;
    KVS_CUDA(cudaGetDevice(&dev));
    if ((int)g_dev.size() <= dev) g_dev.resize(dev + 1);
    DevState& st = g_dev[dev];
    if (!st.ready) {
        st.device = dev;
        KVS_CUDA(cudaDeviceGetAttribute(&st.sms, cudaDevAttrMultiProcessorCount, dev));
        {
            int mp = 0;
            KVS_CUDA(cudaDeviceGetAttribute(&mp, cudaDevAttrMaxPitch, dev));
            st.max_pitch = mp > 0 ? (size_t)mp : 0;
        }
        KVS_CUDA(cudaMalloc(&st.err, sizeof(int32_t)));
        KVS_CUDA(cudaMemset(st.err, 0, sizeof(int32_t)));
        KVS_CUDA(cudaHostAlloc(&st.err_host, sizeof(int32_t), cudaHostAllocDefault));
        for (auto& s : st.up) {
            KVS_CUDA(cudaEventCreateWithFlags(&s.done, cudaEventDisableTiming));
            KVS_CUDA(cudaEventCreateWithFlags(&s.uploaded, cudaEventDisableTiming));
        }
        KVS_CUDA(cudaStreamCreateWithFlags(&st.upload_stream, cudaStreamNonBlocking));
        KVS_CUDA(cudaStreamCreateWithFlags(&st.copy_stream, cudaStreamNonBlocking));
        for (int k = 0; k < kRingSlots; ++k) {
            KVS_CUDA(cudaEventCreateWithFlags(&st.ring_filled[k], cudaEventDisableTiming));
            KVS_CUDA(cudaEventCreateWithFlags(&st.ring_free[k], cudaEventDisableTiming));
        }
        KVS_CUDA(cudaEventCreateWithFlags(&st.ev_fork, cudaEventDisableTiming));
        KVS_CUDA(cudaEventCreateWithFlags(&st.ev_join, cudaEventDisableTiming));
        KVS_CUDA(cudaStreamCreateWithFlags(&st.aux_stream, cudaStreamNonBlocking));
        KVS_CUDA(cudaStreamCreateWithFlags(&st.signal_stream, cudaStreamNonBlocking));
        for (auto& sg : st.sig) KVS_CUDA(cudaEventCreateWithFlags(&sg.done, cudaEventDisableTiming));
        {
            void* fn = nullptr;
            cudaDriverEntryPointQueryResult q{};
            if (cudaGetDriverEntryPointByVersion("cuStreamWaitValue32", &fn, 12000, cudaEnableDefault, &q)
                    == cudaSuccess && q == cudaDriverEntryPointSuccess)
                st.wait_value = (WaitValueFn)fn;
            cudaGetLastError();
        }
        KVS_CUDA(cudaEventCreateWithFlags(&st.ev_aux_fork, cudaEventDisableTiming));
        KVS_CUDA(cudaEventCreateWithFlags(&st.ev_aux_join, cudaEventDisableTiming));
        // Until kvs_query_bw measures them, host-link kernels take a third of the
        // SMs' worth of CTAs: enough to saturate the link, not the whole GPU.
        st.hostlink_ctas = st.store_ctas = std::max(8, st.sms / 3);
        st.few_sm_ctas = std::max(8, st.sms / 8);
        st.report.num_sms = st.sms;
        st.report.hostlink_ctas = st.hostlink_ctas;
        st.report.store_ctas = st.store_ctas;
        st.report.few_sm_ctas = st.few_sm_ctas;
        st.report.chosen_retrieve_host = st.retrieve_host;
        st.report.chosen_store_host = st.store_host;
        st.report.chosen_kernel_device = st.kernel_device;
        st.ready = true;
    }
    *out = &st;
    return KVS_OK;
}

// ---------------------------------------------------------------------------
// Planning
// ---------------------------------------------------------------------------
struct Plan {
    std::vector<uint64_t> planes;
    std::vector<Entry>    entries;       // device-resident first, then host-resident
    std::vector<int32_t>  blocks;        // entries.size() * bpc
    std::vector<int32_t>  demoted;       // block of a writer dropped by de-duplication, else -1
    std::vector<int32_t>  blocks_cmp;    // KVS_F_VALIDATE: the demoted writers, compared
    std::vector<uint64_t> entry_bytes;   // bytes of each entry's chunk buffer
    uint32_t num_device = 0, num_host = 0;
    uint32_t bpc = 0;
    uint64_t row_bytes = 0;
    uint64_t addr_or = 0;                // OR of all addresses and strides (alignment)
    bool     any_dedup = false;
};

bool is_pow2_elem(int e) { return e == 1 || e == 2 || e == 4 || e == 8; }

int validate_geometry(const kvs_geometry* g) {
    if (!g) return fail(KVS_ERR_INVALID_ARG, "geometry is NULL");
    if (g->num_layers <= 0 || g->num_kv_heads <= 0 || g->head_dim <= 0)
        return fail(KVS_ERR_INVALID_ARG, "layers, kv heads and head dim must be positive");
    if (!is_pow2_elem(g->elem_bytes))
        return fail(KVS_ERR_INVALID_ARG, "elem_bytes must be 1, 2, 4 or 8 (got %d)", g->elem_bytes);
    if (g->block_size <= 0 || g->chunk_tokens <= 0 || g->chunk_tokens % g->block_size)
        return fail(KVS_ERR_INVALID_ARG, "chunk_tokens (%d) must be a positive multiple of block_size (%d)",
                    g->chunk_tokens, g->block_size);
    if ((int64_t)g->num_layers * 2 > 65536)
        return fail(KVS_ERR_INVALID_ARG, "too many layers");
    return KVS_OK;
}

// First half of planning: checks every argument and counts entries per class.
// Touches no CUDA state, so invalid calls fail the same way with or without a GPU.
int validate_call(const kvs_geometry* g, const kvs_paged_cache* cache,
                  const kvs_request* reqs, int32_t nreq, Plan& pl) {
    int rc = validate_geometry(g);
    if (rc) return rc;
    if (!cache || !cache->kv_planes) return fail(KVS_ERR_INVALID_ARG, "cache or its plane array is NULL");
    if (cache->num_blocks <= 0 || cache->num_blocks > INT32_MAX)
        return fail(KVS_ERR_INVALID_ARG, "num_blocks must be in [1, 2^31)");
    if (nreq < 0 || (nreq > 0 && !reqs)) return fail(KVS_ERR_INVALID_ARG, "bad request array");

    const int L = g->num_layers, B = g->block_size, C = g->chunk_tokens;
    const int P = 2 * L;
    pl.row_bytes = (uint64_t)g->num_kv_heads * g->head_dim * g->elem_bytes;
    pl.bpc = (uint32_t)((C + B - 1) / B);
    pl.addr_or = pl.row_bytes;
    pl.planes.resize(P);
    for (int p = 0; p < P; ++p) {
        if (!cache->kv_planes[p]) return fail(KVS_ERR_INVALID_ARG, "plane %d is NULL", p);
        pl.planes[p] = (uint64_t)cache->kv_planes[p];
        pl.addr_or |= pl.planes[p];
    }
    // Validate requests, count entries per class.
    for (int32_t r = 0; r < nreq; ++r) {
        const kvs_request& q = reqs[r];
        if (q.first_token < 0 || q.first_token % C)
            return fail(KVS_ERR_INVALID_ARG, "request %d: first_token %lld is not a non-negative multiple of %d",
                        r, (long long)q.first_token, C);
        if (q.num_tokens < 0 || q.num_chunks < 0 || (q.num_chunks > 0 && !q.chunks))
            return fail(KVS_ERR_INVALID_ARG, "request %d: bad token or chunk count", r);
        if (q.first_token + q.num_tokens > INT32_MAX)
            return fail(KVS_ERR_INVALID_ARG, "request %d: token range too large", r);
        int64_t sum = 0;
        for (int32_t j = 0; j < q.num_chunks; ++j) {
            const kvs_chunk& c = q.chunks[j];
            if (!c.base) return fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: base is NULL", r, j);
            if (c.residency != KVS_SRC_HOST_PINNED && c.residency != KVS_SRC_DEVICE)
                return fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: unknown residency %d", r, j, c.residency);
            if (c.num_tokens <= 0 || c.num_tokens > C)
                return fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: num_tokens %d not in [1, %d]",
                            r, j, c.num_tokens, C);
            if (j + 1 < q.num_chunks && c.num_tokens != C)
                return fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: only the last chunk may be partial", r, j);
            sum += c.num_tokens;
            if (c.residency == KVS_SRC_DEVICE) ++pl.num_device; else ++pl.num_host;
        }
        if (sum != q.num_tokens)
            return fail(KVS_ERR_INVALID_ARG, "request %d: chunks hold %lld tokens, num_tokens is %lld",
                        r, (long long)sum, (long long)q.num_tokens);
        if (q.num_tokens > 0) {
            const int64_t need = (q.first_token + q.num_tokens + B - 1) / B;
            if (!q.block_table) return fail(KVS_ERR_INVALID_ARG, "request %d: block_table is NULL", r);
            if (q.block_table_len < need)
                return fail(KVS_ERR_BOUNDS, "request %d: block table has %d entries, %lld needed",
                            r, q.block_table_len, (long long)need);
            for (int64_t k = q.first_token / B; k < need; ++k) {
                const int32_t b = q.block_table[k];
                if (b < 0 || b >= cache->num_blocks)
                    return fail(KVS_ERR_BOUNDS, "request %d: block_table[%lld] = %d outside [0, %lld)",
                                r, (long long)k, b, (long long)cache->num_blocks);
            }
        }
    }

    const uint32_t nent = pl.num_device + pl.num_host;
    const uint64_t runs = (uint64_t)nent * P * pl.bpc;
    const uint64_t ppr = ((uint64_t)B * pl.row_bytes + kPieceBytes - 1) / kPieceBytes;
    if (runs * ppr >= (1ull << 31))
        return fail(KVS_ERR_INVALID_ARG, "call too large: split it (more than 2^31 pieces)");
    return KVS_OK;
}

// With KVS_F_VALIDATE: the memory a call writes may overlap neither itself nor
// the memory it reads (retrieve writes the planes and reads the chunks; store
// writes the chunks and reads the planes), or the copy's result would depend
// on the order of its stores.  Extents: a plane is num_blocks * B rows, a chunk
// of n tokens 2L * n rows.  Sorted by start, a span overlaps an earlier one
// exactly when some earlier span ends after it starts, so one sweep keeping
// the furthest end (over all spans and over written spans) finds every
// conflicting pair's later member.  Host only: no device work.
uint64_t fp8_scale_bytes(const kvs_geometry* g) {
    return ((uint64_t)2 * g->num_layers * g->num_kv_heads * 4 + 255) / 256 * 256;
}

int check_overlaps(const kvs_geometry* g, const kvs_paged_cache* cache, const kvs_request* reqs,
                   int32_t nreq, bool retrieve, bool fp8 = false) {
    struct Span {
        uint64_t lo, hi;
        bool plane;
        int32_t a, b;        // plane index, or (request, chunk)
    };
    const uint64_t row = (uint64_t)g->num_kv_heads * g->head_dim * g->elem_bytes;
    const int P = 2 * g->num_layers;
    std::vector<Span> sp;
    sp.reserve(P);
    for (int p = 0; p < P; ++p) {
        const uint64_t lo = (uint64_t)cache->kv_planes[p];
        sp.push_back({lo, lo + (uint64_t)cache->num_blocks * g->block_size * row, true, p, 0});
    }
    for (int32_t r = 0; r < nreq; ++r)
        for (int32_t j = 0; j < reqs[r].num_chunks; ++j) {
            const kvs_chunk& c = reqs[r].chunks[j];
            const uint64_t lo = (uint64_t)c.base;
            const uint64_t bytes = fp8 ? fp8_scale_bytes(g) + (uint64_t)P * c.num_tokens * row / 2
                                       : (uint64_t)P * c.num_tokens * row;
            sp.push_back({lo, lo + bytes, false, r, j});
        }
    std::sort(sp.begin(), sp.end(), [](const Span& x, const Span& y) { return x.lo < y.lo; });
    auto name = [](const Span& x) {
        char buf[64];
        if (x.plane) snprintf(buf, sizeof buf, "plane %d", x.a);
        else snprintf(buf, sizeof buf, "request %d chunk %d", x.a, x.b);
        return std::string(buf);
    };
    const Span* far_all = nullptr;     // earlier span reaching furthest
    const Span* far_written = nullptr; // same, among written spans
    for (const Span& x : sp) {
        const bool written = (x.plane == retrieve);
        const Span* hit = written ? far_all : far_written;
        if (hit && hit->hi > x.lo)
            return fail(KVS_ERR_ALIAS, "%s overlaps %s (%s)", name(x).c_str(), name(*hit).c_str(),
                        retrieve ? "retrieve writes planes" : "store writes chunks");
        if (!far_all || x.hi > far_all->hi) far_all = &x;
        if (written && (!far_written || x.hi > far_written->hi)) far_written = &x;
    }
    return KVS_OK;
}

// Second half: entries, block ids and de-duplication of shared physical blocks.
int fill_plan(DevState& st, const kvs_geometry* g, const kvs_paged_cache* cache,
              const kvs_request* reqs, int32_t nreq, bool retrieve, uint32_t flags, Plan& pl) {
    const int B = g->block_size;
    const int P = 2 * g->num_layers;
    const bool validate = flags & KVS_F_VALIDATE;
    const bool dedup = retrieve && !(flags & KVS_F_NO_DEDUP);
    const uint32_t nent = pl.num_device + pl.num_host;
    pl.entries.resize(nent);
    pl.entry_bytes.resize(nent);
    pl.blocks.assign((size_t)nent * pl.bpc, -1);

    if (dedup) {
        if (st.stamp.size() < (size_t)cache->num_blocks) {
            st.stamp.assign(cache->num_blocks, 0);
            st.owner.assign(cache->num_blocks, -1);
            st.gen = 0;
        }
        if (++st.gen == 0) {                      // stamp wrap-around
            std::fill(st.stamp.begin(), st.stamp.end(), 0);
            st.gen = 1;
        }
    }

    uint32_t di = 0, hi = pl.num_device;
    for (int32_t r = 0; r < nreq; ++r) {
        const kvs_request& q = reqs[r];
        int64_t s = q.first_token;
        for (int32_t j = 0; j < q.num_chunks; ++j) {
            const kvs_chunk& c = q.chunks[j];
            const uint32_t e = (c.residency == KVS_SRC_DEVICE) ? di++ : hi++;
            uint64_t addr = (uint64_t)c.base;
            if (validate) {
                cudaPointerAttributes at{};
                if (cudaPointerGetAttributes(&at, c.base) != cudaSuccess) {
                    cudaGetLastError();
                    return fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: unknown pointer", r, j);
                }
                if (c.residency == KVS_SRC_DEVICE &&
                    !(at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged))
                    return fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: not device memory", r, j);
                if (c.residency == KVS_SRC_HOST_PINNED) {
                    if (at.type != cudaMemoryTypeHost || !at.devicePointer)
                        return fail(KVS_ERR_INVALID_ARG, "request %d chunk %d: not mapped page-locked host memory", r, j);
                    addr = (uint64_t)at.devicePointer;
                }
            }
            pl.entries[e].chunk = addr;
            pl.entries[e].n_tok = c.num_tokens;
            pl.entries[e].pad = 0;
            pl.entry_bytes[e] = (uint64_t)P * c.num_tokens * pl.row_bytes;
            pl.addr_or |= addr;
            for (int32_t i = 0; i * B < c.num_tokens; ++i) {
                const int64_t t = s + (int64_t)i * B;
                const int32_t blk = q.block_table[t / B];
                const int32_t ntok = std::min<int32_t>(B, c.num_tokens - i * B);
                const int64_t me = ((int64_t)r << 32) | ((int64_t)e * pl.bpc + i);
                if (dedup) {
                    if (st.stamp[blk] == st.gen) {
                        const int64_t prev = st.owner[blk];
                        const int32_t prev_req = (int32_t)(prev >> 32);
                        const int64_t prev_slot = prev & 0xffffffffll;
                        if (prev_req == r)
                            return fail(KVS_ERR_ALIAS, "request %d names physical block %d twice", r, blk);
                        if (!pl.any_dedup) pl.demoted.assign(pl.blocks.size(), -1);
                        pl.any_dedup = true;
                        // keep the writer covering more tokens (earlier request on ties)
                        const uint32_t pe = (uint32_t)(prev_slot / pl.bpc);
                        const int32_t pi = (int32_t)(prev_slot % pl.bpc);
                        const int32_t prev_ntok = std::min<int32_t>(B, pl.entries[pe].n_tok - pi * B);
                        const int64_t my_slot = (int64_t)e * pl.bpc + i;
                        if (ntok > prev_ntok) {
                            pl.blocks[prev_slot] = -1;
                            pl.demoted[prev_slot] = blk;
                            pl.blocks[my_slot] = blk;
                            st.owner[blk] = me;
                        } else {
                            pl.demoted[my_slot] = blk;
                        }
                        continue;
                    }
                    st.stamp[blk] = st.gen;
                    st.owner[blk] = me;
                }
                pl.blocks[(uint64_t)e * pl.bpc + i] = blk;
            }
            s += c.num_tokens;
        }
    }
    // With KVS_F_VALIDATE the demoted writers are compared against what the
    // kept writer put into the block.
    if (pl.any_dedup && validate) pl.blocks_cmp = pl.demoted;
    return KVS_OK;
}

int vec_bytes_for(uint64_t addr_or) {
    int v = 16;
    while (v > 1 && (addr_or & (uint64_t)(v - 1))) v >>= 1;
    return v;
}

// Copies the plan's tables into an upload slot and onto the device (caller stream).
struct Uploaded {
    const Entry*    entries;
    const int32_t*  blocks;
    const int32_t*  blocks_cmp;
    const uint64_t* planes;
    UploadSlot*     slot;
};

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Marks an upload slot in use on every exit path once its copy is enqueued:
// the slot's event is recorded after everything the call enqueued on `s`.
struct SlotGuard {
    UploadSlot* slot = nullptr;
    cudaStream_t s = nullptr;
    ~SlotGuard() {
        if (slot && cudaEventRecord(slot->done, s) == cudaSuccess) slot->used = true;
    }
};

int upload(DevState& st, const Plan& pl, cudaStream_t s, Uploaded& u) {
    const size_t b_pl = align_up(pl.planes.size() * 8, 256);
    const size_t b_en = align_up(pl.entries.size() * sizeof(Entry), 256);
    const size_t b_bl = align_up(pl.blocks.size() * 4, 256);
    const size_t b_bc = align_up(pl.blocks_cmp.size() * 4, 256);
    const size_t need = b_pl + b_en + b_bl + b_bc;
    UploadSlot& sl = st.up[st.next_up];
    st.next_up = (st.next_up + 1) % kUploadSlots;
    if (sl.used) KVS_CUDA(cudaEventSynchronize(sl.done));
    if (sl.cap < need) {
        if (sl.host) { cudaFreeHost(sl.host); sl.host = nullptr; }
        if (sl.dev) { cudaFree(sl.dev); sl.dev = nullptr; }
        const size_t cap = std::max<size_t>(align_up(need * 2, 1 << 16), 1 << 16);
        if (cudaHostAlloc(&sl.host, cap, cudaHostAllocDefault) != cudaSuccess ||
            cudaMalloc(&sl.dev, cap) != cudaSuccess) {
            cudaGetLastError();
            sl.cap = 0;
            return fail(KVS_ERR_NOMEM, "cannot allocate a %zu-byte descriptor slot", cap);
        }
        sl.cap = cap;
    }
    uint8_t* h = (uint8_t*)sl.host;
    memcpy(h, pl.planes.data(), pl.planes.size() * 8);
    memcpy(h + b_pl, pl.entries.data(), pl.entries.size() * sizeof(Entry));
    memcpy(h + b_pl + b_en, pl.blocks.data(), pl.blocks.size() * 4);
    if (b_bc) memcpy(h + b_pl + b_en + b_bl, pl.blocks_cmp.data(), pl.blocks_cmp.size() * 4);
    // The slot's previous readers have finished (its `done` event, waited on
    // above, follows them on the caller's stream), so the copy does not have to
    // queue behind the caller's stream: only the kernels of this call wait for it.
    KVS_CUDA(cudaMemcpyAsync(sl.dev, sl.host, need, cudaMemcpyHostToDevice, st.upload_stream));
    cudaError_t e = cudaEventRecord(sl.uploaded, st.upload_stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, sl.uploaded, 0);
    if (e != cudaSuccess) {
        cudaStreamSynchronize(st.upload_stream);   // the slot is not tracked by `done`
        return fail(KVS_ERR_CUDA, "descriptor upload: %s", cudaGetErrorString(e));
    }
    uint8_t* d = (uint8_t*)sl.dev;
    u.planes = (const uint64_t*)d;
    u.entries = (const Entry*)(d + b_pl);
    u.blocks = (const int32_t*)(d + b_pl + b_en);
    u.blocks_cmp = b_bc ? (const int32_t*)(d + b_pl + b_en + b_bl) : nullptr;
    u.slot = &sl;
    return KVS_OK;
}

Job make_job(DevState& st, const kvs_geometry* g, const kvs_paged_cache* cache, const Plan& pl,
             const Uploaded& u, uint32_t first_entry, uint32_t num_entries, Mode mode,
             uint32_t plane_begin = 0, uint32_t plane_count = 0) {
    Job j{};
    j.entries = u.entries + first_entry;
    j.blocks = u.blocks;
    j.planes = u.planes;
    j.err = st.err;
    j.row_bytes = pl.row_bytes;
    j.num_blocks = cache->num_blocks;
    j.num_entries = num_entries;
    j.entry_base = first_entry;
    j.plane_begin = plane_begin;
    j.num_planes = plane_count ? plane_count : (uint32_t)pl.planes.size() - plane_begin;
    j.blocks_per_chunk = pl.bpc;
    j.piece_bytes = kPieceBytes;
    j.block_size = (uint32_t)g->block_size;
    const uint64_t run_max = (uint64_t)g->block_size * pl.row_bytes;
    j.pieces_per_run = (uint32_t)((run_max + kPieceBytes - 1) / kPieceBytes);
    j.num_pieces = (uint64_t)num_entries * j.num_planes * j.blocks_per_chunk * j.pieces_per_run;
    j.mode = mode;
    return j;
}

// Internal flavours: the double-buffered kernel used for host-resident chunks,
// with L2 prefetches, and with shared-memory stages (KVS_F_FEW_SMS).
constexpr int kKernelLink = 100;
constexpr int kKernelLinkPrefetch = 101;   // retrieval only
constexpr int kKernelLinkStaged = 102;     // retrieval only

int launch_kernel(const Job& j, int flavour, int vec, int grid, cudaStream_t s) {
    if (j.num_pieces == 0) return KVS_OK;
    cudaError_t e = (flavour == KVS_KERNEL_TMA) ? launch_tma(j, grid, s)
                  : (flavour == kKernelLinkStaged && vec == 16) ? launch_link_staged(j, grid, s)
                  : (flavour == kKernelLinkPrefetch && vec == 16) ? launch_link_prefetch(j, grid, s)
                  : ((flavour == kKernelLink || flavour == kKernelLinkPrefetch || flavour == kKernelLinkStaged) && vec == 16)
                      ? launch_link(j, grid, s)
                  : launch_ldg(j, vec, grid, s);
    if (e != cudaSuccess) return fail(KVS_ERR_CUDA, "kernel launch failed: %s", cudaGetErrorString(e));
    ++g_launches;
    return KVS_OK;
}

int ensure_ring(DevState& st, uint64_t max_entry_bytes, cudaStream_t s) {
    const uint64_t want = std::max<uint64_t>(kRingMinSlotBytes, align_up(max_entry_bytes, 1 << 20));
    if (st.ring && st.ring_slot_bytes >= want) return KVS_OK;
    if (st.ring) {
        KVS_CUDA(cudaStreamSynchronize(s));
        KVS_CUDA(cudaStreamSynchronize(st.copy_stream));
        KVS_CUDA(cudaFree(st.ring));
        st.ring = nullptr;
    }
    if (cudaMalloc(&st.ring, want * kRingSlots) != cudaSuccess) {
        cudaGetLastError();
        st.ring_slot_bytes = 0;
        return fail(KVS_ERR_NOMEM, "cannot allocate the %llu-byte HBM staging ring",
                    (unsigned long long)(want * kRingSlots));
    }
    st.ring_slot_bytes = want;
    return KVS_OK;
}

// Host chunks through the copy engine and the HBM ring.  Batches of whole
// chunks fill one ring slot each; the copy stream and the caller's stream
// hand slots back and forth with events.
int run_hbmcopy(DevState& st, const kvs_geometry* g, const kvs_paged_cache* cache, Plan& pl,
                const Uploaded& u, Mode mode, int flavour, int grid, cudaStream_t s,
                const std::vector<const void*>& host_addr) {
    uint64_t max_bytes = 0;
    for (uint32_t e = pl.num_device; e < pl.entries.size(); ++e) max_bytes = std::max(max_bytes, pl.entry_bytes[e]);
    int rc = ensure_ring(st, max_bytes, s);
    if (rc) return rc;
    // Entries in the device copy of the table still point at host memory; the
    // ring kernels use a second upload whose chunk addresses point into slots.
    Plan ring_plan = pl;
    std::vector<uint32_t> batch_first, batch_slot;
    uint64_t used = st.ring_slot_bytes;    // force a new batch at the first entry
    int slot = -1, nb = 0;
    for (uint32_t e = pl.num_device; e < pl.entries.size(); ++e) {
        const uint64_t b = align_up(pl.entry_bytes[e], 256);
        if (used + b > st.ring_slot_bytes) {
            slot = (slot + 1) % kRingSlots;
            batch_first.push_back(e);
            batch_slot.push_back((uint32_t)slot);
            used = 0;
            ++nb;
        }
        ring_plan.entries[e].chunk = (uint64_t)(st.ring + (uint64_t)slot * st.ring_slot_bytes + used);
        ring_plan.addr_or |= ring_plan.entries[e].chunk;
        used += b;
    }
    batch_first.push_back((uint32_t)pl.entries.size());
    Uploaded ru;
    rc = upload(st, ring_plan, s, ru);
    if (rc) return rc;
    SlotGuard ring_guard{ru.slot, s};
    const int vec = vec_bytes_for(ring_plan.addr_or);
    if (flavour == KVS_KERNEL_TMA && vec != 16) flavour = KVS_KERNEL_LDG;

    KVS_CUDA(cudaEventRecord(st.ev_fork, s));
    KVS_CUDA(cudaStreamWaitEvent(st.copy_stream, st.ev_fork, 0));
    for (int b = 0; b < nb; ++b) {
        const uint32_t e0 = batch_first[b], e1 = batch_first[b + 1];
        const int k = (int)batch_slot[b];
        Job j = make_job(st, g, cache, ring_plan, ru, e0, e1 - e0, mode);
        if (mode == MODE_RETRIEVE) {
            KVS_CUDA(cudaStreamWaitEvent(st.copy_stream, st.ring_free[k], 0));
            for (uint32_t e = e0; e < e1; ++e)
                KVS_CUDA(cudaMemcpyAsync((void*)ring_plan.entries[e].chunk, host_addr[e - pl.num_device],
                                         pl.entry_bytes[e], cudaMemcpyHostToDevice, st.copy_stream));
            KVS_CUDA(cudaEventRecord(st.ring_filled[k], st.copy_stream));
            KVS_CUDA(cudaStreamWaitEvent(s, st.ring_filled[k], 0));
            rc = launch_kernel(j, flavour, vec, grid, s);
            if (rc) return rc;
            KVS_CUDA(cudaEventRecord(st.ring_free[k], s));
        } else {
            KVS_CUDA(cudaStreamWaitEvent(s, st.ring_free[k], 0));
            rc = launch_kernel(j, flavour, vec, grid, s);
            if (rc) return rc;
            KVS_CUDA(cudaEventRecord(st.ring_filled[k], s));
            KVS_CUDA(cudaStreamWaitEvent(st.copy_stream, st.ring_filled[k], 0));
            for (uint32_t e = e0; e < e1; ++e)
                KVS_CUDA(cudaMemcpyAsync((void*)host_addr[e - pl.num_device], (const void*)ring_plan.entries[e].chunk,
                                         pl.entry_bytes[e], cudaMemcpyDeviceToHost, st.copy_stream));
            KVS_CUDA(cudaEventRecord(st.ring_free[k], st.copy_stream));
        }
    }
    KVS_CUDA(cudaEventRecord(st.ev_join, st.copy_stream));
    KVS_CUDA(cudaStreamWaitEvent(s, st.ev_join, 0));
    return KVS_OK;
}

// Spacing of the planes when plane p starts at plane 0 + p * pitch for every p
// (one [2L][NB*B*H*D] allocation), with the pitch within the 2D-copy limit;
// 0 otherwise.
uint64_t dma_pitch(const DevState& st, const Plan& pl, uint64_t row_span) {
    const size_t P = pl.planes.size();
    if (P < 2) return row_span;
    if (pl.planes[1] <= pl.planes[0]) return 0;
    const uint64_t pitch = pl.planes[1] - pl.planes[0];
    if (pitch < row_span || pitch > st.max_pitch) return 0;
    for (size_t p = 2; p < P; ++p)
        if (pl.planes[p] != pl.planes[0] + p * pitch) return 0;
    return pitch;
}

// Host chunks by the copy engine alone: for each (chunk, block) one 2D copy
// whose rows are the 2L planes -- source rows n*R apart in the chunk,
// destination rows `pitch` apart in the cache -- each row the block's tokens
// x R bytes.  Blocks dropped by de-duplication are skipped.  No kernel runs.
int run_dma(const kvs_geometry* g, const Plan& pl, uint64_t pitch, bool retrieve, cudaStream_t s,
            const std::vector<const void*>& host_addr) {
    const int B = g->block_size;
    const size_t P = pl.planes.size();
    const uint64_t R = pl.row_bytes;
    for (uint32_t e = pl.num_device; e < pl.entries.size(); ++e) {
        const int32_t n = pl.entries[e].n_tok;
        const uint8_t* chunk = (const uint8_t*)host_addr[e - pl.num_device];
        for (uint32_t i = 0; i < pl.bpc && (int32_t)i * B < n; ++i) {
            const int32_t blk = pl.blocks[(size_t)e * pl.bpc + i];
            if (blk < 0) continue;
            const uint64_t width = (uint64_t)std::min(B, n - (int32_t)i * B) * R;
            uint8_t* c = (uint8_t*)chunk + (uint64_t)i * B * R;
            uint8_t* q = (uint8_t*)pl.planes[0] + (uint64_t)blk * B * R;
            cudaError_t err = retrieve
                ? cudaMemcpy2DAsync(q, pitch, c, (uint64_t)n * R, width, P, cudaMemcpyDefault, s)
                : cudaMemcpy2DAsync(c, (uint64_t)n * R, q, pitch, width, P, cudaMemcpyDefault, s);
            if (err != cudaSuccess)
                return fail(KVS_ERR_CUDA, "2D copy of chunk %u block %u failed: %s", e, i, cudaGetErrorString(err));
        }
    }
    return KVS_OK;
}

int read_error_word(DevState& st, cudaStream_t s) {
    KVS_CUDA(cudaMemcpyAsync(st.err_host, st.err, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
    KVS_CUDA(cudaStreamSynchronize(s));
    const int32_t code = *st.err_host;
    if (code != 0) {
        KVS_CUDA(cudaMemsetAsync(st.err, 0, sizeof(int32_t), s));
        KVS_CUDA(cudaStreamSynchronize(s));
        return fail(code, "device reported error %d", code);
    }
    return KVS_OK;
}

// layers_per_step > 0: layer-wise copy, one launch group per `layers_per_step`
// layers, each preceded by a wait on ready_events[group] and followed by a
// record of layer_events[group] (either if given) on the caller's stream; with
// KVS_F_LAYER_SIGNAL (host chunks, events, no ready events) one resident launch
// signals every group instead.
int copy_call(const kvs_geometry* g, const kvs_paged_cache* cache, const kvs_request* reqs,
              int32_t nreq, void* stream, uint32_t flags, bool retrieve,
              int32_t layers_per_step = 0, void* const* layer_events = nullptr,
              void* const* ready_events = nullptr) {
    const bool f_host = flags & KVS_F_FORCE_HOSTLINK, f_hbm = flags & KVS_F_FORCE_HBMCOPY;
    const bool f_dma = flags & KVS_F_FORCE_DMA;
    const bool f_ldg = flags & KVS_F_FORCE_LDG, f_tma = flags & KVS_F_FORCE_TMA;
    if ((int)f_host + (int)f_hbm + (int)f_dma > 1 || (f_ldg && f_tma))
        return fail(KVS_ERR_INVALID_ARG, "conflicting FORCE flags");
    // KVS_F_FEW_SMS: host chunks over the host link, on the staged kernel (retrieval)
    const bool f_few = retrieve && (flags & KVS_F_FEW_SMS);
    if (f_few && (f_hbm || f_dma || (flags & (KVS_F_PREFETCH_L2 | KVS_F_LAYER_SIGNAL))))
        return fail(KVS_ERR_INVALID_ARG, "KVS_F_FEW_SMS takes the host-link variant, without "
                    "KVS_F_PREFETCH_L2 or KVS_F_LAYER_SIGNAL");
    if ((flags & KVS_F_LAYER_LAUNCHES) && (flags & KVS_F_LAYER_SIGNAL))
        return fail(KVS_ERR_INVALID_ARG, "KVS_F_LAYER_LAUNCHES and KVS_F_LAYER_SIGNAL together");
    if (ready_events && (flags & KVS_F_LAYER_SIGNAL))
        return fail(KVS_ERR_INVALID_ARG, "ready events need one launch per group, not KVS_F_LAYER_SIGNAL");
    if (layers_per_step < 0) return fail(KVS_ERR_INVALID_ARG, "layers_per_step must be positive");
    if (layers_per_step > 0 && (f_hbm || f_dma))
        return fail(KVS_ERR_UNSUPPORTED, "layer-wise copies move host chunks over the host link only");
    Plan pl;
    int rc = validate_call(g, cache, reqs, nreq, pl);
    if (rc) return rc;
    if (flags & KVS_F_VALIDATE) {
        rc = check_overlaps(g, cache, reqs, nreq, retrieve);
        if (rc) return rc;
    }
    const int L = g->num_layers;
    const int lps = layers_per_step > 0 ? std::min(layers_per_step, L) : L;
    const int groups = (L + lps - 1) / lps;
    cudaStream_t s = (cudaStream_t)stream;
    if (pl.num_device + pl.num_host == 0) {
        // nothing to copy: the layer events still mark "ready" in stream order
        if (layers_per_step > 0 && layer_events)
            for (int k = 0; k < groups; ++k)
                if (layer_events[k]) KVS_CUDA(cudaEventRecord((cudaEvent_t)layer_events[k], s));
        return KVS_OK;
    }
    DevState* stp = nullptr;
    rc = get_state(&stp);
    if (rc) return rc;
    DevState& st = *stp;
    rc = fill_plan(st, g, cache, reqs, nreq, retrieve, flags, pl);
    if (rc) return rc;
    const int grid = (int)KVS_F_GET_MAX_CTAS(flags);
    const int vec = vec_bytes_for(pl.addr_or);
    int flavour = f_tma ? KVS_KERNEL_TMA : f_ldg ? KVS_KERNEL_LDG : st.kernel_device;
    if (flavour == KVS_KERNEL_TMA && vec != 16) {
        if (f_tma) return fail(KVS_ERR_UNSUPPORTED, "TMA needs 16-byte aligned chunks, planes and rows");
        flavour = KVS_KERNEL_LDG;
    }
    int host_variant = (f_host || f_few) ? KVS_VARIANT_HOSTLINK : f_hbm ? KVS_VARIANT_HBMCOPY
                     : f_dma ? KVS_VARIANT_DMA : (retrieve ? st.retrieve_host : st.store_host);
    if (layers_per_step > 0) host_variant = KVS_VARIANT_HOSTLINK;
    uint64_t pitch = 0;
    if (host_variant == KVS_VARIANT_DMA && pl.num_host) {
        pitch = dma_pitch(st, pl, (uint64_t)g->block_size * pl.row_bytes);
        if (!pitch) {
            if (f_dma) return fail(KVS_ERR_UNSUPPORTED, "KVS_F_FORCE_DMA needs equally spaced planes "
                                   "(plane p at plane 0 + p * pitch, pitch within the 2D-copy limit)");
            host_variant = KVS_VARIANT_HOSTLINK;
        }
    }
    const Mode mode = retrieve ? MODE_RETRIEVE : MODE_STORE;
    const int host_grid = grid ? grid : f_few ? st.few_sm_ctas : (retrieve ? st.hostlink_ctas : st.store_ctas);

    Uploaded u;
    rc = upload(st, pl, s, u);
    if (rc) return rc;
    SlotGuard guard{u.slot, s};
    // Layer-wise, host chunks only: one persistent launch that publishes each
    // group's completion; the signal stream waits on the flags and records the
    // caller's events.  The kernel is enqueued before any wait, never waits on
    // anything itself, and writes every flag before it ends.
    if (layers_per_step > 0 && layer_events && !pl.num_device && vec == 16 && st.wait_value &&
        (flags & KVS_F_LAYER_SIGNAL)) {
        SignalSlot& sg = st.sig[st.next_sig];
        st.next_sig = (st.next_sig + 1) % kSignalSlots;
        if (sg.used) KVS_CUDA(cudaEventSynchronize(sg.done));
        if (sg.cap < (uint32_t)groups) {
            if (sg.mem) KVS_CUDA(cudaFree(sg.mem));
            sg.mem = nullptr;
            if (cudaMalloc(&sg.mem, (1 + 2 * (size_t)groups) * sizeof(uint32_t)) != cudaSuccess) {
                cudaGetLastError();
                sg.cap = 0;
                return fail(KVS_ERR_NOMEM, "cannot allocate layer flags");
            }
            KVS_CUDA(cudaMemset(sg.mem, 0, (1 + 2 * (size_t)groups) * sizeof(uint32_t)));
            sg.cap = (uint32_t)groups;
            sg.gen = 0;
        }
        if (++sg.gen == 0) ++sg.gen;
        Signal sig{sg.mem + 1, sg.mem + 1 + sg.cap, sg.mem, sg.gen, (uint32_t)groups, (uint32_t)(2 * lps)};
        KVS_CUDA(cudaMemsetAsync(sg.mem, 0, (1 + (size_t)groups) * sizeof(uint32_t), s));
        Job j = make_job(st, g, cache, pl, u, 0, pl.num_host, mode);
        if (j.num_pieces) {
            cudaError_t e = launch_link_signal(j, sig, host_grid, s);
            if (e != cudaSuccess) return fail(KVS_ERR_CUDA, "kernel launch failed: %s", cudaGetErrorString(e));
            ++g_launches;
        }
        KVS_CUDA(cudaEventRecord(sg.done, s));
        sg.used = true;
        bool waits_ok = j.num_pieces > 0;
        for (int k = 0; k < groups; ++k) {
            if (!layer_events[k]) continue;
            if (waits_ok && st.wait_value((CUstream)st.signal_stream, (CUdeviceptr)(sig.flags + k), sig.gen,
                                          CU_STREAM_WAIT_VALUE_GEQ) != CUDA_SUCCESS) {
                st.wait_value = nullptr;            // not available here: events fire at kernel end
                waits_ok = false;
            }
            KVS_CUDA(cudaEventRecord((cudaEvent_t)layer_events[k], waits_ok ? st.signal_stream : s));
        }
        if (!pl.blocks_cmp.empty()) {
            Job jc = make_job(st, g, cache, pl, u, 0, (uint32_t)pl.entries.size(), MODE_COMPARE);
            jc.blocks = u.blocks_cmp;
            rc = launch_kernel(jc, KVS_KERNEL_LDG, vec, grid, s);
            if (rc) return rc;
        }
        if (flags & KVS_F_VALIDATE) {
            KVS_CUDA(cudaEventRecord(u.slot->done, s));   // before the synchronising read
            u.slot->used = true;
            guard.slot = nullptr;
            return read_error_word(st, s);
        }
        return KVS_OK;
    }
    // With both classes present, the HBM-bound device part runs on the aux
    // stream while the link-bound host part runs on the caller's stream.  The
    // host part is launched first: its few CTAs take their SM slots before the
    // whole-GPU device grid fills every SM.
    const bool fork = pl.num_device && pl.num_host;
    for (int k = 0; k < groups; ++k) {
        const uint32_t p0 = (uint32_t)(2 * k * lps);
        const uint32_t np = (uint32_t)(2 * (std::min(L, (k + 1) * lps) - k * lps));
        if (ready_events && ready_events[k])
            KVS_CUDA(cudaStreamWaitEvent(s, (cudaEvent_t)ready_events[k], 0));
        if (fork) {
            KVS_CUDA(cudaEventRecord(st.ev_aux_fork, s));
            KVS_CUDA(cudaStreamWaitEvent(st.aux_stream, st.ev_aux_fork, 0));
        }
        if (pl.num_host) {
            if (host_variant == KVS_VARIANT_HBMCOPY || host_variant == KVS_VARIANT_DMA) {
                std::vector<const void*> host_addr(pl.num_host);
                for (uint32_t e = pl.num_device; e < pl.entries.size(); ++e)
                    host_addr[e - pl.num_device] = (const void*)pl.entries[e].chunk;
                rc = host_variant == KVS_VARIANT_DMA ? run_dma(g, pl, pitch, retrieve, s, host_addr)
                                                     : run_hbmcopy(st, g, cache, pl, u, mode, flavour, grid, s, host_addr);
            } else {
                const int lf = f_few ? kKernelLinkStaged
                             : (retrieve && (flags & KVS_F_PREFETCH_L2)) ? kKernelLinkPrefetch : kKernelLink;
                rc = launch_kernel(make_job(st, g, cache, pl, u, pl.num_device, pl.num_host, mode, p0, np),
                                   lf, vec, host_grid, s);
            }
            if (rc) return rc;
        }
        if (pl.num_device) {
            const cudaStream_t ds = fork ? st.aux_stream : s;
            rc = launch_kernel(make_job(st, g, cache, pl, u, 0, pl.num_device, mode, p0, np), flavour, vec, grid, ds);
            if (rc) return rc;
            if (fork) KVS_CUDA(cudaEventRecord(st.ev_aux_join, st.aux_stream));
        }
        if (fork) KVS_CUDA(cudaStreamWaitEvent(s, st.ev_aux_join, 0));
        if (layers_per_step > 0 && layer_events && layer_events[k])
            KVS_CUDA(cudaEventRecord((cudaEvent_t)layer_events[k], s));
    }
    if (!pl.blocks_cmp.empty()) {
        Job j = make_job(st, g, cache, pl, u, 0, (uint32_t)pl.entries.size(), MODE_COMPARE);
        j.blocks = u.blocks_cmp;
        rc = launch_kernel(j, KVS_KERNEL_LDG, vec, grid, s);
        if (rc) return rc;
    }
    if (flags & KVS_F_VALIDATE) {
        KVS_CUDA(cudaEventRecord(u.slot->done, s));       // before the synchronising read
        u.slot->used = true;
        guard.slot = nullptr;
        return read_error_word(st, s);
    }
    return KVS_OK;
}

// fp8 chunks (E4M3 codes with per-head binary32 scales) <-> BF16 planes.  Host
// chunks run first on the host-link grid, device chunks after them on the
// same stream.  A physical block named by two requests is refused: the
// quantised copies of a shared block differ with each chunk's scales, so no
// single writer would be the right one.
// layers_per_step > 0: layer groups in layer order, each preceded by a wait on
// ready_events[k] and followed by a record of layer_events[k] (either if given).
int fp8_call(const kvs_geometry* g, const kvs_paged_cache* cache, const kvs_request* reqs,
             int32_t nreq, void* stream, uint32_t flags, bool retrieve, int32_t layers_per_step = 0,
             void* const* layer_events = nullptr, void* const* ready_events = nullptr) {
    const uint32_t allowed = KVS_F_VALIDATE | KVS_F_FORCE_HOSTLINK | KVS_F_FORCE_LDG | KVS_F_FEW_SMS | 0xFFFF0000u;
    if (flags & ~allowed)
        return fail(KVS_ERR_UNSUPPORTED, "fp8 calls take only KVS_F_VALIDATE, KVS_F_FORCE_HOSTLINK, "
                    "KVS_F_FORCE_LDG, KVS_F_FEW_SMS and KVS_F_MAX_CTAS");
    const bool few = retrieve && (flags & KVS_F_FEW_SMS);
    Plan pl;
    int rc = validate_call(g, cache, reqs, nreq, pl);
    if (rc) return rc;
    if (g->elem_bytes != 2)
        return fail(KVS_ERR_INVALID_ARG, "fp8 chunks fill BF16 planes: elem_bytes must be 2 (got %d)", g->elem_bytes);
    if (g->head_dim % 16)
        return fail(KVS_ERR_UNSUPPORTED, "fp8 chunks need head_dim a multiple of 16 (got %d)", g->head_dim);
    if ((uint32_t)g->num_kv_heads > kFp8MaxHeads)
        return fail(KVS_ERR_UNSUPPORTED, "fp8 chunks support at most %u kv heads", kFp8MaxHeads);
    for (int32_t r = 0; r < nreq; ++r)
        for (int32_t j = 0; j < reqs[r].num_chunks; ++j)
            if ((uint64_t)reqs[r].chunks[j].base & 15)
                return fail(KVS_ERR_UNSUPPORTED, "request %d chunk %d: fp8 chunks must be 16-byte aligned", r, j);
    if (pl.addr_or & 15) return fail(KVS_ERR_UNSUPPORTED, "fp8 calls need 16-byte aligned planes");
    if (flags & KVS_F_VALIDATE) {
        rc = check_overlaps(g, cache, reqs, nreq, retrieve, true);
        if (rc) return rc;
    }
    if (pl.num_device + pl.num_host == 0) {
        // nothing to copy: the layer events still mark "ready" in stream order
        if (layers_per_step > 0 && layer_events)
            for (int k = 0; k < (g->num_layers + layers_per_step - 1) / layers_per_step; ++k)
                if (layer_events[k]) KVS_CUDA(cudaEventRecord((cudaEvent_t)layer_events[k], (cudaStream_t)stream));
        return KVS_OK;
    }
    DevState* stp = nullptr;
    rc = get_state(&stp);
    if (rc) return rc;
    DevState& st = *stp;
    rc = fill_plan(st, g, cache, reqs, nreq, retrieve, flags & ~KVS_F_NO_DEDUP, pl);
    if (rc) return rc;
    if (pl.any_dedup) {
        for (size_t k = 0; k < pl.demoted.size(); ++k)
            if (pl.demoted[k] >= 0)
                return fail(KVS_ERR_ALIAS, "fp8 retrieval: physical block %d is named by two requests", pl.demoted[k]);
    }
    pl.blocks_cmp.clear();
    cudaStream_t s = (cudaStream_t)stream;
    Uploaded u;
    rc = upload(st, pl, s, u);
    if (rc) return rc;
    SlotGuard guard{u.slot, s};
    const int cap = (int)KVS_F_GET_MAX_CTAS(flags);
    const uint32_t hd = (uint32_t)(g->num_kv_heads * g->head_dim);
    auto fjob = [&](uint32_t first, uint32_t count, uint32_t p0, uint32_t np) {
        Fp8Job f{};
        f.job = make_job(st, g, cache, pl, u, first, count, retrieve ? MODE_RETRIEVE : MODE_STORE, p0, np);
        const uint64_t run_codes = (uint64_t)g->block_size * hd;
        f.job.pieces_per_run = (uint32_t)((run_codes + kFp8PieceCodes - 1) / kFp8PieceCodes);
        f.job.num_pieces = (uint64_t)count * f.job.num_planes * f.job.blocks_per_chunk * f.job.pieces_per_run;
        f.heads = (uint32_t)g->num_kv_heads;
        f.head_dim = (uint32_t)g->head_dim;
        f.scale_bytes = (uint32_t)fp8_scale_bytes(g);
        // floor(2^32 / B) + 1 fits 32 bits for B >= 2; the kernel divides by B = 1 itself
        f.block_magic = g->block_size >= 2 ? (uint32_t)((1ull << 32) / (uint64_t)g->block_size + 1) : 0;
        auto recip = [](uint32_t d, uint32_t& m, uint32_t& p) {
            uint32_t l = 0;
            while ((1ull << l) < d) ++l;
            p = 31 + l;
            m = (uint32_t)(((1ull << p) + d - 1) / d);
        };
        recip(f.job.pieces_per_run, f.ppr_m, f.ppr_p);
        recip(f.job.num_planes * f.job.blocks_per_chunk, f.pe_m, f.pe_p);
        recip(f.job.blocks_per_chunk, f.bpc_m, f.bpc_p);
        f.rows_whole = (kFp8PieceCodes / 16) % (hd / 16) == 0;
        return f;
    };
    // store-back segments: one per (chunk, plane, head)
    auto fp8_segments = [](const Fp8Job& f) {
        return (uint64_t)f.job.num_entries * f.job.num_planes * f.heads;
    };
    auto run = [&](const Fp8Job& f, int grid, bool device_chunks) -> int {
        cudaError_t e = !retrieve ? launch_fp8_store(f, grid, s, (uint32_t)g->chunk_tokens, device_chunks)
                      : (few && !device_chunks) ? launch_fp8_retrieve_staged(f, grid, s)
                                                : launch_fp8_retrieve(f, grid, s);
        if (e != cudaSuccess) return fail(KVS_ERR_CUDA, "fp8 kernel launch failed: %s", cudaGetErrorString(e));
        ++g_launches;
        return KVS_OK;
    };
    const int L = g->num_layers;
    const int lps = layers_per_step > 0 ? std::min(layers_per_step, L) : L;
    const int groups = (L + lps - 1) / lps;
    for (int k = 0; k < groups; ++k) {
        const uint32_t p0 = (uint32_t)(2 * k * lps);
        const uint32_t np = (uint32_t)(2 * (std::min(L, (k + 1) * lps) - k * lps));
        if (ready_events && ready_events[k])
            KVS_CUDA(cudaStreamWaitEvent(s, (cudaEvent_t)ready_events[k], 0));
        if (pl.num_host) {
            const Fp8Job f = fjob(pl.num_device, pl.num_host, p0, np);
            if (f.job.num_pieces >= (1ull << 31) || fp8_segments(f) >= (1ull << 31))
                return fail(KVS_ERR_INVALID_ARG, "call too large: split it");
            // Retrieval: a CTA keeps up to 32 KiB of codes in flight, half a link-kernel
            // CTA's bytes, so it takes twice the link kernel's grid.  Store-back: one CTA
            // per (chunk, plane, head) over the whole GPU for a whole call (193 GB/s, the
            // D2H link); layer by layer it runs beside the compute that produces the KV,
            // where a whole-GPU launch per group displaces that compute, so it takes the
            // host-link store cap (exposed store time per 8B prefill: 7.7 ms uncapped,
            // 2.1 ms at 32 CTAs).
            // KVS_F_FEW_SMS: the staged kernel on the BF16 staged kernel's cap (each of its
            // CTAs holds 112 KiB of codes, about what a BF16 staged CTA holds).
            const int grid = cap ? cap : few ? st.few_sm_ctas : retrieve ? 2 * st.hostlink_ctas
                           : layers_per_step > 0 ? st.store_ctas : 0;
            rc = run(f, grid, false);
            if (rc) return rc;
        }
        if (pl.num_device) {
            const Fp8Job f = fjob(0, pl.num_device, p0, np);
            if (f.job.num_pieces >= (1ull << 31) || fp8_segments(f) >= (1ull << 31))
                return fail(KVS_ERR_INVALID_ARG, "call too large: split it");
            // HBM chunks: uncapped retrievals run one CTA per piece, store-backs stage
            // heads through shared memory
            rc = run(f, cap ? cap : (retrieve ? kFp8PerPiece : 0), true);
            if (rc) return rc;
        }
        if (layers_per_step > 0 && layer_events && layer_events[k])
            KVS_CUDA(cudaEventRecord((cudaEvent_t)layer_events[k], s));
    }
    if (flags & KVS_F_VALIDATE) {
        KVS_CUDA(cudaEventRecord(u.slot->done, s));
        u.slot->used = true;
        guard.slot = nullptr;
        return read_error_word(st, s);
    }
    return KVS_OK;
}

// ---------------------------------------------------------------------------
// Bandwidth probes
// ---------------------------------------------------------------------------
template <class F>
int time_best(cudaStream_t s, int reps, double* best_ms, F&& body) {
    cudaEvent_t a, b;
    KVS_CUDA(cudaEventCreate(&a));
    KVS_CUDA(cudaEventCreate(&b));
    *best_ms = 1e30;
    for (int r = 0; r < reps + 1; ++r) {                 // first run warms up
        KVS_CUDA(cudaEventRecord(a, s));
        int rc = body();
        if (rc) { cudaEventDestroy(a); cudaEventDestroy(b); return rc; }
        KVS_CUDA(cudaEventRecord(b, s));
        KVS_CUDA(cudaEventSynchronize(b));
        float ms = 0;
        KVS_CUDA(cudaEventElapsedTime(&ms, a, b));
        if (r > 0) *best_ms = std::min(*best_ms, (double)ms);
    }
    cudaEventDestroy(a);
    cudaEventDestroy(b);
    return KVS_OK;
}

int query_bw(DevState& st, kvs_bw_report* out, cudaStream_t s, int64_t probe_bytes) {
    if (probe_bytes <= 0) probe_bytes = 1ll << 30;
    probe_bytes = std::max<int64_t>(probe_bytes & ~((int64_t)(8 << 20) - 1), 16 << 20);
    const uint64_t n = (uint64_t)probe_bytes;
    kvs_bw_report rep{};
    rep.num_sms = st.sms;
    rep.probe_bytes = probe_bytes;
    st.hostlink_ctas = st.store_ctas = 0;          // variant probes below use the whole GPU
    uint8_t *d0 = nullptr, *d1 = nullptr, *h = nullptr;
    auto cleanup = [&]() {
        if (d0) cudaFree(d0);
        if (d1) cudaFree(d1);
        if (h) cudaFreeHost(h);
    };
    if (cudaMalloc(&d0, n) != cudaSuccess || cudaMalloc(&d1, n) != cudaSuccess ||
        cudaHostAlloc(&h, n, cudaHostAllocDefault) != cudaSuccess) {
        cudaGetLastError();
        cleanup();
        return fail(KVS_ERR_NOMEM, "cannot allocate %lld-byte probe buffers", (long long)probe_bytes);
    }
    int rc = KVS_OK;
    double ms = 0;
    const int reps = 5;
#define PROBE(field, scale, body)                                               \
    do {                                                                        \
        rc = time_best(s, reps, &ms, [&]() -> int { body; return KVS_OK; });    \
        if (rc) { cleanup(); return rc; }                                       \
        rep.field = (scale) * (double)n / (ms * 1e6);                           \
    } while (0)
    KVS_CUDA(cudaMemsetAsync(d0, 1, n, s));
    memset(h, 2, n);
    PROBE(hbm_copy_gbs, 2.0, KVS_CUDA(launch_flat_copy(d1, d0, n, 0, s)); ++g_launches);
    PROBE(h2d_copy_engine_gbs, 1.0, KVS_CUDA(cudaMemcpyAsync(d0, h, n, cudaMemcpyHostToDevice, s)));
    PROBE(d2h_copy_engine_gbs, 1.0, KVS_CUDA(cudaMemcpyAsync(h, d0, n, cudaMemcpyDeviceToHost, s)));
    PROBE(zero_copy_read_gbs, 1.0, KVS_CUDA(launch_flat_copy(d0, h, n, 0, s)); ++g_launches);
    PROBE(zero_copy_write_gbs, 1.0, KVS_CUDA(launch_flat_copy(h, d0, n, 0, s)); ++g_launches);

    // Scatter / gather probes on an 8B-like geometry: 8 layers, 8 KV heads,
    // head_dim 128, bf16, B = 16, C = 256 (8 MiB chunks), random block table.
    kvs_geometry g{8, 8, 128, 2, 16, 256};
    const uint64_t chunk_bytes = 2ull * g.num_layers * g.chunk_tokens * g.num_kv_heads * g.head_dim * g.elem_bytes;
    const int nchunks = (int)(n / chunk_bytes);
    const int64_t tokens = (int64_t)nchunks * g.chunk_tokens;
    const int64_t nblocks = tokens / g.block_size;
    const uint64_t plane_bytes = (uint64_t)nblocks * g.block_size * g.num_kv_heads * g.head_dim * g.elem_bytes;
    std::vector<void*> planes(2 * g.num_layers);
    for (int p = 0; p < 2 * g.num_layers; ++p) planes[p] = d1 + (uint64_t)p * plane_bytes;
    std::vector<int32_t> table(nblocks);
    for (int64_t k = 0; k < nblocks; ++k) table[k] = (int32_t)k;
    uint64_t x = 0x9E3779B97F4A7C15ull;                          // fixed shuffle (xorshift)
    for (int64_t k = nblocks - 1; k > 0; --k) {
        x ^= x << 13; x ^= x >> 7; x ^= x << 17;
        std::swap(table[k], table[(int64_t)(x % (uint64_t)(k + 1))]);
    }
    kvs_paged_cache cache{planes.data(), nblocks};
    std::vector<kvs_chunk> hc(nchunks), dc(nchunks);
    for (int c = 0; c < nchunks; ++c) {
        hc[c] = {h + (uint64_t)c * chunk_bytes, g.chunk_tokens, KVS_SRC_HOST_PINNED};
        dc[c] = {d0 + (uint64_t)c * chunk_bytes, g.chunk_tokens, KVS_SRC_DEVICE};
    }
    kvs_request rh{0, tokens, hc.data(), nchunks, (int32_t)nblocks, table.data()};
    kvs_request rd{0, tokens, dc.data(), nchunks, (int32_t)nblocks, table.data()};
    const uint64_t moved = (uint64_t)tokens * chunk_bytes / g.chunk_tokens;
    auto probe_call = [&](const kvs_request* r, bool retrieve, uint32_t fl, double* field) -> int {
        double best = 0;
        int rc2 = time_best(s, reps, &best, [&]() -> int {
            return copy_call(&g, &cache, r, 1, (void*)s, fl, retrieve);
        });
        if (rc2) return rc2;
        *field = (double)moved / (best * 1e6);
        return KVS_OK;
    };
    if ((rc = probe_call(&rh, true, KVS_F_FORCE_HOSTLINK, &rep.retrieve_gbs[0])) ||
        (rc = probe_call(&rh, true, KVS_F_FORCE_HBMCOPY, &rep.retrieve_gbs[1])) ||
        (rc = probe_call(&rh, true, KVS_F_FORCE_DMA, &rep.retrieve_dma_gbs)) ||
        (rc = probe_call(&rh, false, KVS_F_FORCE_HOSTLINK, &rep.store_gbs[0])) ||
        (rc = probe_call(&rh, false, KVS_F_FORCE_HBMCOPY, &rep.store_gbs[1])) ||
        (rc = probe_call(&rh, false, KVS_F_FORCE_DMA, &rep.store_dma_gbs)) ||
        (rc = probe_call(&rd, true, KVS_F_FORCE_LDG, &rep.device_kernel_gbs[0])) ||
        (rc = probe_call(&rd, true, KVS_F_FORCE_TMA, &rep.device_kernel_gbs[1]))) {
        cleanup();
        return rc;
    }
    // Host-link grid cap: four times the smallest grid within 1% of the best
    // rate on an idle GPU.  A grid that fills every SM buys nothing once the
    // link is saturated and starves kernels on other streams; the margin covers
    // the longer load latency when other kernels load the GPU (measured beside
    // a bf16 GEMM loop, the idle minimum keeps under half of the link).
    {
        const int full = st.sms * link_ctas_per_sm();
        const int cand[] = {8, 12, 16, 24, 32, 48, 64, 96, 128, full};
        constexpr int ncand = 10;
        double gb[2][ncand] = {};
        for (int dir = 0; dir < 2; ++dir) {
            double best = 0;
            for (int k = 0; k < ncand; ++k) {
                rc = probe_call(&rh, dir == 0, KVS_F_FORCE_HOSTLINK | KVS_F_MAX_CTAS(cand[k]), &gb[dir][k]);
                if (rc) { cleanup(); return rc; }
                best = std::max(best, gb[dir][k]);
            }
            int pick = 0;
            for (int k = 0; k < ncand; ++k)
                if (gb[dir][k] >= 0.99 * best) { pick = cand[k]; break; }
            pick *= 4;
            if (pick >= full) pick = 0;
            if (dir == 0) rep.hostlink_ctas = pick; else rep.store_ctas = pick;
        }
    }
    // KVS_F_FEW_SMS cap: 1.25 x the smallest grid within 3% of the staged
    // kernel's best rate on an idle GPU.  Beside a bf16 GEMM loop that keeps the
    // link at 96-98% on 8-10 SMs, where the plain kernel needs 16 or more.
    {
        const int cand[] = {8, 12, 16, 20, 24, 32};
        double gb[6] = {}, best = 0;
        for (int k = 0; k < 6; ++k) {
            rc = probe_call(&rh, true, KVS_F_FEW_SMS | KVS_F_MAX_CTAS(cand[k]), &gb[k]);
            if (rc) { cleanup(); return rc; }
            best = std::max(best, gb[k]);
        }
        int pick = cand[5];
        for (int k = 0; k < 6; ++k)
            if (gb[k] >= 0.97 * best) { pick = cand[k]; break; }
        rep.few_sm_ctas = (pick * 5 / 4 + 1) & ~1;
        rep.few_sm_gbs = best;
    }
#undef PROBE
    KVS_CUDA(cudaStreamSynchronize(s));
    cleanup();
    st.hostlink_ctas = rep.hostlink_ctas;
    st.store_ctas = rep.store_ctas;
    st.few_sm_ctas = rep.few_sm_ctas;
    // The probe's buffer is small.  On GB300 the copy engine's rate from pinned
    // host memory is erratic on buffers of tens of GiB (13-210 GB/s on 40 GiB,
    // by box and allocation), where SM loads keep the link's rate, so the
    // copy-engine variant is taken only when it wins the probe clearly.
    // The same holds for the DMA variant (the copy engine again).  kvs_tune
    // measures the caller's own call instead.
    constexpr double kHbmcopyMargin = 1.05;
    auto pick = [&](double hostlink, double hbmcopy, double dma) {
        int v = KVS_VARIANT_HOSTLINK;
        double best = hostlink;
        if (hbmcopy > kHbmcopyMargin * hostlink && hbmcopy > best) { v = KVS_VARIANT_HBMCOPY; best = hbmcopy; }
        if (dma > kHbmcopyMargin * hostlink && dma > best) v = KVS_VARIANT_DMA;
        return v;
    };
    st.retrieve_host = pick(rep.retrieve_gbs[0], rep.retrieve_gbs[1], rep.retrieve_dma_gbs);
    st.store_host = pick(rep.store_gbs[0], rep.store_gbs[1], rep.store_dma_gbs);
    st.kernel_device = rep.device_kernel_gbs[1] > rep.device_kernel_gbs[0] ? KVS_KERNEL_TMA : KVS_KERNEL_LDG;
    rep.chosen_retrieve_host = st.retrieve_host;
    rep.chosen_store_host = st.store_host;
    rep.chosen_kernel_device = st.kernel_device;
    st.report = rep;
    if (out) *out = rep;
    return KVS_OK;
}

int tune(DevState& st, const kvs_geometry* g, const kvs_paged_cache* cache, const kvs_request* reqs,
         int32_t nreq, cudaStream_t s, uint32_t flags, int32_t direction, int32_t reps, kvs_tune_report* out) {
    if (direction != KVS_DIR_RETRIEVE && direction != KVS_DIR_STORE)
        return fail(KVS_ERR_INVALID_ARG, "direction must be KVS_DIR_RETRIEVE or KVS_DIR_STORE");
    if (reps < 1 || reps > 1000) return fail(KVS_ERR_INVALID_ARG, "reps must be in [1, 1000]");
    const bool retrieve = direction == KVS_DIR_RETRIEVE;
    Plan pl;
    int rc = validate_call(g, cache, reqs, nreq, pl);
    if (rc) return rc;
    kvs_tune_report rep{};
    rep.direction = direction;
    int64_t host_bytes = 0;
    for (int32_t r = 0; r < nreq; ++r)
        for (int32_t j = 0; j < reqs[r].num_chunks; ++j)
            if (reqs[r].chunks[j].residency == KVS_SRC_HOST_PINNED)
                host_bytes += (int64_t)2 * g->num_layers * reqs[r].chunks[j].num_tokens * (int64_t)pl.row_bytes;
    rep.host_bytes = host_bytes;
    rep.chosen = retrieve ? st.retrieve_host : st.store_host;
    rep.chosen_kernel_device = st.kernel_device;
    const uint32_t cap = flags & 0xFFFF0000u, base = flags & ~0xFFFF0000u;
    auto timed = [&](const kvs_request* rq, int32_t n, uint32_t fl, int64_t bytes, double* gbs) -> int {
        int rc2 = copy_call(g, cache, rq, n, (void*)s, base | fl, retrieve);      // untimed (validated if asked)
        if (rc2) return rc2;
        double best = 0;
        rc2 = time_best(s, reps, &best, [&]() -> int {
            return copy_call(g, cache, rq, n, (void*)s, (base & ~KVS_F_VALIDATE) | fl, retrieve);
        });
        if (rc2) return rc2;
        *gbs = (double)bytes / (best * 1e6);
        return KVS_OK;
    };
    if (host_bytes > 0) {
        const bool dma_ok = dma_pitch(st, pl, (uint64_t)g->block_size * pl.row_bytes) != 0;
        const uint32_t cand[3] = {KVS_F_FORCE_HOSTLINK | cap, KVS_F_FORCE_HBMCOPY, KVS_F_FORCE_DMA};
        for (int v = 0; v < 3; ++v) {
            if (v == 2 && !dma_ok) continue;
            rc = timed(reqs, nreq, cand[v], host_bytes, &rep.gbs[v]);
            if (rc) return rc;
        }
        int v = 0;
        for (int k = 1; k < 3; ++k)
            if (rep.gbs[k] > rep.gbs[v]) v = k;
        const int chosen = v == 0 ? KVS_VARIANT_HOSTLINK : v == 1 ? KVS_VARIANT_HBMCOPY : KVS_VARIANT_DMA;
        if (retrieve) {
            st.retrieve_host = chosen;
            if (chosen == KVS_VARIANT_HOSTLINK && cap) st.hostlink_ctas = (int)KVS_F_GET_MAX_CTAS(flags);
        } else {
            st.store_host = chosen;
            if (chosen == KVS_VARIANT_HOSTLINK && cap) st.store_ctas = (int)KVS_F_GET_MAX_CTAS(flags);
        }
        rep.chosen = chosen;
    }
    // Device-resident chunks: the LDG and TMA kernels on those chunks alone.  Each
    // becomes a one-chunk request starting at its own first token (a multiple of
    // chunk_tokens: every chunk before it is full), with the request's block table.
    std::vector<kvs_chunk> dch;
    std::vector<kvs_request> dreq;
    int64_t device_bytes = 0;
    for (int32_t r = 0; r < nreq; ++r)
        for (int32_t j = 0; j < reqs[r].num_chunks; ++j)
            if (reqs[r].chunks[j].residency == KVS_SRC_DEVICE) dch.push_back(reqs[r].chunks[j]);
    dreq.reserve(dch.size());
    for (int32_t r = 0, k = 0; r < nreq; ++r) {
        int64_t s0 = reqs[r].first_token;
        for (int32_t j = 0; j < reqs[r].num_chunks; ++j) {
            const kvs_chunk& c = reqs[r].chunks[j];
            if (c.residency == KVS_SRC_DEVICE) {
                dreq.push_back({s0, c.num_tokens, &dch[k++], 1, reqs[r].block_table_len, reqs[r].block_table});
                device_bytes += (int64_t)2 * g->num_layers * c.num_tokens * (int64_t)pl.row_bytes;
            }
            s0 += c.num_tokens;
        }
    }
    rep.device_bytes = device_bytes;
    if (device_bytes > 0) {
        rc = timed(dreq.data(), (int32_t)dreq.size(), KVS_F_FORCE_LDG, device_bytes, &rep.device_gbs[0]);
        if (rc) return rc;
        if (vec_bytes_for(pl.addr_or) == 16) {      // TMA needs 16-byte aligned planes and rows
            rc = timed(dreq.data(), (int32_t)dreq.size(), KVS_F_FORCE_TMA, device_bytes, &rep.device_gbs[1]);
            if (rc == KVS_ERR_UNSUPPORTED) { rep.device_gbs[1] = 0; rc = KVS_OK; t_error.clear(); }
            if (rc) return rc;
        }
        st.kernel_device = rep.device_gbs[1] > rep.device_gbs[0] ? KVS_KERNEL_TMA : KVS_KERNEL_LDG;
        rep.chosen_kernel_device = st.kernel_device;
    }
    KVS_CUDA(cudaStreamSynchronize(s));
    if (out) *out = rep;
    return KVS_OK;
}

}  // namespace

void set_last_error(const char* msg) { t_error = msg; }

int hostlink_grid(bool retrieve) {
    std::lock_guard<std::mutex> lk(g_mu);
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    if (dev < (int)g_dev.size() && g_dev[dev].ready)
        return retrieve ? g_dev[dev].hostlink_ctas : g_dev[dev].store_ctas;
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return std::max(8, sms / 3);          // the built-in default of get_state
}

}  // namespace kvs

using namespace kvs;

extern "C" {

int kvs_retrieve(const kvs_geometry* geom, const kvs_paged_cache* cache, const kvs_request* requests,
                 int32_t num_requests, void* cuda_stream, uint32_t flags) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    return copy_call(geom, cache, requests, num_requests, cuda_stream, flags, true);
}

int kvs_store(const kvs_geometry* geom, const kvs_paged_cache* cache, const kvs_request* requests,
              int32_t num_requests, void* cuda_stream, uint32_t flags) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    return copy_call(geom, cache, requests, num_requests, cuda_stream, flags, false);
}

int kvs_retrieve_fp8(const kvs_geometry* geom, const kvs_paged_cache* cache, const kvs_request* requests,
                     int32_t num_requests, void* cuda_stream, uint32_t flags) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    return fp8_call(geom, cache, requests, num_requests, cuda_stream, flags, true);
}

int kvs_store_fp8(const kvs_geometry* geom, const kvs_paged_cache* cache, const kvs_request* requests,
                  int32_t num_requests, void* cuda_stream, uint32_t flags) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    return fp8_call(geom, cache, requests, num_requests, cuda_stream, flags, false);
}

int kvs_retrieve_fp8_layers(const kvs_geometry* geom, const kvs_paged_cache* cache, const kvs_request* requests,
                            int32_t num_requests, int32_t layers_per_step, void* const* layer_events,
                            void* cuda_stream, uint32_t flags) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    if (layers_per_step <= 0) return fail(KVS_ERR_INVALID_ARG, "layers_per_step must be positive");
    return fp8_call(geom, cache, requests, num_requests, cuda_stream, flags, true, layers_per_step, layer_events);
}

int kvs_store_fp8_layers(const kvs_geometry* geom, const kvs_paged_cache* cache, const kvs_request* requests,
                         int32_t num_requests, int32_t layers_per_step, void* const* ready_events,
                         void* const* layer_events, void* cuda_stream, uint32_t flags) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    if (layers_per_step <= 0) return fail(KVS_ERR_INVALID_ARG, "layers_per_step must be positive");
    return fp8_call(geom, cache, requests, num_requests, cuda_stream, flags, false, layers_per_step, layer_events,
                    ready_events);
}

int kvs_retrieve_layers(const kvs_geometry* geom, const kvs_paged_cache* cache, const kvs_request* requests,
                        int32_t num_requests, int32_t layers_per_step, void* const* layer_events,
                        void* cuda_stream, uint32_t flags) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    if (layers_per_step <= 0) return fail(KVS_ERR_INVALID_ARG, "layers_per_step must be positive");
    return copy_call(geom, cache, requests, num_requests, cuda_stream, flags, true, layers_per_step, layer_events);
}

int kvs_store_layers(const kvs_geometry* geom, const kvs_paged_cache* cache, const kvs_request* requests,
                     int32_t num_requests, int32_t layers_per_step, void* const* ready_events,
                     void* const* layer_events, void* cuda_stream, uint32_t flags) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    if (layers_per_step <= 0) return fail(KVS_ERR_INVALID_ARG, "layers_per_step must be positive");
    return copy_call(geom, cache, requests, num_requests, cuda_stream, flags, false, layers_per_step, layer_events,
                     ready_events);
}

int kvs_query_bw(kvs_bw_report* out, void* cuda_stream, int64_t probe_bytes) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    DevState* st = nullptr;
    int rc = get_state(&st);
    if (rc) return rc;
    return query_bw(*st, out, (cudaStream_t)cuda_stream, probe_bytes);
}

int kvs_tune(const kvs_geometry* geom, const kvs_paged_cache* cache, const kvs_request* requests,
             int32_t num_requests, void* cuda_stream, uint32_t flags, int32_t direction, int32_t reps,
             kvs_tune_report* out) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    if (direction != KVS_DIR_RETRIEVE && direction != KVS_DIR_STORE)
        return fail(KVS_ERR_INVALID_ARG, "direction must be KVS_DIR_RETRIEVE or KVS_DIR_STORE");
    if (reps < 1 || reps > 1000) return fail(KVS_ERR_INVALID_ARG, "reps must be in [1, 1000]");
    // kernel choices that kvs_tune's candidates would not carry: refused rather than ignored
    const uint32_t forced = KVS_F_FORCE_HOSTLINK | KVS_F_FORCE_HBMCOPY | KVS_F_FORCE_DMA | KVS_F_FORCE_LDG |
                            KVS_F_FORCE_TMA | KVS_F_LAYER_LAUNCHES | KVS_F_LAYER_SIGNAL | KVS_F_FEW_SMS |
                            KVS_F_PREFETCH_L2;
    if (flags & forced)
        return fail(KVS_ERR_INVALID_ARG, "kvs_tune chooses the variant: no FORCE, layer, KVS_F_FEW_SMS or "
                    "KVS_F_PREFETCH_L2 flags");
    Plan pl;
    int rc = validate_call(geom, cache, requests, num_requests, pl);      // before any device state
    if (rc) return rc;
    DevState* st = nullptr;
    rc = get_state(&st);
    if (rc) return rc;
    return tune(*st, geom, cache, requests, num_requests, (cudaStream_t)cuda_stream, flags, direction, reps, out);
}

int kvs_get_choice(kvs_bw_report* out) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    if (!out) return fail(KVS_ERR_INVALID_ARG, "out is NULL");
    DevState* st = nullptr;
    int rc = get_state(&st);
    if (rc) return rc;
    *out = st->report;
    out->chosen_retrieve_host = st->retrieve_host;
    out->chosen_store_host = st->store_host;
    out->chosen_kernel_device = st->kernel_device;
    out->num_sms = st->sms;
    out->hostlink_ctas = st->hostlink_ctas;
    out->store_ctas = st->store_ctas;
    out->few_sm_ctas = st->few_sm_ctas;
    return KVS_OK;
}

int kvs_check_errors(void* cuda_stream) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    DevState* st = nullptr;
    int rc = get_state(&st);
    if (rc) return rc;
    return read_error_word(*st, (cudaStream_t)cuda_stream);
}

int kvs_enqueue_error_read(void* cuda_stream, int32_t* host_word) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    if (!host_word) return fail(KVS_ERR_INVALID_ARG, "host_word is NULL");
    DevState* st = nullptr;
    int rc = get_state(&st);
    if (rc) return rc;
    const cudaStream_t s = (cudaStream_t)cuda_stream;
    KVS_CUDA(cudaMemcpyAsync(host_word, st->err, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
    KVS_CUDA(cudaMemsetAsync(st->err, 0, sizeof(int32_t), s));
    return KVS_OK;
}

const char* kvs_last_error(void) { return t_error.c_str(); }

int kvs_shutdown(void) {
    // The allocation-free entry point takes its own lock and then this one (for
    // the host-link cap), so its address is forgotten after this lock is released.
    {
        std::lock_guard<std::mutex> lk(g_mu);
        int prev = 0;
        cudaGetDevice(&prev);
        for (auto& st : g_dev) {
            if (!st.ready) continue;
            cudaSetDevice(st.device);
            cudaDeviceSynchronize();
            for (auto& sl : st.up) {
                if (sl.host) cudaFreeHost(sl.host);
                if (sl.dev) cudaFree(sl.dev);
                if (sl.done) cudaEventDestroy(sl.done);
                if (sl.uploaded) cudaEventDestroy(sl.uploaded);
            }
            if (st.upload_stream) cudaStreamDestroy(st.upload_stream);
            for (int k = 0; k < kRingSlots; ++k) {
                cudaEventDestroy(st.ring_filled[k]);
                cudaEventDestroy(st.ring_free[k]);
            }
            cudaEventDestroy(st.ev_fork);
            cudaEventDestroy(st.ev_join);
            cudaEventDestroy(st.ev_aux_fork);
            cudaEventDestroy(st.ev_aux_join);
            if (st.aux_stream) cudaStreamDestroy(st.aux_stream);
            for (auto& sg : st.sig) {
                if (sg.mem) cudaFree(sg.mem);
                if (sg.done) cudaEventDestroy(sg.done);
            }
            if (st.signal_stream) cudaStreamDestroy(st.signal_stream);
            if (st.ring) cudaFree(st.ring);
            if (st.copy_stream) cudaStreamDestroy(st.copy_stream);
            if (st.err) cudaFree(st.err);
            if (st.err_host) cudaFreeHost(st.err_host);
            st = DevState{};
    }
    g_dev.clear();
    cudaSetDevice(prev);
    }
    noalloc_forget_devices();
    return KVS_OK;
}

int kvs_version(void) { return KVS_VERSION; }

int64_t kvs_stat_launches(void) {
    std::lock_guard<std::mutex> lk(g_mu);
    return g_launches;
}

int kvs_selftest_wait_timeout(void* cuda_stream, int64_t limit_ns) {
    std::lock_guard<std::mutex> lk(g_mu);
    t_error.clear();
    if (limit_ns <= 0 || limit_ns > 2000000000ll)
        return fail(KVS_ERR_INVALID_ARG, "limit_ns must be in (0, 2e9]");
    DevState* st = nullptr;
    int rc = get_state(&st);
    if (rc) return rc;
    cudaStream_t s = (cudaStream_t)cuda_stream;
    KVS_CUDA(launch_stall(st->err, (uint64_t)limit_ns, s));
    ++g_launches;
    return read_error_word(*st, s);
}

}  // extern "C"

// runtime.cu — host side of libkvg: the C ABI declared in include/kvg.h.
//
// Owns stores (serialized blocks in HBM or pinned-host slabs), caches (page
// pool, device page tables, host mirror of the free list and of each
// sequence's pages), per-object scratch (leaf digests, split-K partials) and
// device status words.  Every call validates its arguments on the host before
// it enqueues anything, then plans launches for the kernels in
// copy_kernels.cu, sha256_kernels.cu and attn_kernels.cu.
#include <algorithm>
#include <atomic>
#include <cerrno>
#include <cstdarg>
#include <chrono>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <deque>
#include <mutex>
#include <string>
#include <unordered_map>
#include <thread>
#include <vector>

#include <fcntl.h>
#include <sys/stat.h>
#include <unistd.h>

#include <nvtx3/nvToolsExt.h>

#include "common.cuh"

using namespace kvg;

namespace {
// NVTX range around each ABI call, so a profiler's timeline names the
// library call that enqueued each kernel.
struct Trace {
    explicit Trace(const char *name) { nvtxRangePushA(name); }
    ~Trace() { nvtxRangePop(); }
};
}  // namespace

namespace kvg {
static std::atomic<uint64_t> g_launches{0};
void count_launches(uint64_t n) { g_launches.fetch_add(n, std::memory_order_relaxed); }
uint64_t launch_count() { return g_launches.load(std::memory_order_relaxed); }
int env_knob(const char *name, int fallback) {
    const char *e = getenv(name);
    const int v = e ? atoi(e) : 0;
    return v > 0 ? v : fallback;
}
}  // namespace kvg

namespace {

thread_local std::string g_last_error;

kvg_status fail(kvg_status st, const char *fmt, ...) __attribute__((format(printf, 2, 3)));
kvg_status fail(kvg_status st, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return st;
}

kvg_status cuda_fail(cudaError_t e, const char *where) {
    return fail(KVG_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

#define KVG_CUDA(call)                                      \
    do {                                                    \
        cudaError_t e_ = (call);                            \
        if (e_ != cudaSuccess) return cuda_fail(e_, #call); \
    } while (0)

struct DeviceGuard {
    int prev = -1;
    bool ok = true;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        if (prev != dev) ok = cudaSetDevice(dev) == cudaSuccess;
    }
    ~DeviceGuard() {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

uint64_t round_up(uint64_t x, uint64_t m) { return (x + m - 1) / m * m; }

int sm_count(int dev) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 1;
    return n;
}

int elem_bytes(const kvg_dims &d) { return d.kv_dtype == KVG_KV_E4M3 ? 1 : 2; }

bool dims_valid(const kvg_dims &d) {
    if (d.n_layers <= 0 || d.n_kv_heads <= 0 || d.page_size <= 0) return false;
    if (d.head_dim != 64 && d.head_dim != 128 && d.head_dim != 256) return false;
    if (d.rope_style != KVG_ROPE_HALF && d.rope_style != KVG_ROPE_INTERLEAVED) return false;
    if (d.kv_dtype != KVG_KV_BF16 && d.kv_dtype != KVG_KV_E4M3) return false;
    if (d.kv_dtype == KVG_KV_E4M3 && !(std::isfinite(d.k_scale) && d.k_scale > 0.f && std::isfinite(d.v_scale) &&
                                       d.v_scale > 0.f))
        return false;
    const uint64_t pb = (uint64_t)elem_bytes(d) * d.n_kv_heads * d.page_size * d.head_dim;
    return pb % 16 == 0 && pb <= (1ull << 31);
}

bool same_geometry(const kvg_dims &a, const kvg_dims &b) {
    if (a.kv_dtype != b.kv_dtype) return false;
    if (a.kv_dtype == KVG_KV_E4M3 && (a.k_scale != b.k_scale || a.v_scale != b.v_scale)) return false;
    return a.n_layers == b.n_layers && a.n_kv_heads == b.n_kv_heads && a.head_dim == b.head_dim &&
           a.page_size == b.page_size;
}

uint64_t page_bytes_of(const kvg_dims &d) { return (uint64_t)elem_bytes(d) * d.n_kv_heads * d.page_size * d.head_dim; }

struct BlockLayout {
    int64_t n_tokens, n_pages;
    uint64_t pos_off, dig_off, pages_off, total;
};

BlockLayout layout_for(const kvg_dims &d, int64_t n_tokens) {
    BlockLayout b;
    b.n_tokens = n_tokens;
    b.n_pages = (n_tokens + d.page_size - 1) / d.page_size;
    b.pos_off = 256;
    b.dig_off = round_up(b.pos_off + 4ull * n_tokens, 256);
    b.pages_off = round_up(b.dig_off + (uint64_t)d.n_layers * 2 * b.n_pages * 32, 4096);
    b.total = b.pages_off + (uint64_t)d.n_layers * 2 * b.n_pages * page_bytes_of(d);
    return b;
}

void build_header(uint8_t h[256], const kvg_dims &d, const BlockLayout &b) {
    memset(h, 0, 256);
    memcpy(h, "KVGBLK01", 8);
    uint32_t u32;
    int32_t i32;
    int64_t i64;
    uint64_t u64;
    double f64;
    u32 = 1; memcpy(h + 8, &u32, 4);
    u32 = 256; memcpy(h + 12, &u32, 4);
    i32 = d.n_layers; memcpy(h + 16, &i32, 4);
    i32 = d.n_kv_heads; memcpy(h + 20, &i32, 4);
    i32 = d.head_dim; memcpy(h + 24, &i32, 4);
    i32 = d.page_size; memcpy(h + 28, &i32, 4);
    i64 = b.n_tokens; memcpy(h + 32, &i64, 8);
    i64 = b.n_pages; memcpy(h + 40, &i64, 8);
    f64 = d.rope_theta; memcpy(h + 48, &f64, 8);
    i32 = d.rope_style; memcpy(h + 56, &i32, 4);
    i32 = d.kv_dtype == KVG_KV_E4M3 ? 2 : 1; memcpy(h + 60, &i32, 4);  // block dtype code
    u64 = b.pos_off; memcpy(h + 64, &u64, 8);
    u64 = b.dig_off; memcpy(h + 72, &u64, 8);
    u64 = b.pages_off; memcpy(h + 80, &u64, 8);
    u64 = b.total; memcpy(h + 88, &u64, 8);
    if (d.kv_dtype == KVG_KV_E4M3) {  // per-tensor scales (the digest is written at 96..127 later)
        memcpy(h + 128, &d.k_scale, 4);
        memcpy(h + 132, &d.v_scale, 4);
    }
}

// Chunk of a page that one CTA copies: <= 64 KiB, divides the page, whole rows.
int32_t copy_chunk_bytes(const kvg_dims &d) {
    uint64_t c = page_bytes_of(d);
    const uint64_t row = (uint64_t)elem_bytes(d) * d.head_dim;
    while (c > 65536 && c % 2 == 0 && (c / 2) % row == 0 && (c / 2) % 16 == 0) c /= 2;
    return (int32_t)c;
}

// Growable device scratch.  Growing frees the old buffer (cudaFree waits for
// the device), so work still using it has finished.
struct Scratch {
    void *ptr = nullptr;
    size_t cap = 0;
    cudaError_t ensure(size_t bytes) {
        if (bytes <= cap) return cudaSuccess;
        if (ptr) cudaFree(ptr);
        ptr = nullptr;
        cap = 0;
        size_t want = std::max(bytes, (size_t)1 << 20);
        cudaError_t e = cudaMalloc(&ptr, want);
        if (e != cudaSuccess) return e;
        cap = want;
        return cudaSuccess;
    }
    void release() {
        if (ptr) cudaFree(ptr);
        ptr = nullptr;
        cap = 0;
    }
};

}  // namespace

// ------------------------------------------------------------------- store --

struct kvg_store {
    kvg_dims dims;
    int32_t residency = KVG_RESIDENCY_HBM;
    uint64_t capacity = 0;
    uint64_t reserved_bytes = 0;  // slab bytes allocated so far
    int device = 0;
    int n_sm = 1;
    struct Slab {
        uint8_t *host = nullptr;  // pinned-host slabs
        uint8_t *dev = nullptr;   // device-accessible address
        uint64_t size = 0, used = 0;
    };
    std::vector<Slab> slabs;
    struct Blk {
        uint8_t *dev;   // device-accessible start of the serialized block (pool stores: its metadata)
        uint8_t *host;  // host address (pinned-host store) or nullptr
        BlockLayout lay;
        int64_t min_pos, max_pos;
        std::vector<int32_t> pids;  // pool stores: the block's pages in the cache pool
    };
    std::vector<Blk> blocks;
    Scratch leaf;
    DevStatus *status = nullptr;
    kvg_cache *pool_cache = nullptr;  // KVG_RESIDENCY_CACHE_POOL: the cache holding the pages
    // block-file loads into an HBM store: a pinned bounce slot, a stream and
    // an event per reader thread (allocated by the first load)
    std::vector<uint8_t *> bounce;
    std::vector<cudaStream_t> load_streams;
    std::vector<cudaEvent_t> load_events;
    // deposits: the block digest (one serial SHA-256 chain) runs on its own
    // stream after the page digests; a pinned-host store's blocks are
    // assembled and hashed in an HBM staging buffer, then copied out
    cudaStream_t digest_stream = nullptr;
    cudaEvent_t pages_done = nullptr, stage_free = nullptr;
    bool pages_recorded = false;  // a deposit's page hashing (which uses `leaf`) may still run
    bool stage_used = false;
    Scratch stage;
};

// The store's leaf-digest scratch is shared by deposits (which return before
// their page hashing has run) and verified imports: its next user's stream
// waits for the last deposit's page hashing.
static cudaError_t wait_for_leaf_scratch(kvg_store *s, cudaStream_t st) {
    return s->pages_recorded ? cudaStreamWaitEvent(st, s->pages_done, 0) : cudaSuccess;
}

static kvg_status store_alloc(kvg_store *s, uint64_t bytes, uint8_t **dev, uint8_t **host) {
    for (auto &sl : s->slabs) {
        const uint64_t at = round_up(sl.used, 4096);
        if (at + bytes <= sl.size) {
            *dev = sl.dev + at;
            *host = sl.host ? sl.host + at : nullptr;
            sl.used = at + bytes;
            return KVG_OK;
        }
    }
    const uint64_t slab = std::max<uint64_t>(bytes, 1ull << 30);
    if (s->reserved_bytes + slab > s->capacity) {
        if (s->reserved_bytes + bytes > s->capacity)
            return fail(KVG_ERR_CAPACITY, "store full: %llu of %llu bytes reserved, block needs %llu",
                        (unsigned long long)s->reserved_bytes, (unsigned long long)s->capacity,
                        (unsigned long long)bytes);
    }
    const uint64_t size = std::min<uint64_t>(slab, s->capacity - s->reserved_bytes);
    kvg_store::Slab sl;
    sl.size = size;
    if (s->residency != KVG_RESIDENCY_PINNED_HOST) {
        cudaError_t e = cudaMalloc(&sl.dev, size);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return fail(KVG_ERR_OOM, "cudaMalloc(%llu): %s", (unsigned long long)size, cudaGetErrorString(e));
        }
    } else {
        cudaError_t e = cudaHostAlloc(reinterpret_cast<void **>(&sl.host), size,
                                      cudaHostAllocMapped | cudaHostAllocPortable);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return fail(KVG_ERR_OOM, "cudaHostAlloc(%llu): %s", (unsigned long long)size, cudaGetErrorString(e));
        }
        e = cudaHostGetDevicePointer(reinterpret_cast<void **>(&sl.dev), sl.host, 0);
        if (e != cudaSuccess) {
            cudaFreeHost(sl.host);
            return cuda_fail(e, "cudaHostGetDevicePointer");
        }
    }
    s->reserved_bytes += size;
    sl.used = bytes;
    *dev = sl.dev;
    *host = sl.host;
    s->slabs.push_back(sl);
    return KVG_OK;
}

// Gives back the most recent allocation of its slab (a block that was not
// added after all, e.g. an import whose digests did not verify); any other
// region stays allocated.
static void store_unalloc(kvg_store *s, const uint8_t *dev, uint64_t bytes) {
    for (auto &sl : s->slabs) {
        if (dev >= sl.dev && dev + bytes == sl.dev + sl.used) {
            sl.used = (uint64_t)(dev - sl.dev);
            return;
        }
    }
}

extern "C" kvg_status kvg_store_create(const kvg_dims *dims, int32_t residency, uint64_t capacity_bytes,
                                       int32_t device, kvg_store **out) {
    if (!dims || !out) return fail(KVG_ERR_ARG, "null argument");
    *out = nullptr;
    if (!dims_valid(*dims)) return fail(KVG_ERR_ARG, "unsupported geometry");
    if (residency != KVG_RESIDENCY_HBM && residency != KVG_RESIDENCY_PINNED_HOST)
        return fail(KVG_ERR_ARG, "bad residency %d", residency);
    int ndev = 0;
    KVG_CUDA(cudaGetDeviceCount(&ndev));
    if (device < 0 || device >= ndev) return fail(KVG_ERR_ARG, "bad device %d", device);
    DeviceGuard g(device);
    if (!g.ok) return fail(KVG_ERR_CUDA, "cudaSetDevice(%d) failed", device);
    kvg_store *s = new kvg_store();
    s->dims = *dims;
    s->residency = residency;
    s->capacity = capacity_bytes;
    s->device = device;
    s->n_sm = sm_count(device);
    cudaError_t e = cudaMalloc(&s->status, sizeof(DevStatus));
    if (e != cudaSuccess) {
        delete s;
        return cuda_fail(e, "cudaMalloc(status)");
    }
    cudaMemset(s->status, 0, sizeof(DevStatus));
    *out = s;
    return KVG_OK;
}

static void pool_release_blocks(kvg_store *s);

extern "C" void kvg_store_destroy(kvg_store *s) {
    if (!s) return;
    DeviceGuard g(s->device);
    cudaDeviceSynchronize();
    if (s->pool_cache) pool_release_blocks(s);
    for (auto &sl : s->slabs) {
        if (sl.host)
            cudaFreeHost(sl.host);
        else if (sl.dev)
            cudaFree(sl.dev);
    }
    s->leaf.release();
    if (s->status) cudaFree(s->status);
    for (uint8_t *b : s->bounce) cudaFreeHost(b);
    for (cudaStream_t st : s->load_streams) cudaStreamDestroy(st);
    for (cudaEvent_t e : s->load_events) cudaEventDestroy(e);
    if (s->digest_stream) cudaStreamDestroy(s->digest_stream);
    if (s->pages_done) cudaEventDestroy(s->pages_done);
    if (s->stage_free) cudaEventDestroy(s->stage_free);
    s->stage.release();
    delete s;
}

extern "C" kvg_status kvg_store_block_info(kvg_store *s, uint64_t id, kvg_block_info *out) {
    if (!s || !out) return fail(KVG_ERR_ARG, "null argument");
    if (id >= s->blocks.size()) return fail(KVG_ERR_NOT_FOUND, "no block %llu", (unsigned long long)id);
    DeviceGuard g(s->device);
    const auto &b = s->blocks[id];
    memset(out, 0, sizeof *out);
    out->n_tokens = b.lay.n_tokens;
    out->n_pages = b.lay.n_pages;
    out->residency = s->residency;
    out->bytes = b.host ? (const void *)b.host : (const void *)b.dev;
    out->total_bytes = b.lay.total;
    out->positions_offset = b.lay.pos_off;
    out->digests_offset = b.lay.dig_off;
    out->pages_offset = b.lay.pages_off;
    KVG_CUDA(cudaDeviceSynchronize());
    if (b.host)
        memcpy(out->block_digest, b.host + 96, 32);
    else
        KVG_CUDA(cudaMemcpy(out->block_digest, b.dev + 96, 32, cudaMemcpyDeviceToHost));
    return KVG_OK;
}

extern "C" kvg_status kvg_store_prefetch(kvg_store *s, uint64_t id, void *stream) {
    Trace trace_("kvg_store_prefetch");
    if (!s) return fail(KVG_ERR_ARG, "null store");
    if (id >= s->blocks.size()) return fail(KVG_ERR_NOT_FOUND, "no block %llu", (unsigned long long)id);
    if (s->residency != KVG_RESIDENCY_PINNED_HOST) return KVG_OK;  // HBM and pool blocks need no translations
    const auto &b = s->blocks[id];
    DeviceGuard g(s->device);
    // one load per host page (the system page size, at least 4 KiB): the
    // block starts 4 KiB-aligned in its slab and its size is a multiple of 16
    static const uint32_t stride = (uint32_t)std::max<long>(4096, sysconf(_SC_PAGESIZE));
    KVG_CUDA(launch_touch(b.dev, b.lay.total, stride, s->n_sm, static_cast<cudaStream_t>(stream)));
    return KVG_OK;
}

// Hashes every page of a block (contiguous pages region) and its block digest
// against `expected` digests (nullable: then writes them), on stream st.
static kvg_status hash_block(kvg_store *s, uint8_t *blk_dev, const BlockLayout &lay, bool verify,
                             cudaStream_t st) {
    const kvg_dims &d = s->dims;
    const uint64_t pb = page_bytes_of(d);
    const int64_t m = (int64_t)((pb + kLeafBytes - 1) / kLeafBytes);
    const int64_t n_pages = (int64_t)d.n_layers * 2 * lay.n_pages;
    KVG_CUDA(wait_for_leaf_scratch(s, st));
    KVG_CUDA(s->leaf.ensure((size_t)n_pages * m * 32));
    PageSource src{blk_dev + lay.pages_off, pb, nullptr, 1, 0};
    uint32_t *leaf = static_cast<uint32_t *>(s->leaf.ptr);
    KVG_CUDA(launch_sha256_leaves(src, n_pages, leaf, s->n_sm, st));
    uint8_t *dig = blk_dev + lay.dig_off;
    KVG_CUDA(launch_sha256_pages(leaf, n_pages, m, verify ? nullptr : dig, verify ? dig : nullptr,
                                 s->status, -1, st));
    KVG_CUDA(launch_sha256_serial(blk_dev + lay.pos_off, 4ull * lay.n_tokens, dig,
                                  (uint64_t)n_pages * 32, verify ? nullptr : blk_dev + 96,
                                  verify ? blk_dev + 96 : nullptr, s->status, st));
    return KVG_OK;
}

// Zeroes a serialized block's alignment gaps (after the position tags and
// after the page digests): the layout defines them as zero, and reused
// memory (a staging buffer, a slab freed and allocated again) is not.
static kvg_status zero_block_gaps(uint8_t *base, const BlockLayout &lay, int32_t n_layers, cudaStream_t st) {
    const uint64_t pos_end = lay.pos_off + 4ull * (uint64_t)lay.n_tokens;
    const uint64_t dig_end = lay.dig_off + (uint64_t)n_layers * 2 * (uint64_t)lay.n_pages * 32;
    if (lay.dig_off > pos_end) KVG_CUDA(cudaMemsetAsync(base + pos_end, 0, lay.dig_off - pos_end, st));
    if (lay.pages_off > dig_end) KVG_CUDA(cudaMemsetAsync(base + dig_end, 0, lay.pages_off - dig_end, st));
    return KVG_OK;
}

static void minmax_positions(const int32_t *pos, int64_t n, int64_t *mn, int64_t *mx) {
    int64_t a = INT64_MAX, b = INT64_MIN;
    for (int64_t i = 0; i < n; ++i) {
        a = std::min<int64_t>(a, pos[i]);
        b = std::max<int64_t>(b, pos[i]);
    }
    *mn = n ? a : 0;
    *mx = n ? b : 0;
}

// Pool-resident blocks (KVG_RESIDENCY_CACHE_POOL), defined after kvg_cache.
static kvg_status pool_export(kvg_store *s, uint64_t id, uint8_t *dst);
static kvg_status pool_import(kvg_store *s, const uint8_t *h, const BlockLayout &lay, uint32_t flags,
                              uint64_t *block_id_out);

// Validates a serialized block header against the store's geometry and the
// bytes available (n_bytes), and gives the block's layout.
static kvg_status parse_block_header(const kvg_store *s, const uint8_t *h, uint64_t n_bytes, BlockLayout *out) {
    if (n_bytes < 256 || memcmp(h, "KVGBLK01", 8) != 0) return fail(KVG_ERR_FORMAT, "bad magic");
    uint32_t ver, hb;
    int32_t L, Hkv, D, P, style, dtype;
    int64_t n_tok, n_pg;
    uint64_t po, dof, pgo, tot;
    memcpy(&ver, h + 8, 4);
    memcpy(&hb, h + 12, 4);
    memcpy(&L, h + 16, 4);
    memcpy(&Hkv, h + 20, 4);
    memcpy(&D, h + 24, 4);
    memcpy(&P, h + 28, 4);
    memcpy(&n_tok, h + 32, 8);
    memcpy(&n_pg, h + 40, 8);
    memcpy(&style, h + 56, 4);
    memcpy(&dtype, h + 60, 4);
    memcpy(&po, h + 64, 8);
    memcpy(&dof, h + 72, 8);
    memcpy(&pgo, h + 80, 8);
    memcpy(&tot, h + 88, 8);
    const kvg_dims &d = s->dims;
    if (ver != 1 || hb != 256 || (dtype != 1 && dtype != 2)) return fail(KVG_ERR_FORMAT, "unsupported version/dtype");
    if (L != d.n_layers || Hkv != d.n_kv_heads || D != d.head_dim || P != d.page_size)
        return fail(KVG_ERR_FORMAT, "geometry differs from the store's");
    if (dtype != (d.kv_dtype == KVG_KV_E4M3 ? 2 : 1)) return fail(KVG_ERR_FORMAT, "element type differs from the store's");
    if (dtype == 2) {
        float ks, vs;
        memcpy(&ks, h + 128, 4);
        memcpy(&vs, h + 132, 4);
        if (ks != d.k_scale || vs != d.v_scale) return fail(KVG_ERR_FORMAT, "fp8 scales differ from the store's");
    }
    if (n_tok <= 0 || n_tok > (1ll << 31)) return fail(KVG_ERR_FORMAT, "bad n_tokens");
    const BlockLayout lay = layout_for(d, n_tok);
    if (n_pg != lay.n_pages || po != lay.pos_off || dof != lay.dig_off || pgo != lay.pages_off ||
        tot != lay.total || n_bytes < tot)
        return fail(KVG_ERR_FORMAT, "layout fields inconsistent");
    *out = lay;
    return KVG_OK;
}

// After the block's bytes are in the store: the optional digest check (a
// block that fails it is not added and its space is given back) and the
// registration.  positions: host copy of the block's position tags.
static kvg_status finish_store_add(kvg_store *s, uint8_t *dev, uint8_t *host, const BlockLayout &lay,
                                   const int32_t *positions, uint32_t flags, uint64_t *block_id_out) {
    if (flags & KVG_GRAFT_VERIFY) {
        KVG_CUDA(cudaMemset(s->status, 0, sizeof(DevStatus)));
        kvg_status st = hash_block(s, dev, lay, true, 0);
        if (st != KVG_OK) return st;
        KVG_CUDA(cudaDeviceSynchronize());
        DevStatus hs;
        KVG_CUDA(cudaMemcpy(&hs, s->status, sizeof hs, cudaMemcpyDeviceToHost));
        KVG_CUDA(cudaMemset(s->status, 0, sizeof(DevStatus)));
        if (hs.n_mismatch) {
            store_unalloc(s, dev, lay.total);
            return fail(KVG_ERR_DIGEST, "import: %d digest mismatches (block not added)", hs.n_mismatch);
        }
    }
    kvg_store::Blk b{dev, host, lay, 0, 0};
    minmax_positions(positions, lay.n_tokens, &b.min_pos, &b.max_pos);
    s->blocks.push_back(b);
    *block_id_out = s->blocks.size() - 1;
    return KVG_OK;
}

extern "C" kvg_status kvg_store_import(kvg_store *s, const void *bytes, uint64_t n_bytes, uint32_t flags,
                                       uint64_t *block_id_out) {
    Trace trace_("kvg_store_import");
    if (!s || !bytes || !block_id_out) return fail(KVG_ERR_ARG, "null argument");
    const uint8_t *h = static_cast<const uint8_t *>(bytes);
    BlockLayout lay;
    kvg_status pst = parse_block_header(s, h, n_bytes, &lay);
    if (pst != KVG_OK) return pst;
    DeviceGuard g(s->device);
    if (s->pool_cache) return pool_import(s, h, lay, flags, block_id_out);
    uint8_t *dev = nullptr, *host = nullptr;
    kvg_status st = store_alloc(s, lay.total, &dev, &host);
    if (st != KVG_OK) return st;
    if (host)
        memcpy(host, h, lay.total);
    else
        KVG_CUDA(cudaMemcpy(dev, h, lay.total, cudaMemcpyHostToDevice));
    return finish_store_add(s, dev, host, lay, reinterpret_cast<const int32_t *>(h + lay.pos_off), flags,
                            block_id_out);
}

extern "C" kvg_status kvg_store_export(kvg_store *s, uint64_t id, void *dst, uint64_t dst_bytes) {
    Trace trace_("kvg_store_export");
    if (!s || !dst) return fail(KVG_ERR_ARG, "null argument");
    if (id >= s->blocks.size()) return fail(KVG_ERR_NOT_FOUND, "no block %llu", (unsigned long long)id);
    const auto &b = s->blocks[id];
    if (dst_bytes < b.lay.total) return fail(KVG_ERR_CAPACITY, "destination too small");
    DeviceGuard g(s->device);
    KVG_CUDA(cudaDeviceSynchronize());
    if (s->pool_cache) return pool_export(s, id, static_cast<uint8_t *>(dst));
    if (b.host)
        memcpy(dst, b.host, b.lay.total);
    else
        KVG_CUDA(cudaMemcpy(dst, b.dev, b.lay.total, cudaMemcpyDeviceToHost));
    return KVG_OK;
}

// Block files are read and written in chunks of this size by up to
// kLoadThreads threads.
constexpr uint64_t kLoadChunk = 16ull << 20;
constexpr unsigned kLoadThreads = 8;

static bool pread_full(int fd, uint8_t *dst, uint64_t n, uint64_t off) {
    while (n) {
        const ssize_t r = pread(fd, dst, n, (off_t)off);
        if (r < 0 && errno == EINTR) continue;
        if (r <= 0) return false;
        dst += r;
        off += (uint64_t)r;
        n -= (uint64_t)r;
    }
    return true;
}

static bool pwrite_full(int fd, const uint8_t *src, uint64_t n, uint64_t off) {
    while (n) {
        const ssize_t r = pwrite(fd, src, n, (off_t)off);
        if (r < 0 && errno == EINTR) continue;
        if (r <= 0) return false;
        src += r;
        off += (uint64_t)r;
        n -= (uint64_t)r;
    }
    return true;
}

// One pinned bounce slot (kLoadChunk bytes), stream and event per thread of a
// block-file transfer, kept by the store for later loads and saves.
static kvg_status ensure_bounce(kvg_store *s, int n_thr) {
    while ((int)s->bounce.size() < n_thr) {
        uint8_t *b = nullptr;
        cudaStream_t st = nullptr;
        cudaEvent_t ev = nullptr;
        // the three are kept together or not at all
        if (cudaHostAlloc(reinterpret_cast<void **>(&b), kLoadChunk, cudaHostAllocDefault) != cudaSuccess) {
            cudaGetLastError();
            return fail(KVG_ERR_OOM, "pinned bounce buffer for block-file transfers");
        }
        cudaError_t e = cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
        if (e != cudaSuccess) {
            if (st) cudaStreamDestroy(st);
            cudaFreeHost(b);
            return cuda_fail(e, "stream or event for block-file transfers");
        }
        s->bounce.push_back(b);
        s->load_streams.push_back(st);
        s->load_events.push_back(ev);
    }
    return KVG_OK;
}

static int transfer_threads(uint64_t total) {
    const int64_t n_chunks = (int64_t)((total + kLoadChunk - 1) / kLoadChunk);
    const unsigned hc = std::thread::hardware_concurrency();
    return (int)std::min<int64_t>(std::max<int64_t>(n_chunks, 1), std::max(1u, std::min(hc ? hc : 1u, kLoadThreads)));
}

// Writes bytes [0, total) of a block to the open file with one writer (writes
// to one file do not scale with threads): a pinned-host store's bytes
// directly; an HBM store's through two pinned bounce slots, the next chunk's
// copy to the host running while the current chunk is written.
static kvg_status save_streamed(kvg_store *s, int fd, uint64_t total, const uint8_t *dev, const uint8_t *host) {
    if (host) return pwrite_full(fd, host, total, 0) ? KVG_OK : fail(KVG_ERR_ARG, "short write of a block file");
    const int64_t n_chunks = (int64_t)((total + kLoadChunk - 1) / kLoadChunk);
    kvg_status st = ensure_bounce(s, 2);
    if (st != KVG_OK) return st;
    auto issue = [&](int64_t i) {
        const uint64_t off = (uint64_t)i * kLoadChunk;
        return cudaMemcpyAsync(s->bounce[i & 1], dev + off, std::min<uint64_t>(kLoadChunk, total - off),
                               cudaMemcpyDeviceToHost, s->load_streams[i & 1]);
    };
    KVG_CUDA(issue(0));
    for (int64_t i = 0; i < n_chunks; ++i) {
        if (i + 1 < n_chunks) KVG_CUDA(issue(i + 1));
        KVG_CUDA(cudaStreamSynchronize(s->load_streams[i & 1]));
        const uint64_t off = (uint64_t)i * kLoadChunk;
        if (!pwrite_full(fd, s->bounce[i & 1], std::min<uint64_t>(kLoadChunk, total - off), off)) {
            KVG_CUDA(cudaStreamSynchronize(s->load_streams[(i + 1) & 1]));
            return fail(KVG_ERR_ARG, "short write of a block file");
        }
    }
    return KVG_OK;
}

extern "C" kvg_status kvg_store_save(kvg_store *s, uint64_t id, const char *path) {
    Trace trace_("kvg_store_save");
    if (!s || !path) return fail(KVG_ERR_ARG, "null argument");
    if (id >= s->blocks.size()) return fail(KVG_ERR_NOT_FOUND, "no block %llu", (unsigned long long)id);
    const auto &b = s->blocks[id];
    DeviceGuard g(s->device);
    KVG_CUDA(cudaDeviceSynchronize());  // the deposit's kernels have written the block
    const int fd = open(path, O_WRONLY | O_CREAT | O_TRUNC | O_CLOEXEC, 0644);
    if (fd < 0) return fail(KVG_ERR_ARG, "cannot open %s for writing", path);
    kvg_status st = KVG_OK;
    if (s->pool_cache) {  // pool-resident blocks: gathered into host memory first
        std::vector<uint8_t> buf(b.lay.total);
        st = kvg_store_export(s, id, buf.data(), buf.size());
        if (st == KVG_OK && !pwrite_full(fd, buf.data(), buf.size(), 0)) st = fail(KVG_ERR_ARG, "short write to %s", path);
    } else {
        st = save_streamed(s, fd, b.lay.total, b.dev, b.host);
    }
    if (close(fd) != 0 && st == KVG_OK) st = fail(KVG_ERR_ARG, "short write to %s", path);
    return st;
}

// Reads bytes [0, total) of the open block file into the store's space: a
// pinned-host store receives them directly (reader threads on disjoint
// chunks); an HBM store through one pinned bounce slot per reader thread,
// each chunk's copy to HBM on the thread's stream while the next chunk is
// read.  Every copy has completed when this returns.
static kvg_status stream_file(kvg_store *s, int fd, uint64_t total, uint8_t *dev, uint8_t *host) {
    const int64_t n_chunks = (int64_t)((total + kLoadChunk - 1) / kLoadChunk);
    const int n_thr = transfer_threads(total);
    if (!host) {
        kvg_status st = ensure_bounce(s, n_thr);
        if (st != KVG_OK) return st;
    }
    std::atomic<int> bad{0};  // 1: a read failed, 2: a CUDA call failed
    auto worker = [&](int w) {
        if (!host && cudaSetDevice(s->device) != cudaSuccess) {
            bad = 2;
            return;
        }
        for (int64_t i = w; i < n_chunks && bad.load() == 0; i += n_thr) {
            const uint64_t off = (uint64_t)i * kLoadChunk;
            const uint64_t len = std::min<uint64_t>(kLoadChunk, total - off);
            if (host) {
                if (!pread_full(fd, host + off, len, off)) bad = 1;
                continue;
            }
            // the slot's previous chunk has been copied before it is overwritten
            if (i >= n_thr && cudaEventSynchronize(s->load_events[w]) != cudaSuccess) {
                bad = 2;
                return;
            }
            if (!pread_full(fd, s->bounce[w], len, off)) {
                bad = 1;
                return;
            }
            if (cudaMemcpyAsync(dev + off, s->bounce[w], len, cudaMemcpyHostToDevice, s->load_streams[w]) !=
                    cudaSuccess ||
                cudaEventRecord(s->load_events[w], s->load_streams[w]) != cudaSuccess) {
                bad = 2;
                return;
            }
        }
    };
    std::vector<std::thread> threads;
    for (int w = 1; w < n_thr; ++w) threads.emplace_back(worker, w);
    worker(0);
    for (auto &t : threads) t.join();
    if (!host)
        for (int w = 0; w < n_thr; ++w) KVG_CUDA(cudaStreamSynchronize(s->load_streams[w]));
    if (bad.load() == 1) return fail(KVG_ERR_FORMAT, "block file read failed");
    if (bad.load() == 2) return fail(KVG_ERR_CUDA, "copy of a block-file chunk failed");
    return KVG_OK;
}

extern "C" kvg_status kvg_store_load(kvg_store *s, const char *path, uint32_t flags, uint64_t *block_id_out) {
    Trace trace_("kvg_store_load");
    if (!s || !path || !block_id_out) return fail(KVG_ERR_ARG, "null argument");
    const int fd = open(path, O_RDONLY | O_CLOEXEC);
    if (fd < 0) return fail(KVG_ERR_ARG, "cannot open %s", path);
    struct FdGuard {
        int fd;
        ~FdGuard() { close(fd); }
    } fd_guard{fd};
    struct stat sb;
    if (fstat(fd, &sb) != 0) return fail(KVG_ERR_ARG, "cannot stat %s", path);
    const uint64_t fsize = (uint64_t)sb.st_size;
    uint8_t hdr[256];
    if (fsize < 256 || !pread_full(fd, hdr, 256, 0)) return fail(KVG_ERR_FORMAT, "%s: shorter than a block header", path);
    BlockLayout lay;
    kvg_status st = parse_block_header(s, hdr, fsize, &lay);
    if (st != KVG_OK) return st;
    DeviceGuard g(s->device);
    if (s->pool_cache) {  // the block's pages go to pool pages: read whole, then the pool import
        std::vector<uint8_t> buf(lay.total);
        if (!pread_full(fd, buf.data(), lay.total, 0)) return fail(KVG_ERR_FORMAT, "%s: read failed", path);
        return pool_import(s, buf.data(), lay, flags, block_id_out);
    }
    std::vector<int32_t> pos((size_t)lay.n_tokens);
    if (!pread_full(fd, reinterpret_cast<uint8_t *>(pos.data()), 4ull * lay.n_tokens, lay.pos_off))
        return fail(KVG_ERR_FORMAT, "%s: read failed", path);
    uint8_t *dev = nullptr, *host = nullptr;
    st = store_alloc(s, lay.total, &dev, &host);
    if (st != KVG_OK) return st;
    st = stream_file(s, fd, lay.total, dev, host);
    if (st != KVG_OK) {
        store_unalloc(s, dev, lay.total);
        return st;
    }
    return finish_store_add(s, dev, host, lay, pos.data(), flags, block_id_out);
}

// ------------------------------------------------------------------- cache --

constexpr int kHostVerifyChunks = 16;  // page-range chunks of a verified host-store graft
constexpr int32_t kMaxGraftsPerBatch = 4096;

struct kvg_cache {
    kvg_dims dims;
    int32_t n_pages = 0, max_seqs = 0, max_slots = 0, max_pages = 0;
    int device = 0, n_sm = 1;
    uint64_t page_bytes = 0;
    uint8_t *pool = nullptr;
    int32_t *page_table = nullptr, *page_fill = nullptr, *positions = nullptr;
    DevStatus *status = nullptr;
    std::deque<int32_t> free_list;
    std::vector<std::vector<int32_t>> seq_pages;
    std::vector<std::vector<int32_t>> seq_fill;  // host copy of page_fill for each sequence's pages
    std::vector<int32_t> n_slots;
    std::vector<int32_t> layer_window;  // per layer: 0 = global attention, W > 0 = last W tokens
    Scratch leaf, part_o, part_ml;
    // the split-K partials are shared by every decode of the cache: a decode
    // on another stream than the previous one waits for that one's last
    // kernel (part_ev, recorded after each decode) instead of racing on them
    cudaEvent_t part_ev = nullptr;
    cudaStream_t part_stream = nullptr;
    bool part_used = false;
    CUtensorMap pool_map;  // decode kernel's 2-D view of the pool
    // library stream and events for hashing a host-store graft's pages while
    // the next pages still cross the host link (made on first use)
    cudaStream_t aux = nullptr;
    cudaEvent_t aux_ev[kHostVerifyChunks + 1] = {};
    // kvg_graft_batch's job table: staged in pinned host memory, copied to
    // batch_dev on the call's stream; batch_ev marks when the copy has read it
    Scratch batch_dev;
    uint8_t *batch_host = nullptr;
    size_t batch_host_cap = 0;
    cudaEvent_t batch_ev = nullptr;
    std::vector<uint8_t> pinned;  // per page: owned by a pool-resident store block
    std::vector<int32_t> alias;   // per pinned page: sequences whose page tables point at it
    // cos/sin tables of the deltas grafts have used (cos[D/2] then sin[D/2]),
    // so a batch that re-bases many grafts does not recompute them each call
    std::unordered_map<int64_t, std::vector<float>> rope_memo;
    double rope_memo_theta = 0.0;  // the RoPE base the memo's tables were made with
};

// ---------------------------------------------- store inside a cache pool --

static std::vector<int32_t> take_pages(kvg_cache *c, int64_t n);

extern "C" kvg_status kvg_store_create_in_cache(kvg_cache *c, uint64_t capacity_bytes, kvg_store **out) {
    if (!c || !out) return fail(KVG_ERR_ARG, "null argument");
    *out = nullptr;
    DeviceGuard g(c->device);
    kvg_store *s = new kvg_store();
    s->dims = c->dims;
    s->residency = KVG_RESIDENCY_CACHE_POOL;
    s->capacity = capacity_bytes;
    s->device = c->device;
    s->n_sm = c->n_sm;
    s->pool_cache = c;
    cudaError_t e = cudaMalloc(&s->status, sizeof(DevStatus));
    if (e != cudaSuccess) {
        delete s;
        return cuda_fail(e, "cudaMalloc(status)");
    }
    cudaMemset(s->status, 0, sizeof(DevStatus));
    *out = s;
    return KVG_OK;
}

// Metadata region of a pool-resident block: the serialized layout up to
// pages_off (header, positions, digests), then the block's page ids.
static uint64_t pool_meta_bytes(const BlockLayout &lay) { return lay.pages_off + 4ull * lay.n_pages; }

// Hashes a pool-resident block's pages (digests into its metadata, or
// compared with them when verify) and its block digest.
static kvg_status pool_hash(kvg_store *s, uint8_t *meta, const BlockLayout &lay, bool verify, cudaStream_t st) {
    kvg_cache *c = s->pool_cache;
    const uint64_t pb = c->page_bytes;
    const int64_t m = (int64_t)((pb + kLeafBytes - 1) / kLeafBytes);
    const int64_t n_pages = (int64_t)s->dims.n_layers * 2 * lay.n_pages;
    KVG_CUDA(wait_for_leaf_scratch(s, st));
    KVG_CUDA(s->leaf.ensure((size_t)n_pages * m * 32));
    PageSource src{c->pool, pb, reinterpret_cast<const int32_t *>(meta + lay.pages_off), (int32_t)lay.n_pages,
                   (int64_t)c->n_pages};
    uint32_t *leaf = static_cast<uint32_t *>(s->leaf.ptr);
    KVG_CUDA(launch_sha256_leaves(src, n_pages, leaf, s->n_sm, st));
    uint8_t *dig = meta + lay.dig_off;
    KVG_CUDA(launch_sha256_pages(leaf, n_pages, m, verify ? nullptr : dig, verify ? dig : nullptr, s->status, -1, st));
    KVG_CUDA(launch_sha256_serial(meta + lay.pos_off, 4ull * lay.n_tokens, dig, (uint64_t)n_pages * 32,
                                  verify ? nullptr : meta + 96, verify ? meta + 96 : nullptr, s->status, st));
    return KVG_OK;
}

static kvg_status pool_write_pids(uint8_t *meta, const BlockLayout &lay, const std::vector<int32_t> &pids,
                                  cudaStream_t st) {
    int32_t *dst = reinterpret_cast<int32_t *>(meta + lay.pages_off);
    for (size_t base = 0; base < pids.size(); base += kMaxPagesPerLaunch) {
        IntsParams ip{};
        ip.dst = dst + base;
        ip.vals.n = (int32_t)std::min<size_t>(kMaxPagesPerLaunch, pids.size() - base);
        for (int32_t i = 0; i < ip.vals.n; ++i) ip.vals.pid[i] = pids[base + i];
        KVG_CUDA(launch_write_ints(ip, st));
    }
    return KVG_OK;
}

static void pool_unpin(kvg_cache *c, const std::vector<int32_t> &pids) {
    for (int32_t pid : pids) {
        c->pinned[pid] = 0;
        c->free_list.push_back(pid);
    }
}

// A destroyed pool-resident store gives its pages back unless a sequence
// still points at them (those stay reserved until the cache is destroyed).
static void pool_release_blocks(kvg_store *s) {
    kvg_cache *c = s->pool_cache;
    for (auto &b : s->blocks)
        for (int32_t pid : b.pids)
            if (c->alias[pid] == 0) {
                c->pinned[pid] = 0;
                c->free_list.push_back(pid);
            }
}

static kvg_status pool_export(kvg_store *s, uint64_t id, uint8_t *dst) {
    const auto &b = s->blocks[id];
    kvg_cache *c = s->pool_cache;
    KVG_CUDA(cudaMemcpy(dst, b.dev, b.lay.pages_off, cudaMemcpyDeviceToHost));
    const uint64_t pb = c->page_bytes;
    const int64_t npb = b.lay.n_pages;
    for (int64_t lkv = 0; lkv < (int64_t)s->dims.n_layers * 2; ++lkv)
        for (int64_t j = 0; j < npb; ++j)
            KVG_CUDA(cudaMemcpy(dst + b.lay.pages_off + (uint64_t)(lkv * npb + j) * pb,
                                c->pool + ((uint64_t)lkv * c->n_pages + b.pids[j]) * pb, pb, cudaMemcpyDeviceToHost));
    return KVG_OK;
}

static kvg_status pool_import(kvg_store *s, const uint8_t *h, const BlockLayout &lay, uint32_t flags,
                              uint64_t *block_id_out) {
    kvg_cache *c = s->pool_cache;
    if (lay.n_pages > (int64_t)c->free_list.size()) return fail(KVG_ERR_CAPACITY, "cache pool has too few free pages");
    uint8_t *meta = nullptr, *host = nullptr;
    kvg_status st = store_alloc(s, pool_meta_bytes(lay), &meta, &host);
    if (st != KVG_OK) return st;
    auto pids = take_pages(c, lay.n_pages);
    for (int32_t pid : pids) c->pinned[pid] = 1;
    const uint64_t pb = c->page_bytes;
    KVG_CUDA(cudaMemcpy(meta, h, lay.pages_off, cudaMemcpyHostToDevice));
    KVG_CUDA(cudaMemcpy(meta + lay.pages_off, pids.data(), 4 * pids.size(), cudaMemcpyHostToDevice));
    for (int64_t lkv = 0; lkv < (int64_t)s->dims.n_layers * 2; ++lkv)
        for (int64_t j = 0; j < lay.n_pages; ++j)
            KVG_CUDA(cudaMemcpy(c->pool + ((uint64_t)lkv * c->n_pages + pids[j]) * pb,
                                h + lay.pages_off + (uint64_t)(lkv * lay.n_pages + j) * pb, pb, cudaMemcpyHostToDevice));
    if (flags & KVG_GRAFT_VERIFY) {
        KVG_CUDA(cudaMemset(s->status, 0, sizeof(DevStatus)));
        st = pool_hash(s, meta, lay, true, 0);
        if (st != KVG_OK) return st;
        KVG_CUDA(cudaDeviceSynchronize());
        DevStatus hs;
        KVG_CUDA(cudaMemcpy(&hs, s->status, sizeof hs, cudaMemcpyDeviceToHost));
        KVG_CUDA(cudaMemset(s->status, 0, sizeof(DevStatus)));
        if (hs.n_mismatch) {
            pool_unpin(c, pids);
            store_unalloc(s, meta, pool_meta_bytes(lay));
            return fail(KVG_ERR_DIGEST, "import: %d digest mismatches (block not added)", hs.n_mismatch);
        }
    }
    kvg_store::Blk b{meta, nullptr, lay, 0, 0, pids};
    minmax_positions(reinterpret_cast<const int32_t *>(h + lay.pos_off), lay.n_tokens, &b.min_pos, &b.max_pos);
    s->blocks.push_back(b);
    *block_id_out = s->blocks.size() - 1;
    return KVG_OK;
}

extern "C" kvg_status kvg_cache_create(const kvg_dims *dims, int32_t n_pages, int32_t max_seqs,
                                       int32_t max_slots, int32_t device, kvg_cache **out) {
    if (!dims || !out) return fail(KVG_ERR_ARG, "null argument");
    *out = nullptr;
    if (!dims_valid(*dims)) return fail(KVG_ERR_ARG, "unsupported geometry");
    if (n_pages <= 0 || max_seqs <= 0 || max_slots <= 0) return fail(KVG_ERR_ARG, "bad sizes");
    int ndev = 0;
    KVG_CUDA(cudaGetDeviceCount(&ndev));
    if (device < 0 || device >= ndev) return fail(KVG_ERR_ARG, "bad device %d", device);
    DeviceGuard g(device);
    if (!g.ok) return fail(KVG_ERR_CUDA, "cudaSetDevice(%d) failed", device);
    kvg_cache *c = new kvg_cache();
    c->dims = *dims;
    c->n_pages = n_pages;
    c->max_seqs = max_seqs;
    c->max_slots = max_slots;
    c->max_pages = (max_slots + dims->page_size - 1) / dims->page_size;
    c->device = device;
    c->n_sm = sm_count(device);
    c->page_bytes = page_bytes_of(*dims);
    const uint64_t pool_bytes = (uint64_t)dims->n_layers * 2 * n_pages * c->page_bytes;
    auto cleanup = [&](kvg_status st) {
        kvg_cache_destroy(c);
        return st;
    };
    cudaError_t e = cudaMalloc(&c->pool, pool_bytes);
    if (e != cudaSuccess) {
        cudaGetLastError();
        c->pool = nullptr;
        return cleanup(fail(KVG_ERR_OOM, "pool cudaMalloc(%llu): %s", (unsigned long long)pool_bytes,
                            cudaGetErrorString(e)));
    }
    const size_t tbl = (size_t)max_seqs * c->max_pages * 4;
    const size_t pos = (size_t)max_seqs * max_slots * 4;
    if (cudaMalloc(&c->page_table, tbl) != cudaSuccess || cudaMalloc(&c->page_fill, tbl) != cudaSuccess ||
        cudaMalloc(&c->positions, pos) != cudaSuccess || cudaMalloc(&c->status, sizeof(DevStatus)) != cudaSuccess) {
        cudaGetLastError();
        return cleanup(fail(KVG_ERR_OOM, "cache tables allocation failed"));
    }
    if (cudaMemset(c->page_table, 0xFF, tbl) != cudaSuccess || cudaMemset(c->page_fill, 0, tbl) != cudaSuccess ||
        cudaMemset(c->positions, 0xFF, pos) != cudaSuccess ||
        cudaMemset(c->status, 0, sizeof(DevStatus)) != cudaSuccess)
        return cleanup(fail(KVG_ERR_CUDA, "cache tables init failed"));
    const uint64_t pool_rows = (uint64_t)dims->n_layers * 2 * n_pages * dims->n_kv_heads * dims->page_size;
    if (pool_rows > 0x7fffffffull)
        return cleanup(fail(KVG_ERR_ARG, "pool of %llu rows exceeds the decode kernel's 2^31-row addressing",
                            (unsigned long long)pool_rows));
    if (make_pool_tensor_map(&c->pool_map, c->pool, dims->head_dim, dims->kv_dtype == KVG_KV_E4M3, pool_rows) !=
        cudaSuccess)
        return cleanup(fail(KVG_ERR_CUDA, "tensor map of the pool could not be encoded"));
    // the allocation-free decode's static scratch becomes resident on this
    // device now, while the caller expects allocations, not at its first call
    if (cudaError_t ne = noalloc_prepare_device(device); ne != cudaSuccess)
        return cleanup(fail(KVG_ERR_CUDA, "static decode scratch lookup: %s", cudaGetErrorString(ne)));
    for (int32_t i = 0; i < n_pages; ++i) c->free_list.push_back(i);
    c->pinned.assign(n_pages, 0);
    c->alias.assign(n_pages, 0);
    c->seq_pages.assign(max_seqs, {});
    c->n_slots.assign(max_seqs, 0);
    c->seq_fill.resize(max_seqs);
    c->layer_window.assign(dims->n_layers, 0);
    if (cudaDeviceSynchronize() != cudaSuccess) return cleanup(fail(KVG_ERR_CUDA, "init sync failed"));
    *out = c;
    return KVG_OK;
}

extern "C" void kvg_cache_destroy(kvg_cache *c) {
    if (!c) return;
    DeviceGuard g(c->device);
    cudaDeviceSynchronize();
    for (cudaEvent_t &e : c->aux_ev)
        if (e) cudaEventDestroy(e);
    if (c->aux) cudaStreamDestroy(c->aux);
    if (c->batch_ev) cudaEventDestroy(c->batch_ev);
    if (c->part_ev) cudaEventDestroy(c->part_ev);
    if (c->batch_host) cudaFreeHost(c->batch_host);
    c->batch_dev.release();
    if (c->pool) cudaFree(c->pool);
    if (c->page_table) cudaFree(c->page_table);
    if (c->page_fill) cudaFree(c->page_fill);
    if (c->positions) cudaFree(c->positions);
    if (c->status) cudaFree(c->status);
    c->leaf.release();
    c->part_o.release();
    c->part_ml.release();
    delete c;
}

extern "C" kvg_status kvg_cache_set_free_order(kvg_cache *c, const int32_t *order, int32_t n) {
    if (!c || !order) return fail(KVG_ERR_ARG, "null argument");
    if (n != c->n_pages || (int32_t)c->free_list.size() != c->n_pages)
        return fail(KVG_ERR_ARG, "free order needs every page free and n == n_pages");
    std::vector<char> seen(n, 0);
    for (int32_t i = 0; i < n; ++i) {
        if (order[i] < 0 || order[i] >= n || seen[order[i]]) return fail(KVG_ERR_ARG, "not a permutation");
        seen[order[i]] = 1;
    }
    c->free_list.assign(order, order + n);
    return KVG_OK;
}

extern "C" kvg_status kvg_cache_view_get(const kvg_cache *c, kvg_cache_view *v) {
    if (!c || !v) return fail(KVG_ERR_ARG, "null argument");
    v->pool = c->pool;
    v->page_table = c->page_table;
    v->page_fill = c->page_fill;
    v->positions = c->positions;
    v->pool_bytes = (uint64_t)c->dims.n_layers * 2 * c->n_pages * c->page_bytes;
    v->page_bytes = c->page_bytes;
    v->n_pages = c->n_pages;
    v->max_seqs = c->max_seqs;
    v->max_slots = c->max_slots;
    v->max_pages = c->max_pages;
    return KVG_OK;
}

extern "C" kvg_status kvg_cache_seq_info(const kvg_cache *c, int32_t seq, int32_t *n_slots, int32_t *n_pages) {
    if (!c) return fail(KVG_ERR_ARG, "null argument");
    if (seq < 0 || seq >= c->max_seqs) return fail(KVG_ERR_ARG, "bad seq %d", seq);
    if (n_slots) *n_slots = c->n_slots[seq];
    if (n_pages) *n_pages = (int32_t)c->seq_pages[seq].size();
    return KVG_OK;
}

static std::vector<int32_t> take_pages(kvg_cache *c, int64_t n) {
    std::vector<int32_t> v;
    v.reserve(n);
    for (int64_t i = 0; i < n; ++i) {
        v.push_back(c->free_list.front());
        c->free_list.pop_front();
    }
    return v;
}

// Mirrors on the host the fill counts the kernels write for the pages that
// hold slots [slot_begin, slot_end) of `seq` (rows below the fill are valid).
static void note_fills(kvg_cache *c, int32_t seq, int64_t slot_begin, int64_t slot_end) {
    const int64_t P = c->dims.page_size;
    auto &f = c->seq_fill[seq];
    f.resize(c->seq_pages[seq].size(), 0);
    for (int64_t pg = slot_begin / P; pg * P < slot_end; ++pg) f[pg] = (int32_t)std::min<int64_t>(P, slot_end - pg * P);
}

extern "C" kvg_status kvg_cache_append(kvg_cache *c, int32_t seq, const void *k, const void *v,
                                       const int32_t *positions, int32_t n, void *stream) {
    Trace trace_("kvg_cache_append");
    if (!c) return fail(KVG_ERR_ARG, "null cache");
    if (seq < 0 || seq >= c->max_seqs) return fail(KVG_ERR_ARG, "bad seq %d", seq);
    if (n < 0) return fail(KVG_ERR_ARG, "negative n");
    if (n == 0) return KVG_OK;
    if (!k || !v || !positions) return fail(KVG_ERR_ARG, "null buffer");
    if ((reinterpret_cast<uintptr_t>(k) | reinterpret_cast<uintptr_t>(v)) & 15)
        return fail(KVG_ERR_ARG, "k/v must be 16-byte aligned");
    const int64_t P = c->dims.page_size;
    const int64_t s0 = c->n_slots[seq];
    if (s0 + n > c->max_slots) return fail(KVG_ERR_CAPACITY, "append past max_slots");
    const int64_t have = (int64_t)c->seq_pages[seq].size();
    const int64_t need = (s0 + n + P - 1) / P - have;
    if (need > (int64_t)c->free_list.size()) return fail(KVG_ERR_CAPACITY, "out of free pages");
    DeviceGuard g(c->device);
    auto got = take_pages(c, std::max<int64_t>(need, 0));
    auto &sp = c->seq_pages[seq];
    sp.insert(sp.end(), got.begin(), got.end());
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int64_t rows_per_launch = (int64_t)(kMaxPagesPerLaunch - 1) * P;
    for (int64_t row0 = 0; row0 < n; row0 += rows_per_launch) {
        const int64_t nr = std::min<int64_t>(rows_per_launch, n - row0);
        const int64_t s = s0 + row0;
        AppendParams p{};
        p.k = static_cast<const uint16_t *>(k);
        p.v = static_cast<const uint16_t *>(v);
        p.pos = positions;
        p.pool = c->pool;
        p.pool_pages = c->n_pages;
        p.n_layers = c->dims.n_layers;
        p.n_kv_heads = c->dims.n_kv_heads;
        p.page_size = (int32_t)P;
        p.head_dim = c->dims.head_dim;
        p.n = (int32_t)nr;
        p.row0 = (int32_t)row0;
        p.slot0 = (int32_t)s;
        p.page0 = (int32_t)(s / P);
        p.n_rows_total = n;
        p.pos_row = c->positions + (int64_t)seq * c->max_slots;
        p.table_row = c->page_table + (int64_t)seq * c->max_pages;
        p.fill_row = c->page_fill + (int64_t)seq * c->max_pages;
        const int64_t last = (s + nr - 1) / P;
        p.pids.n = (int32_t)(last - p.page0 + 1);
        for (int32_t i = 0; i < p.pids.n; ++i) p.pids.pid[i] = sp[p.page0 + i];
        // long appends move rows with tensor copies; short ones (a box would
        // mostly carry rows that are not stored) with a warp per row; an fp8
        // cache quantizes each row on the way
        cudaError_t e = cudaErrorNotSupported;
        if (c->dims.kv_dtype == KVG_KV_E4M3) {
            p.k_inv_scale = 1.0f / c->dims.k_scale;
            p.v_inv_scale = 1.0f / c->dims.v_scale;
            e = launch_append_e4m3(p, c->n_sm, st);
        } else {
            if (nr >= append_tma_rows(p.page_size, p.head_dim)) e = launch_append_tma(p, c->status, c->n_sm, st);
            if (e == cudaErrorNotSupported) e = launch_append(p, c->n_sm, st);
        }
        KVG_CUDA(e);
    }
    c->n_slots[seq] = (int32_t)(s0 + n);
    note_fills(c, seq, s0, s0 + n);
    return KVG_OK;
}

extern "C" kvg_status kvg_cache_append_batch(kvg_cache *c, const int32_t *seq_ids, int32_t B, const void *k,
                                             const void *v, const int32_t *positions, void *stream) {
    Trace trace_("kvg_cache_append_batch");
    if (!c || !seq_ids || !k || !v || !positions) return fail(KVG_ERR_ARG, "null argument");
    if (B <= 0 || B > kMaxBatchPerLaunch) return fail(KVG_ERR_ARG, "B must be in [1, %d]", kMaxBatchPerLaunch);
    if ((reinterpret_cast<uintptr_t>(k) | reinterpret_cast<uintptr_t>(v)) & 15)
        return fail(KVG_ERR_ARG, "k/v must be 16-byte aligned");
    const int64_t P = c->dims.page_size;
    std::vector<char> seen(c->max_seqs, 0);
    int64_t need = 0;
    for (int32_t b = 0; b < B; ++b) {
        const int32_t sq = seq_ids[b];
        if (sq < 0 || sq >= c->max_seqs) return fail(KVG_ERR_ARG, "bad seq id %d", sq);
        if (seen[sq]) return fail(KVG_ERR_ARG, "seq id %d repeated", sq);
        seen[sq] = 1;
        if (c->n_slots[sq] + 1 > c->max_slots) return fail(KVG_ERR_CAPACITY, "append past max_slots (seq %d)", sq);
        if (c->n_slots[sq] % P == 0 && (int64_t)c->seq_pages[sq].size() * P <= c->n_slots[sq]) ++need;
    }
    if (need > (int64_t)c->free_list.size()) return fail(KVG_ERR_CAPACITY, "out of free pages");
    DeviceGuard g(c->device);
    AppendBatchParams p{};
    p.k = static_cast<const uint16_t *>(k);
    p.v = static_cast<const uint16_t *>(v);
    p.pos = positions;
    p.pool = c->pool;
    p.pool_pages = c->n_pages;
    p.n_layers = c->dims.n_layers;
    p.n_kv_heads = c->dims.n_kv_heads;
    p.page_size = (int32_t)P;
    p.head_dim = c->dims.head_dim;
    p.B = B;
    p.max_pages = c->max_pages;
    p.max_slots = c->max_slots;
    p.page_table = c->page_table;
    p.page_fill = c->page_fill;
    p.positions = c->positions;
    for (int32_t b = 0; b < B; ++b) {
        const int32_t sq = seq_ids[b];
        const int64_t s = c->n_slots[sq];
        auto &sp = c->seq_pages[sq];
        if ((int64_t)sp.size() * P <= s) {
            sp.push_back(c->free_list.front());
            c->free_list.pop_front();
        }
        p.seq[b] = sq;
        p.pid[b] = sp[s / P];
        p.slot[b] = (int32_t)s;
        c->n_slots[sq] = (int32_t)(s + 1);
        note_fills(c, sq, s, s + 1);
    }
    if (c->dims.kv_dtype == KVG_KV_E4M3) {
        p.k_inv_scale = 1.0f / c->dims.k_scale;
        p.v_inv_scale = 1.0f / c->dims.v_scale;
        KVG_CUDA(launch_append_batch_e4m3(p, c->n_sm, static_cast<cudaStream_t>(stream)));
    } else {
        KVG_CUDA(launch_append_batch(p, c->n_sm, static_cast<cudaStream_t>(stream)));
    }
    return KVG_OK;
}

extern "C" kvg_status kvg_cache_release(kvg_cache *c, int32_t seq, void *stream) {
    Trace trace_("kvg_cache_release");
    if (!c) return fail(KVG_ERR_ARG, "null cache");
    if (seq < 0 || seq >= c->max_seqs) return fail(KVG_ERR_ARG, "bad seq %d", seq);
    DeviceGuard g(c->device);
    for (int32_t pid : c->seq_pages[seq]) {
        if (c->pinned[pid])
            --c->alias[pid];  // a pool-resident block's page: not the sequence's to free
        else
            c->free_list.push_back(pid);
    }
    c->seq_pages[seq].clear();
    c->seq_fill[seq].clear();
    c->n_slots[seq] = 0;
    KVG_CUDA(launch_reset_seq(c->page_table + (int64_t)seq * c->max_pages,
                              c->page_fill + (int64_t)seq * c->max_pages, c->max_pages,
                              c->positions + (int64_t)seq * c->max_slots, c->max_slots,
                              static_cast<cudaStream_t>(stream)));
    return KVG_OK;
}

// ----------------------------------------------------------------- deposit --

// Deposit into a pool-resident store: the rows are copied into pool pages
// that the block owns from then on (taken from the free list for good).
static kvg_status pool_deposit(kvg_store *s, kvg_cache *c, int32_t seq, int32_t slot0, int32_t n,
                               const BlockLayout &lay, cudaStream_t st, uint64_t *block_id_out) {
    if (lay.n_pages > (int64_t)c->free_list.size()) return fail(KVG_ERR_CAPACITY, "cache pool has too few free pages");
    uint8_t *meta = nullptr, *host = nullptr;
    kvg_status stt = store_alloc(s, pool_meta_bytes(lay), &meta, &host);
    if (stt != KVG_OK) return stt;
    auto pids = take_pages(c, lay.n_pages);
    for (int32_t pid : pids) c->pinned[pid] = 1;
    HeaderParams hp;
    hp.dst = meta;
    build_header(hp.bytes, s->dims, lay);
    KVG_CUDA(launch_write_header(hp, st));
    stt = zero_block_gaps(meta, lay, s->dims.n_layers, st);
    if (stt != KVG_OK) return stt;
    const int64_t P = c->dims.page_size;
    const auto &sp = c->seq_pages[seq];
    const int64_t j_first = slot0 / P;
    for (int64_t base = 0; base < lay.n_pages; base += kMaxPagesPerLaunch) {
        GatherParams p{};
        p.pool = c->pool;
        p.dst = c->pool;
        p.page_bytes = c->page_bytes;
        p.pool_pages = c->n_pages;
        p.n_layers = c->dims.n_layers;
        p.npb = (int32_t)std::min<int64_t>(kMaxPagesPerLaunch, lay.n_pages - base);
        p.page_base = (int32_t)base;
        p.block_pages = (int32_t)lay.n_pages;
        p.n_kv_heads = c->dims.n_kv_heads;
        p.page_size = (int32_t)P;
        p.head_dim = c->dims.head_dim;
        p.n_tokens = n;
        p.src_pos = c->positions + (int64_t)seq * c->max_slots + slot0 + base * P;
        p.dst_pos = reinterpret_cast<int32_t *>(meta + lay.pos_off) + base * P;
        p.pids.n = p.npb;
        p.dst_pids.n = p.npb;
        for (int32_t i = 0; i < p.npb; ++i) {
            p.pids.pid[i] = sp[j_first + base + i];
            p.dst_pids.pid[i] = pids[base + i];
        }
        KVG_CUDA(launch_gather(p, s->n_sm, st));
    }
    stt = pool_write_pids(meta, lay, pids, st);
    if (stt != KVG_OK) return stt;
    stt = pool_hash(s, meta, lay, false, st);
    if (stt != KVG_OK) return stt;
    KVG_CUDA(cudaStreamSynchronize(st));
    kvg_store::Blk b{meta, nullptr, lay, 0, 0, pids};
    std::vector<int32_t> pos(n);
    KVG_CUDA(cudaMemcpy(pos.data(), meta + lay.pos_off, 4ull * n, cudaMemcpyDeviceToHost));
    minmax_positions(pos.data(), n, &b.min_pos, &b.max_pos);
    s->blocks.push_back(b);
    *block_id_out = s->blocks.size() - 1;
    return KVG_OK;
}

extern "C" kvg_status kvg_deposit(kvg_store *s, const kvg_cache *cc, int32_t seq, int32_t slot0, int32_t n,
                                  void *stream, uint64_t *block_id_out) {
    Trace trace_("kvg_deposit");
    kvg_cache *c = const_cast<kvg_cache *>(cc);
    if (!s || !c || !block_id_out) return fail(KVG_ERR_ARG, "null argument");
    if (!same_geometry(s->dims, c->dims)) return fail(KVG_ERR_ARG, "store and cache geometry differ");
    if (s->device != c->device) return fail(KVG_ERR_ARG, "store and cache on different devices");
    if (seq < 0 || seq >= c->max_seqs) return fail(KVG_ERR_ARG, "bad seq %d", seq);
    const int64_t P = c->dims.page_size;
    if (n <= 0 || slot0 < 0 || slot0 % P || (int64_t)slot0 + n > c->n_slots[seq])
        return fail(KVG_ERR_ARG, "bad range [%d, %d) of %d slots", slot0, slot0 + n, c->n_slots[seq]);
    DeviceGuard g(s->device);
    const BlockLayout lay = layout_for(s->dims, n);
    if (s->pool_cache) {
        if (s->pool_cache != c) return fail(KVG_ERR_ARG, "a pool-resident store deposits from its own cache");
        return pool_deposit(s, c, seq, slot0, n, lay, static_cast<cudaStream_t>(stream), block_id_out);
    }
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (!s->digest_stream) {
        KVG_CUDA(cudaStreamCreateWithFlags(&s->digest_stream, cudaStreamNonBlocking));
        KVG_CUDA(cudaEventCreateWithFlags(&s->pages_done, cudaEventDisableTiming));
        KVG_CUDA(cudaEventCreateWithFlags(&s->stage_free, cudaEventDisableTiming));
    }
    uint8_t *dev = nullptr, *host = nullptr;
    kvg_status stt = store_alloc(s, lay.total, &dev, &host);
    if (stt != KVG_OK) return stt;
    // where the block is assembled and hashed: in place in an HBM store; for
    // a pinned-host store in the HBM staging buffer (hashing host memory over
    // the link is slow), copied out at the end
    uint8_t *tgt = dev;
    if (host) {
        if (s->stage_used) KVG_CUDA(cudaStreamWaitEvent(st, s->stage_free, 0));  // the last deposit's copy-out
        cudaError_t e = s->stage.ensure(lay.total);
        if (e != cudaSuccess) {
            store_unalloc(s, dev, lay.total);
            return cuda_fail(e, "deposit staging buffer");
        }
        tgt = static_cast<uint8_t *>(s->stage.ptr);
    }
    HeaderParams hp;
    hp.dst = tgt;
    build_header(hp.bytes, s->dims, lay);
    KVG_CUDA(launch_write_header(hp, st));
    stt = zero_block_gaps(tgt, lay, s->dims.n_layers, st);
    if (stt != KVG_OK) return stt;
    const auto &sp = c->seq_pages[seq];
    const int64_t j_first = slot0 / P;
    for (int64_t base = 0; base < lay.n_pages; base += kMaxPagesPerLaunch) {
        GatherParams p{};
        p.pool = c->pool;
        p.dst = tgt + lay.pages_off;
        p.page_bytes = c->page_bytes;
        p.pool_pages = c->n_pages;
        p.n_layers = c->dims.n_layers;
        p.npb = (int32_t)std::min<int64_t>(kMaxPagesPerLaunch, lay.n_pages - base);
        p.page_base = (int32_t)base;
        p.block_pages = (int32_t)lay.n_pages;
        p.n_kv_heads = c->dims.n_kv_heads;
        p.page_size = (int32_t)P;
        p.head_dim = c->dims.head_dim;
        p.n_tokens = n;
        p.src_pos = c->positions + (int64_t)seq * c->max_slots + slot0 + base * P;
        p.dst_pos = reinterpret_cast<int32_t *>(tgt + lay.pos_off) + base * P;
        p.pids.n = p.npb;
        for (int32_t i = 0; i < p.npb; ++i) p.pids.pid[i] = sp[j_first + base + i];
        KVG_CUDA(launch_gather(p, s->n_sm, st));
    }
    // the position tags bound later relocations (host-side checks): read once
    std::vector<int32_t> pos(n);
    KVG_CUDA(cudaMemcpyAsync(pos.data(), tgt + lay.pos_off, 4ull * n, cudaMemcpyDeviceToHost, st));
    KVG_CUDA(cudaStreamSynchronize(st));
    // page digests on the caller's stream; the block digest (one serial chain
    // over the position tags and every page digest) on the store's digest
    // stream, so the call does not wait for it and consecutive deposits
    // overlap it.  Everything that reads a block digest (block info, export,
    // save) synchronizes the device first.
    const kvg_dims &d = s->dims;
    const uint64_t pb = page_bytes_of(d);
    const int64_t m = (int64_t)((pb + kLeafBytes - 1) / kLeafBytes);
    const int64_t n_pages = (int64_t)d.n_layers * 2 * lay.n_pages;
    KVG_CUDA(wait_for_leaf_scratch(s, st));
    KVG_CUDA(s->leaf.ensure((size_t)n_pages * m * 32));
    PageSource src{tgt + lay.pages_off, pb, nullptr, 1, 0};
    uint32_t *leaf = static_cast<uint32_t *>(s->leaf.ptr);
    KVG_CUDA(launch_sha256_leaves(src, n_pages, leaf, s->n_sm, st));
    KVG_CUDA(launch_sha256_pages(leaf, n_pages, m, tgt + lay.dig_off, nullptr, s->status, -1, st));
    KVG_CUDA(cudaEventRecord(s->pages_done, st));
    s->pages_recorded = true;
    KVG_CUDA(cudaStreamWaitEvent(s->digest_stream, s->pages_done, 0));
    KVG_CUDA(launch_sha256_serial(tgt + lay.pos_off, 4ull * n, tgt + lay.dig_off, (uint64_t)n_pages * 32, tgt + 96,
                                  nullptr, s->status, s->digest_stream));
    if (host) {
        // everything but the header follows the page digests on the caller's
        // stream; the header (with the block digest) follows the digest
        KVG_CUDA(cudaMemcpyAsync(host + lay.pos_off, tgt + lay.pos_off, lay.total - lay.pos_off,
                                 cudaMemcpyDeviceToHost, st));
        KVG_CUDA(cudaMemcpyAsync(host, tgt, lay.pos_off, cudaMemcpyDeviceToHost, s->digest_stream));
        KVG_CUDA(cudaEventRecord(s->stage_free, s->digest_stream));
        s->stage_used = true;
    }
    kvg_store::Blk b{dev, host, lay, 0, 0};
    minmax_positions(pos.data(), n, &b.min_pos, &b.max_pos);
    s->blocks.push_back(b);
    *block_id_out = s->blocks.size() - 1;
    return KVG_OK;
}

// ------------------------------------------------------------------- graft --

static kvg_status read_status(kvg_cache *c, kvg_graft_report *report) {
    DevStatus hs;
    KVG_CUDA(cudaMemcpy(&hs, c->status, sizeof hs, cudaMemcpyDeviceToHost));
    KVG_CUDA(cudaMemset(c->status, 0, sizeof(DevStatus)));
    if (report) {
        report->seq = hs.seq;
        report->n_mismatch = hs.n_mismatch;
        report->n_listed = std::min(hs.n_mismatch, (int32_t)KVG_REPORT_MAX_PAGES);
        for (int i = 0; i < report->n_listed; ++i) report->mismatch_pages[i] = hs.list[i];
    }
    if (hs.err == KVG_ERR_DIGEST || hs.n_mismatch)
        return fail(KVG_ERR_DIGEST, "digest mismatch on %d page(s) (seq %d)", hs.n_mismatch, hs.seq);
    if (hs.err) return fail((kvg_status)hs.err, "device check failed (detail %d)", hs.err_detail);
    return KVG_OK;
}

// Hashes the block's pages as restored in the cache (from_store == false:
// pages named by the sequence's device page table from page index j0) or as
// stored (from_store == true), comparing with the stored digests.
static kvg_status enqueue_verify(kvg_store *s, const kvg_store::Blk &blk, kvg_cache *c, int32_t seq, int64_t j0,
                                 bool from_store, cudaStream_t st) {
    (void)s;
    const uint64_t pb = c->page_bytes;
    const int64_t npb = blk.lay.n_pages;
    const int64_t m = (int64_t)((pb + kLeafBytes - 1) / kLeafBytes);
    const int64_t n_pages = (int64_t)c->dims.n_layers * 2 * npb;
    KVG_CUDA(c->leaf.ensure((size_t)n_pages * m * 32));
    PageSource src;
    if (!from_store)
        src = PageSource{c->pool, pb, c->page_table + (int64_t)seq * c->max_pages + j0, (int32_t)npb,
                         (int64_t)c->n_pages};
    else
        src = PageSource{blk.dev + blk.lay.pages_off, pb, nullptr, 1, 0};
    uint32_t *leaf = static_cast<uint32_t *>(c->leaf.ptr);
    KVG_CUDA(launch_sha256_leaves(src, n_pages, leaf, c->n_sm, st));
    KVG_CUDA(launch_sha256_pages(leaf, n_pages, m, nullptr, blk.dev + blk.lay.dig_off, c->status, seq, st));
    return KVG_OK;
}

static kvg_status finish_verify(kvg_cache *c, int32_t seq, uint32_t flags, int32_t checked, cudaStream_t st,
                                kvg_graft_report *report) {
    if (report) {
        memset(report, 0, sizeof *report);
        report->seq = seq;
        report->n_pages_checked = checked;
    }
    if (flags & KVG_GRAFT_SYNC) {
        KVG_CUDA(cudaStreamSynchronize(st));
        kvg_status r = read_status(c, report);
        if (report) report->n_pages_checked = checked;
        return r;
    }
    return KVG_OK;
}

// Own-position graft of a pool-resident block by aliasing: the sequence's
// page table points at the block's full pages (shared, read-only: appends
// never write a full page); a partially filled last page is copied into a
// page of the sequence, because the sequence's appends fill it.
// Per-chunk completion events of a graft (kvg_graft_chunked): chunk k of
// n_chunks maps to event k * n_events / n_chunks, recorded on the graft's
// stream after the last chunk that maps to it.
struct ChunkEvents {
    void *const *events = nullptr;
    int32_t max_events = 0;
    int32_t *end_slot = nullptr;
    int32_t *n_out = nullptr;
};

// A graft done in one piece (pool-resident blocks): one event, at its end.
static cudaError_t record_single_chunk(const ChunkEvents &ce, cudaStream_t st, int64_t end_slot) {
    if (!ce.events) return cudaSuccess;
    if (ce.n_out) *ce.n_out = 1;
    ce.end_slot[0] = (int32_t)end_slot;
    return cudaEventRecord(static_cast<cudaEvent_t>(ce.events[0]), st);
}

static kvg_status pool_graft(kvg_store *s, const kvg_store::Blk &blk, kvg_cache *c, int32_t seq, int64_t dst,
                             int64_t delta, uint32_t flags, cudaStream_t st, kvg_graft_report *report,
                             const ChunkEvents &ce) {
    if (s->pool_cache != c) return fail(KVG_ERR_ARG, "a pool-resident block grafts only into its own cache");
    if (delta != 0) return fail(KVG_ERR_ARG, "relocation needs a copying store (HBM or pinned host)");
    const int64_t P = c->dims.page_size, n = blk.lay.n_tokens, npb = blk.lay.n_pages;
    if (npb > kMaxPagesPerLaunch) return fail(KVG_ERR_ARG, "pool-resident blocks are limited to %d pages", kMaxPagesPerLaunch);
    const bool partial = n % P != 0;
    if (partial && c->free_list.empty()) return fail(KVG_ERR_CAPACITY, "out of free pages");
    std::vector<int32_t> pages(blk.pids);
    if (partial) pages.back() = take_pages(c, 1)[0];
    for (int64_t j = 0; j < npb; ++j)
        if (pages[j] == blk.pids[j]) ++c->alias[pages[j]];
    auto &sp = c->seq_pages[seq];
    const int64_t jdst = dst / P;
    sp.insert(sp.end(), pages.begin(), pages.end());
    c->n_slots[seq] = (int32_t)(dst + n);
    note_fills(c, seq, dst, dst + n);
    if (partial) {
        GatherParams p{};
        p.pool = c->pool;
        p.dst = c->pool;
        p.page_bytes = c->page_bytes;
        p.pool_pages = c->n_pages;
        p.n_layers = c->dims.n_layers;
        p.npb = 1;
        p.page_base = (int32_t)(npb - 1);
        p.block_pages = (int32_t)npb;
        p.n_kv_heads = c->dims.n_kv_heads;
        p.page_size = (int32_t)P;
        p.head_dim = c->dims.head_dim;
        p.n_tokens = n;
        p.src_pos = nullptr;
        p.pids.n = 1;
        p.pids.pid[0] = blk.pids.back();
        p.dst_pids.n = 1;
        p.dst_pids.pid[0] = pages.back();
        KVG_CUDA(launch_gather(p, c->n_sm, st));
    }
    AliasParams ap{};
    ap.src_pos = reinterpret_cast<const int32_t *>(blk.dev + blk.lay.pos_off);
    ap.table_row = c->page_table + (int64_t)seq * c->max_pages + jdst;
    ap.fill_row = c->page_fill + (int64_t)seq * c->max_pages + jdst;
    ap.dst_pos = c->positions + (int64_t)seq * c->max_slots + dst;
    ap.n_tokens = n;
    ap.page_size = (int32_t)P;
    ap.pids.n = (int32_t)npb;
    for (int64_t j = 0; j < npb; ++j) ap.pids.pid[j] = pages[j];
    KVG_CUDA(launch_alias(ap, c->n_sm, st));
    KVG_CUDA(record_single_chunk(ce, st, dst + n));
    if (flags & KVG_GRAFT_VERIFY) {
        kvg_status r = enqueue_verify(s, blk, c, seq, jdst, false, st);
        if (r != KVG_OK) return r;
    }
    return finish_verify(c, seq, flags, (flags & KVG_GRAFT_VERIFY) ? (int32_t)(c->dims.n_layers * 2 * npb) : 0,
                         st, report);
}

// A copy out of a pinned-host store waits on the host link: 32 CTAs keep it
// at its limit (211 GB/s on the GB300 measured, the same as with 608), and the
// other SMs stay free for the work that runs beside the graft (appends,
// decodes, the digest check); with a CTA on every SM the copy held them all
// and an append beside it finished only when the graft did.
static int host_copy_grid_cap() {
    static const int cap = env_knob("KVG_HOST_COPY_CTAS", 32);
    return cap;
}

// cos and sin of delta * w_i, w_i = theta^(-2i/D), i < D/2 (Sec. 4.2's
// re-basing of a block by delta positions): fp64 on the host, rounded to the
// fp32 the kernels rotate with.  One function for every graft path, so a
// re-based block gets the same bytes whichever entry point grafts it.
static void rope_table(const kvg_dims &d, int64_t delta, float *cosv, float *sinv) {
    const int half = d.head_dim / 2;
    for (int i = 0; i < half; ++i) {
        const double w = std::pow(d.rope_theta, -2.0 * i / d.head_dim);
        const double a = (double)delta * w;
        cosv[i] = (float)std::cos(a);
        sinv[i] = (float)std::sin(a);
    }
}

// rope_table for dims d (a store's; head_dim equal to the cache's),
// remembered per delta on the cache: at most 4,096 tables are kept, and the
// memo is cleared when it would grow past that or when d's RoPE base differs
// from the one its tables were made with.
static const float *rope_table_memo(kvg_cache *c, const kvg_dims &d, int64_t delta) {
    if (c->rope_memo_theta != d.rope_theta) {
        c->rope_memo.clear();
        c->rope_memo_theta = d.rope_theta;
    }
    auto it = c->rope_memo.find(delta);
    if (it != c->rope_memo.end()) return it->second.data();
    if (c->rope_memo.size() >= 4096) c->rope_memo.clear();
    const int half = d.head_dim / 2;
    std::vector<float> t((size_t)2 * half);
    rope_table(d, delta, t.data(), t.data() + half);
    return c->rope_memo.emplace(delta, std::move(t)).first->second.data();
}

static kvg_status graft_impl(kvg_store *s, uint64_t block_id, kvg_cache *c, int32_t seq, int32_t dst_slot,
                             int64_t delta, uint32_t flags, void *stream, kvg_graft_report *report,
                             const ChunkEvents &ce) {
    if (!s || !c) return fail(KVG_ERR_ARG, "null argument");
    if (block_id >= s->blocks.size()) return fail(KVG_ERR_NOT_FOUND, "no block %llu", (unsigned long long)block_id);
    if (!same_geometry(s->dims, c->dims)) return fail(KVG_ERR_ARG, "store and cache geometry differ");
    if (s->device != c->device) return fail(KVG_ERR_ARG, "store and cache on different devices");
    if (seq < 0 || seq >= c->max_seqs) return fail(KVG_ERR_ARG, "bad seq %d", seq);
    if (flags & ~(uint32_t)(KVG_GRAFT_VERIFY | KVG_GRAFT_SYNC)) return fail(KVG_ERR_ARG, "unknown flags");
    const auto &blk = s->blocks[block_id];
    const int64_t P = c->dims.page_size;
    const int64_t boundary = (c->n_slots[seq] + P - 1) / P * P;
    const int64_t dst = dst_slot < 0 ? boundary : dst_slot;
    if (dst != boundary) return fail(KVG_ERR_ARG, "dst_slot %d is not the next page boundary %lld", dst_slot, (long long)boundary);
    const int64_t n = blk.lay.n_tokens, npb = blk.lay.n_pages;
    if (dst + n > c->max_slots) return fail(KVG_ERR_CAPACITY, "graft past max_slots");
    if (!s->pool_cache && npb > (int64_t)c->free_list.size()) return fail(KVG_ERR_CAPACITY, "out of free pages");
    if (blk.min_pos + delta < 0 || blk.max_pos + delta >= (1ll << 31))
        return fail(KVG_ERR_POSITION, "position tags + delta leave [0, 2^31)");
    if (delta != 0 && c->dims.kv_dtype != KVG_KV_BF16) return fail(KVG_ERR_ARG, "relocation needs a bf16 cache");
    DeviceGuard g(c->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (s->pool_cache) return pool_graft(s, blk, c, seq, dst, delta, flags, st, report, ce);
    auto pids = take_pages(c, npb);
    auto &sp = c->seq_pages[seq];
    const int64_t jdst = dst / P;
    sp.insert(sp.end(), pids.begin(), pids.end());
    c->n_slots[seq] = (int32_t)(dst + n);
    note_fills(c, seq, dst, dst + n);

    GraftParams p{};
    p.src = blk.dev + blk.lay.pages_off;
    p.pool = c->pool;
    p.page_bytes = c->page_bytes;
    p.pool_pages = c->n_pages;
    p.n_layers = c->dims.n_layers;
    p.block_pages = (int32_t)npb;
    p.chunk_bytes = copy_chunk_bytes(c->dims);
    p.n_kv_heads = c->dims.n_kv_heads;
    p.page_size = (int32_t)P;
    p.head_dim = c->dims.head_dim;
    p.n_tokens = n;
    p.delta = delta;
    p.rotate = 0;
    if (delta != 0) {
        p.rotate = s->dims.rope_style == KVG_ROPE_HALF ? 1 : 2;
        rope_table(s->dims, delta, p.cosv, p.sinv);
    }
    const int32_t *bpos = reinterpret_cast<const int32_t *>(blk.dev + blk.lay.pos_off);
    // A verified own-position graft from an HBM store reads each page once:
    // the copy and the leaf hashes are one kernel, and only the page digests
    // follow.  From a pinned-host store the copy instead moves page-range
    // chunks with the copy kernel (whose wide reads keep the host link at its
    // limit) and a library stream hashes each chunk's restored pages in HBM
    // while the next chunk crosses the link; the last, short chunk goes
    // through the one-pass kernel.
    const bool host_src = s->residency == KVG_RESIDENCY_PINNED_HOST;
    const int host_copy_ctas = host_copy_grid_cap();
    const bool verify0 = (flags & KVG_GRAFT_VERIFY) && delta == 0;
    const bool piped = verify0 && s->residency == KVG_RESIDENCY_PINNED_HOST;
    const bool fused = verify0 && !piped;
    const int64_t m = (int64_t)((c->page_bytes + kLeafBytes - 1) / kLeafBytes);
    if (verify0) KVG_CUDA(c->leaf.ensure((size_t)c->dims.n_layers * 2 * npb * m * 32));
    int64_t step = kMaxPagesPerLaunch;
    // piped: equal chunks, then two short ones (3/128 and 1/128 of the block,
    // at least three pages and one): a chunk is hashed while the next one
    // crosses the link, and only the last chunk's hash and the page digests
    // follow the transfer, so each chunk's hash must fit in the next one's copy
    std::vector<int64_t> tails;
    if (piped) {
        if (!c->aux) {
            KVG_CUDA(cudaStreamCreateWithFlags(&c->aux, cudaStreamNonBlocking));
            for (cudaEvent_t &e : c->aux_ev) KVG_CUDA(cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
        }
        if (npb > kHostVerifyChunks) {
            const int64_t t1 = std::min<int64_t>(std::max<int64_t>(1, npb / 128), kMaxPagesPerLaunch / 3);
            tails = {3 * t1, t1};
            const int64_t body = npb - 4 * t1;
            step = std::min<int64_t>(step, (body + kHostVerifyChunks - 3) / (kHostVerifyChunks - 2));
        } else {
            step = 1;
        }
    }
    std::vector<std::pair<int64_t, int32_t>> plan;  // (first page, pages) per chunk
    int64_t tail_pages = 0;
    for (int64_t t : tails) tail_pages += t;
    for (int64_t base = 0; base < npb - tail_pages;) {
        const int64_t k = std::min<int64_t>(step, npb - tail_pages - base);
        plan.push_back({base, (int32_t)k});
        base += k;
    }
    for (int64_t t : tails) {
        const int64_t base = plan.empty() ? 0 : plan.back().first + plan.back().second;
        plan.push_back({base, (int32_t)t});
    }
    const int64_t n_chunks = (int64_t)plan.size();
    const int64_t n_ev = ce.events ? std::min<int64_t>(ce.max_events, n_chunks) : 0;
    if (ce.n_out) *ce.n_out = (int32_t)n_ev;
    for (int64_t chunk = 0; chunk < n_chunks; ++chunk) {
        const int64_t base = plan[chunk].first;
        p.npb = plan[chunk].second;
        p.page_base = (int32_t)base;
        p.src_pos = bpos + base * P;
        p.dst_pos = c->positions + (int64_t)seq * c->max_slots + dst + base * P;
        p.table_row = c->page_table + (int64_t)seq * c->max_pages + jdst + base;
        p.fill_row = c->page_fill + (int64_t)seq * c->max_pages + jdst + base;
        p.pids.n = p.npb;
        for (int32_t i = 0; i < p.npb; ++i) p.pids.pid[i] = pids[base + i];
        // piped: the last (short) chunk is copied and hashed in one pass, so
        // its hash needs no second read after it has crossed the link
        const bool one_pass = fused || (piped && chunk == n_chunks - 1);
        // the ring form for bf16 caches only: it shortens the window it shares
        // with the bf16 append (a shared-memory-staged kernel), but starves
        // beside the fp8 append (a register kernel: the SMs it runs on are set
        // up without room for the ring's shared memory)
        if (one_pass)
            KVG_CUDA(launch_graft_verify(p, static_cast<uint32_t *>(c->leaf.ptr), c->n_sm, st,
                                         c->dims.kv_dtype == KVG_KV_BF16, !host_src));
        else
            KVG_CUDA(launch_graft_copy(p, c->n_sm, st, host_src ? host_copy_ctas : 0, c->status));
        if (n_ev > 0) {
            const int64_t j = chunk * n_ev / n_chunks;
            if (chunk == n_chunks - 1 || (chunk + 1) * n_ev / n_chunks != j) {
                KVG_CUDA(cudaEventRecord(static_cast<cudaEvent_t>(ce.events[j]), st));
                ce.end_slot[j] = (int32_t)(dst + std::min<int64_t>((base + p.npb) * P, n));
            }
        }
        if (piped && !one_pass) {
            // (more than kHostVerifyChunks chunks only past 16 x 1,024 pages per
            // plane; an event is re-recorded after its wait is enqueued)
            cudaEvent_t ev = c->aux_ev[chunk % kHostVerifyChunks];
            KVG_CUDA(cudaEventRecord(ev, st));
            KVG_CUDA(cudaStreamWaitEvent(c->aux, ev, 0));
            PageSource src{c->pool, c->page_bytes, c->page_table + (int64_t)seq * c->max_pages + jdst + base, p.npb,
                           (int64_t)c->n_pages};
            src.out_plane_stride = npb;
            src.out_j0 = (int32_t)base;
            KVG_CUDA(launch_sha256_leaves(src, (int64_t)c->dims.n_layers * 2 * p.npb,
                                          static_cast<uint32_t *>(c->leaf.ptr), c->n_sm, c->aux));
        }
    }
    if (piped) {
        KVG_CUDA(cudaEventRecord(c->aux_ev[kHostVerifyChunks], c->aux));
        KVG_CUDA(cudaStreamWaitEvent(st, c->aux_ev[kHostVerifyChunks], 0));
    }
    if (verify0) {
        KVG_CUDA(launch_sha256_pages(static_cast<const uint32_t *>(c->leaf.ptr), (int64_t)c->dims.n_layers * 2 * npb, m,
                                     nullptr, blk.dev + blk.lay.dig_off, c->status, seq, st));
    } else if (flags & KVG_GRAFT_VERIFY) {
        kvg_status r = enqueue_verify(s, blk, c, seq, jdst, true, st);
        if (r != KVG_OK) return r;
    }
    return finish_verify(c, seq, flags, (flags & KVG_GRAFT_VERIFY) ? (int32_t)(c->dims.n_layers * 2 * npb) : 0,
                         st, report);
}

extern "C" kvg_status kvg_graft(kvg_store *s, uint64_t block_id, kvg_cache *c, int32_t seq, int32_t dst_slot,
                                int64_t delta, uint32_t flags, void *stream, kvg_graft_report *report) {
    Trace trace_("kvg_graft");
    return graft_impl(s, block_id, c, seq, dst_slot, delta, flags, stream, report, ChunkEvents{});
}

extern "C" kvg_status kvg_graft_chunked(kvg_store *s, uint64_t block_id, kvg_cache *c, int32_t seq,
                                        int32_t dst_slot, int64_t delta, uint32_t flags, void *stream,
                                        kvg_graft_report *report, void *const *events, int32_t max_events,
                                        int32_t *chunk_end_slot, int32_t *n_chunks) {
    Trace trace_("kvg_graft_chunked");
    if (!events || max_events < 1 || !chunk_end_slot || !n_chunks)
        return fail(KVG_ERR_ARG, "events, max_events >= 1, chunk_end_slot and n_chunks are required");
    for (int32_t i = 0; i < max_events; ++i)
        if (!events[i]) return fail(KVG_ERR_ARG, "null event %d", i);
    *n_chunks = 0;
    ChunkEvents ce;
    ce.events = events;
    ce.max_events = max_events;
    ce.end_slot = chunk_end_slot;
    ce.n_out = n_chunks;
    return graft_impl(s, block_id, c, seq, dst_slot, delta, flags, stream, report, ce);
}

extern "C" kvg_status kvg_graft_batch(kvg_store *s, const uint64_t *block_ids, kvg_cache *c, const int32_t *seq_ids,
                                      const int64_t *deltas, int32_t n, uint32_t flags, void *stream,
                                      kvg_graft_report *report) {
    Trace trace_("kvg_graft_batch");
    if (!s || !c || !block_ids || !seq_ids) return fail(KVG_ERR_ARG, "null argument");
    if (n <= 0 || n > kMaxGraftsPerBatch) return fail(KVG_ERR_ARG, "n must be in [1, %d]", kMaxGraftsPerBatch);
    if (!same_geometry(s->dims, c->dims)) return fail(KVG_ERR_ARG, "store and cache geometry differ");
    if (s->device != c->device) return fail(KVG_ERR_ARG, "store and cache on different devices");
    if (s->pool_cache) return fail(KVG_ERR_ARG, "a pool-resident store grafts with kvg_graft (aliasing)");
    if (flags & ~(uint32_t)(KVG_GRAFT_VERIFY | KVG_GRAFT_SYNC)) return fail(KVG_ERR_ARG, "unknown flags");
    const int64_t P = c->dims.page_size;
    // every check before any state changes: the batch happens whole or not at all
    std::unordered_map<int32_t, int64_t> slots;
    int64_t pages = 0;
    for (int32_t i = 0; i < n; ++i) {
        const int32_t seq = seq_ids[i];
        if (seq < 0 || seq >= c->max_seqs) return fail(KVG_ERR_ARG, "bad seq %d (graft %d)", seq, i);
        if (block_ids[i] >= s->blocks.size())
            return fail(KVG_ERR_NOT_FOUND, "no block %llu (graft %d)", (unsigned long long)block_ids[i], i);
        const auto &blk = s->blocks[block_ids[i]];
        auto it = slots.emplace(seq, (int64_t)c->n_slots[seq]).first;
        const int64_t dst = (it->second + P - 1) / P * P;
        if (dst + blk.lay.n_tokens > c->max_slots) return fail(KVG_ERR_CAPACITY, "graft %d past max_slots", i);
        if (blk.lay.n_pages > kMaxPagesPerLaunch) return fail(KVG_ERR_ARG, "graft %d: block too long for a batch", i);
        const int64_t delta = deltas ? deltas[i] : 0;
        if (blk.min_pos + delta < 0 || blk.max_pos + delta >= (1ll << 31))
            return fail(KVG_ERR_POSITION, "graft %d: position tags + delta leave [0, 2^31)", i);
        if (delta != 0 && c->dims.kv_dtype != KVG_KV_BF16)
            return fail(KVG_ERR_ARG, "graft %d: relocation needs a bf16 cache", i);
        it->second = dst + blk.lay.n_tokens;
        pages += blk.lay.n_pages;
    }
    if (pages > (int64_t)c->free_list.size()) return fail(KVG_ERR_CAPACITY, "out of free pages");
    DeviceGuard g(c->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // one cos/sin table per distinct nonzero delta, in order of first use
    std::vector<int64_t> table_delta;
    std::vector<int32_t> trig_of(n, -1);
    std::unordered_map<int64_t, int32_t> table_of;
    for (int32_t i = 0; i < n; ++i) {
        const int64_t delta = deltas ? deltas[i] : 0;
        if (delta == 0) continue;
        auto f = table_of.emplace(delta, (int32_t)table_delta.size());
        if (f.second) table_delta.push_back(delta);
        trig_of[i] = f.first->second;
    }
    const int half = c->dims.head_dim / 2;
    // the job table: metas, jobs, then the cos/sin tables, in pinned host memory
    const size_t meta_bytes = (size_t)n * sizeof(GraftMeta);
    const size_t trig_off = (meta_bytes + (size_t)pages * sizeof(GraftJob) + 15) / 16 * 16;
    const size_t bytes = trig_off + table_delta.size() * 2 * half * sizeof(float);
    if (!c->batch_ev) KVG_CUDA(cudaEventCreateWithFlags(&c->batch_ev, cudaEventDisableTiming));
    KVG_CUDA(cudaEventSynchronize(c->batch_ev));  // the previous batch's copy has read the staging
    if (bytes > c->batch_host_cap) {
        if (c->batch_host) cudaFreeHost(c->batch_host);
        c->batch_host = nullptr;
        c->batch_host_cap = 0;
        const size_t want = std::max(bytes, (size_t)1 << 16);
        KVG_CUDA(cudaHostAlloc(reinterpret_cast<void **>(&c->batch_host), want, cudaHostAllocDefault));
        c->batch_host_cap = want;
    }
    KVG_CUDA(c->batch_dev.ensure(bytes));
    GraftMeta *metas = reinterpret_cast<GraftMeta *>(c->batch_host);
    GraftJob *jobs = reinterpret_cast<GraftJob *>(c->batch_host + meta_bytes);
    std::vector<std::pair<int32_t, int64_t>> verify_at;  // (seq, first page index) per graft
    int32_t job = 0;
    for (int32_t i = 0; i < n; ++i) {
        const int32_t seq = seq_ids[i];
        const auto &blk = s->blocks[block_ids[i]];
        const int64_t nt = blk.lay.n_tokens, npb = blk.lay.n_pages;
        const int64_t dst = (c->n_slots[seq] + P - 1) / P * P;
        auto pids = take_pages(c, npb);
        auto &sp = c->seq_pages[seq];
        const int64_t jdst = dst / P;
        sp.insert(sp.end(), pids.begin(), pids.end());
        c->n_slots[seq] = (int32_t)(dst + nt);
        note_fills(c, seq, dst, dst + nt);
        GraftMeta &m = metas[i];
        m.src_pos = reinterpret_cast<const int32_t *>(blk.dev + blk.lay.pos_off);
        m.dst_pos = c->positions + (int64_t)seq * c->max_slots + dst;
        m.table_row = c->page_table + (int64_t)seq * c->max_pages + jdst;
        m.fill_row = c->page_fill + (int64_t)seq * c->max_pages + jdst;
        m.n_tokens = nt;
        m.delta = deltas ? deltas[i] : 0;
        m.npb = (int32_t)npb;
        m.first_job = job;
        m.trig = trig_of[i];
        m.pad_ = 0;
        for (int64_t j = 0; j < npb; ++j, ++job)
            jobs[job] = GraftJob{blk.dev + blk.lay.pages_off + (uint64_t)j * c->page_bytes, (int32_t)npb, pids[j], i,
                                 (int32_t)j};
        verify_at.push_back({seq, jdst});
    }
    float *trig = reinterpret_cast<float *>(c->batch_host + trig_off);
    for (size_t t = 0; t < table_delta.size(); ++t)
        memcpy(trig + t * 2 * half, rope_table_memo(c, s->dims, table_delta[t]), (size_t)2 * half * sizeof(float));
    KVG_CUDA(cudaMemcpyAsync(c->batch_dev.ptr, c->batch_host, bytes, cudaMemcpyHostToDevice, st));
    KVG_CUDA(cudaEventRecord(c->batch_ev, st));
    GraftBatchParams p{};
    p.metas = static_cast<const GraftMeta *>(c->batch_dev.ptr);
    p.jobs = reinterpret_cast<const GraftJob *>(static_cast<uint8_t *>(c->batch_dev.ptr) + meta_bytes);
    p.trig = reinterpret_cast<const float *>(static_cast<uint8_t *>(c->batch_dev.ptr) + trig_off);
    p.n_jobs = pages;
    p.n_grafts = n;
    p.n_layers = c->dims.n_layers;
    p.page_size = (int32_t)P;
    p.chunk_bytes = copy_chunk_bytes(c->dims);
    p.n_kv_heads = c->dims.n_kv_heads;
    p.head_dim = c->dims.head_dim;
    p.page_bytes = c->page_bytes;
    p.pool_pages = c->n_pages;
    p.pool = c->pool;
    // the store's RoPE pairing and base, as kvg_graft uses them
    const int rotate = table_delta.empty() ? 0 : s->dims.rope_style == KVG_ROPE_HALF ? 1 : 2;
    KVG_CUDA(launch_graft_batch(p, c->n_sm, st, s->residency == KVG_RESIDENCY_PINNED_HOST ? host_copy_grid_cap() : 0,
                                rotate));
    // verification: own-position grafts hash their restored pages; re-based
    // ones hash the stored pages (their key pages differ by design)
    if (flags & KVG_GRAFT_VERIFY)
        for (int32_t i = 0; i < n; ++i) {
            kvg_status r = enqueue_verify(s, s->blocks[block_ids[i]], c, verify_at[i].first, verify_at[i].second,
                                          trig_of[i] >= 0, st);
            if (r != KVG_OK) return r;
        }
    return finish_verify(c, n == 1 ? seq_ids[0] : -1, flags,
                         (flags & KVG_GRAFT_VERIFY) ? (int32_t)(c->dims.n_layers * 2 * pages) : 0, st, report);
}

extern "C" kvg_status kvg_verify(kvg_store *s, uint64_t block_id, kvg_cache *c, int32_t seq, int32_t slot0,
                                 uint32_t flags, void *stream, kvg_graft_report *report) {
    Trace trace_("kvg_verify");
    if (!s || !c) return fail(KVG_ERR_ARG, "null argument");
    if (block_id >= s->blocks.size()) return fail(KVG_ERR_NOT_FOUND, "no block %llu", (unsigned long long)block_id);
    if (!same_geometry(s->dims, c->dims)) return fail(KVG_ERR_ARG, "store and cache geometry differ");
    if (s->device != c->device) return fail(KVG_ERR_ARG, "store and cache on different devices");
    if (seq < 0 || seq >= c->max_seqs) return fail(KVG_ERR_ARG, "bad seq %d", seq);
    if (flags & ~(uint32_t)(KVG_GRAFT_VERIFY | KVG_GRAFT_SYNC)) return fail(KVG_ERR_ARG, "unknown flags");
    const auto &blk = s->blocks[block_id];
    const int64_t P = c->dims.page_size;
    if (slot0 < 0 || slot0 % P) return fail(KVG_ERR_ARG, "slot0 must be page-aligned");
    const int64_t j0 = slot0 / P;
    if (j0 + blk.lay.n_pages > (int64_t)c->seq_pages[seq].size())
        return fail(KVG_ERR_ARG, "range exceeds the sequence's pages");
    DeviceGuard g(c->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    kvg_status r = enqueue_verify(s, blk, c, seq, j0, false, st);
    if (r != KVG_OK) return r;
    return finish_verify(c, seq, flags, (int32_t)(c->dims.n_layers * 2 * blk.lay.n_pages), st, report);
}

// ------------------------------------------------------------------ decode --

// First row read by a windowed layer: the last `window` valid rows of the
// sequence, counted back over its pages' fills (a page's valid rows are
// [0, fill)).  Returns the page index and the row within it.
static void window_start(const kvg_cache *c, int32_t seq, int64_t window, int32_t *page, int32_t *row) {
    const auto &f = c->seq_fill[seq];
    int64_t acc = 0;
    for (int64_t j = (int64_t)f.size() - 1; j >= 0; --j) {
        if (acc + f[j] >= window) {
            *page = (int32_t)j;
            *row = (int32_t)(f[j] - (window - acc));
            return;
        }
        acc += f[j];
    }
    *page = 0;
    *row = 0;
}

// The launches of one decode call: the layers run are grouped by their
// window (one group when no layer is windowed), each group split into
// launches of at most kMaxLayersPerLaunch layers and kMaxBatchPerLaunch rows.
// Fills every field but the per-call ones (q, out, scale, heads, scratch,
// workers); *max_units gets the largest layers x rows x kv heads of a launch.
// page_begin / page_end: only the sequence's pages [page_begin, page_end)
// are read (a split decode over a slot range); the defaults read them all.
static kvg_status plan_decode(const kvg_cache *c, int32_t layer, const int32_t *seq_ids, int32_t B,
                              std::vector<DecodeParams> *plan, int64_t *max_units, int32_t page_begin = 0,
                              int32_t page_end = INT32_MAX) {
    const kvg_dims &d = c->dims;
    const int TOK = decode_tile_tokens(d.head_dim, d.kv_dtype == KVG_KV_E4M3);
    const int tpp = (d.page_size + TOK - 1) / TOK;
    // (window, [(cache layer, q layer)]) in order of first appearance
    std::vector<std::pair<int32_t, std::vector<std::pair<int32_t, int32_t>>>> groups;
    for (int32_t l = layer < 0 ? 0 : layer; l < (layer < 0 ? d.n_layers : layer + 1); ++l) {
        const int32_t w = c->layer_window[l];
        auto it = std::find_if(groups.begin(), groups.end(), [w](const auto &g) { return g.first == w; });
        if (it == groups.end()) {
            groups.push_back({w, {}});
            it = groups.end() - 1;
        }
        it->second.push_back({l, layer < 0 ? l : 0});
    }
    plan->clear();
    *max_units = 0;
    for (const auto &grp : groups) {
        const int64_t W = grp.first;
        for (size_t l0 = 0; l0 < grp.second.size(); l0 += kMaxLayersPerLaunch) {
            const int32_t nl = (int32_t)std::min<size_t>(kMaxLayersPerLaunch, grp.second.size() - l0);
            for (int64_t b0 = 0; b0 < B; b0 += kMaxBatchPerLaunch) {
                const int32_t nb = (int32_t)std::min<int64_t>(kMaxBatchPerLaunch, B - b0);
                plan->emplace_back();
                DecodeParams &p = plan->back();
                memset(&p, 0, sizeof p);
                int32_t acc = 0;
                for (int32_t i = 0; i < nb; ++i) {
                    const int32_t sq = seq_ids[b0 + i];
                    const int32_t np = (int32_t)c->seq_pages[sq].size();
                    int32_t pg = 0, row = 0;
                    if (W > 0) window_start(c, sq, W, &pg, &row);
                    int32_t t0 = pg * tpp + row / TOK, lo = row % TOK;
                    if (page_begin > 0 && (int64_t)page_begin * tpp > t0) {
                        t0 = page_begin * tpp;
                        lo = 0;
                    }
                    const int32_t t1 = std::min(np, page_end) * tpp;
                    p.rows.seq[i] = sq;
                    p.rows.tile0[i] = t0;
                    p.rows.lo[i] = lo;
                    p.rows.pref_tiles[i] = acc;
                    acc += std::max(0, t1 - t0);
                }
                p.rows.pref_tiles[nb] = acc;
                for (int32_t i = 0; i < nl; ++i) {
                    p.layers[i] = (int16_t)grp.second[l0 + i].first;
                    p.qlayers[i] = (int16_t)grp.second[l0 + i].second;
                }
                p.n_layers_run = nl;
                p.n_tiles = (int64_t)nl * d.n_kv_heads * acc;
                p.B = nb;
                p.b0 = (int32_t)b0;
                p.pool = c->pool;
                p.pool_pages = c->n_pages;
                p.n_kv_heads = d.n_kv_heads;
                p.page_size = d.page_size;
                p.page_table = c->page_table;
                p.page_fill = c->page_fill;
                p.max_pages = c->max_pages;
                p.status = c->status;
                *max_units = std::max<int64_t>(*max_units, (int64_t)nl * nb * d.n_kv_heads);
            }
        }
    }
    return KVG_OK;
}

extern "C" kvg_status kvg_cache_set_layer_windows(kvg_cache *c, const int32_t *windows, int32_t n) {
    if (!c) return fail(KVG_ERR_ARG, "null cache");
    if (n == 0) {
        std::fill(c->layer_window.begin(), c->layer_window.end(), 0);
        return KVG_OK;
    }
    if (!windows || n != c->dims.n_layers) return fail(KVG_ERR_ARG, "need one window per layer (%d)", c->dims.n_layers);
    for (int32_t l = 0; l < n; ++l)
        if (windows[l] < 0) return fail(KVG_ERR_ARG, "negative window for layer %d", l);
    c->layer_window.assign(windows, windows + n);
    return KVG_OK;
}

// Decode attention over the sequences' pages [page_begin, page_end): bf16
// out (state == null), or the softmax state written or merged into `state`.
static kvg_status decode_impl(const char *what, kvg_cache *c, int32_t layer, const int32_t *seq_ids, int32_t B,
                              const void *q, int32_t n_q_heads, void *out, float scale, void *stream,
                              int32_t page_begin, int32_t page_end, float *state, int32_t merge) {
    if (!c || !seq_ids || !q || !(out || state)) return fail(KVG_ERR_ARG, "%s: null argument", what);
    const kvg_dims &d = c->dims;
    if (layer < -1 || layer >= d.n_layers) return fail(KVG_ERR_ARG, "bad layer %d", layer);
    if (B <= 0 || B > 4096) return fail(KVG_ERR_ARG, "B must be in [1, 4096]");
    if (n_q_heads <= 0 || n_q_heads % d.n_kv_heads) return fail(KVG_ERR_ARG, "n_q_heads must be a multiple of n_kv_heads");
    const int G = n_q_heads / d.n_kv_heads;
    const bool fp8 = d.kv_dtype == KVG_KV_E4M3;
    if (!decode_supported(d.head_dim, G, fp8))
        return fail(KVG_ERR_ARG, "unsupported head_dim %d / group %d%s", d.head_dim, G, fp8 ? " (fp8)" : "");
    if ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(out) | reinterpret_cast<uintptr_t>(state)) & 15)
        return fail(KVG_ERR_ARG, "q/out/state must be 16-byte aligned");
    for (int32_t b = 0; b < B; ++b)
        if (seq_ids[b] < 0 || seq_ids[b] >= c->max_seqs) return fail(KVG_ERR_ARG, "bad seq id %d", seq_ids[b]);
    DeviceGuard g(c->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int w_max = decode_max_warps(d.head_dim, G, fp8, c->n_sm);
    if (w_max <= 0) return fail(KVG_ERR_CUDA, "decode kernel cannot be made resident");
    std::vector<DecodeParams> plan;
    int64_t max_units = 0;
    kvg_status r = plan_decode(c, layer, seq_ids, B, &plan, &max_units, page_begin, page_end);
    if (r != KVG_OK) return r;
    const size_t slots = (size_t)max_units + (size_t)w_max;
    if (!c->part_ev) KVG_CUDA(cudaEventCreateWithFlags(&c->part_ev, cudaEventDisableTiming));
    if (c->part_used && st != c->part_stream) KVG_CUDA(cudaStreamWaitEvent(st, c->part_ev, 0));
    KVG_CUDA(c->part_o.ensure(slots * G * d.head_dim * sizeof(float)));
    KVG_CUDA(c->part_ml.ensure(slots * G * sizeof(float2)));
    for (DecodeParams &p : plan) {
        p.n_warps = (int32_t)std::min<int64_t>(w_max, std::max<int64_t>(p.n_tiles, 1));
        p.n_q_heads = n_q_heads;
        p.q = static_cast<const __nv_bfloat16 *>(q);
        p.q_row_stride_b = B;
        p.qscale = scale * 1.4426950408889634f * (fp8 ? d.k_scale : 1.f);
        p.vscale = fp8 ? d.v_scale : 1.f;
        p.part_o = static_cast<float *>(c->part_o.ptr);
        p.part_ml = static_cast<float2 *>(c->part_ml.ptr);
        p.out = static_cast<__nv_bfloat16 *>(out);
        p.state = state;
        p.state_merge = merge;
        KVG_CUDA(launch_decode(d.head_dim, G, fp8, p, c->pool_map, st));
        KVG_CUDA(launch_combine(d.head_dim, G, p, st));
    }
    KVG_CUDA(cudaEventRecord(c->part_ev, st));
    c->part_stream = st;
    c->part_used = true;
    return KVG_OK;
}

extern "C" kvg_status kvg_decode_attention(kvg_cache *c, int32_t layer, const int32_t *seq_ids, int32_t B,
                                           const void *q, int32_t n_q_heads, void *out, float scale,
                                           void *stream) {
    Trace trace_("kvg_decode_attention");
    if (!out) return fail(KVG_ERR_ARG, "null argument");
    return decode_impl("kvg_decode_attention", c, layer, seq_ids, B, q, n_q_heads, out, scale, stream, 0, INT32_MAX,
                       nullptr, 0);
}

extern "C" kvg_status kvg_decode_attention_range(kvg_cache *c, int32_t layer, const int32_t *seq_ids, int32_t B,
                                                 const void *q, int32_t n_q_heads, float scale, int32_t slot_begin,
                                                 int32_t slot_end, uint32_t flags, float *state, void *stream) {
    Trace trace_("kvg_decode_attention_range");
    if (!c || !state) return fail(KVG_ERR_ARG, "null argument");
    if (flags & ~(uint32_t)KVG_DECODE_MERGE) return fail(KVG_ERR_ARG, "unknown flags");
    const int32_t P = c->dims.page_size;
    if (slot_begin < 0 || slot_end < slot_begin) return fail(KVG_ERR_ARG, "need 0 <= slot_begin <= slot_end");
    if (slot_begin % P || (slot_end % P && slot_end < c->max_slots))
        return fail(KVG_ERR_ARG, "slot_begin and slot_end must be multiples of page_size %d (or slot_end >= max_slots)", P);
    const int32_t pb = slot_begin / P;
    const int32_t pe = slot_end >= c->max_slots ? INT32_MAX : slot_end / P;
    return decode_impl("kvg_decode_attention_range", c, layer, seq_ids, B, q, n_q_heads, nullptr, scale, stream, pb,
                       pe, state, (flags & KVG_DECODE_MERGE) ? 1 : 0);
}

extern "C" kvg_status kvg_decode_state_finish(const float *state, int64_t n_rows, int32_t head_dim, void *out,
                                              void *stream) {
    Trace trace_("kvg_decode_state_finish");
    if (n_rows < 0 || (n_rows > 0 && (!state || !out))) return fail(KVG_ERR_ARG, "null argument or negative n_rows");
    if (head_dim != 64 && head_dim != 128 && head_dim != 256) return fail(KVG_ERR_ARG, "head_dim must be 64, 128 or 256");
    if ((reinterpret_cast<uintptr_t>(state) | reinterpret_cast<uintptr_t>(out)) & 15)
        return fail(KVG_ERR_ARG, "state/out must be 16-byte aligned");
    KVG_CUDA(launch_state_finish(state, n_rows, head_dim, static_cast<__nv_bfloat16 *>(out),
                                 static_cast<cudaStream_t>(stream)));
    return KVG_OK;
}

// ------------------------------------------------------------------ digest --

namespace {
std::mutex g_digest_mu;
Scratch g_digest_leaf[64];
DevStatus *g_digest_status[64] = {};
// Paged digests share the device's leaf scratch: each call's stream waits for
// the previous call's last kernel (recorded here), so calls on different
// streams run one after the other on the GPU instead of racing on it.
cudaEvent_t g_digest_done[64] = {};
}  // namespace

extern "C" kvg_status kvg_digest(const void *bytes, uint64_t n, int32_t mode, uint64_t page_bytes, uint8_t *out,
                                 void *stream) {
    Trace trace_("kvg_digest");
    if (!out || (n && !bytes)) return fail(KVG_ERR_ARG, "null argument");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int dev = 0;
    KVG_CUDA(cudaGetDevice(&dev));
    if (dev < 0 || dev >= 64) return fail(KVG_ERR_ARG, "device ordinal out of range");
    if (mode == KVG_SHA256_PLAIN) {
        KVG_CUDA(launch_sha256_serial(static_cast<const uint8_t *>(bytes), n, nullptr, 0, out, nullptr, nullptr, st));
        return KVG_OK;
    }
    if (mode != KVG_SHA256_PAGED) return fail(KVG_ERR_ARG, "bad mode %d", mode);
    if (page_bytes == 0 || n % page_bytes) return fail(KVG_ERR_ARG, "n must be a multiple of page_bytes");
    if (page_bytes % 16 || reinterpret_cast<uintptr_t>(bytes) % 16)
        return fail(KVG_ERR_ARG, "paged mode needs 16-byte aligned pages");
    const int64_t n_pages = (int64_t)(n / page_bytes);
    const int64_t m = (int64_t)((page_bytes + kLeafBytes - 1) / kLeafBytes);
    std::lock_guard<std::mutex> lk(g_digest_mu);
    if (!g_digest_status[dev]) {
        KVG_CUDA(cudaMalloc(&g_digest_status[dev], sizeof(DevStatus)));
        KVG_CUDA(cudaMemset(g_digest_status[dev], 0, sizeof(DevStatus)));
    }
    if (!g_digest_done[dev]) {
        KVG_CUDA(cudaEventCreateWithFlags(&g_digest_done[dev], cudaEventDisableTiming));
    } else {
        const size_t need = (size_t)n_pages * m * 32;
        // a larger scratch replaces the old one: the previous call must be done with it
        if (need > g_digest_leaf[dev].cap) KVG_CUDA(cudaEventSynchronize(g_digest_done[dev]));
        KVG_CUDA(cudaStreamWaitEvent(st, g_digest_done[dev], 0));
    }
    KVG_CUDA(g_digest_leaf[dev].ensure((size_t)n_pages * m * 32));
    PageSource src{static_cast<const uint8_t *>(bytes), page_bytes, nullptr, 1, 0};
    uint32_t *leaf = static_cast<uint32_t *>(g_digest_leaf[dev].ptr);
    KVG_CUDA(launch_sha256_leaves(src, n_pages, leaf, sm_count(dev), st));
    KVG_CUDA(launch_sha256_pages(leaf, n_pages, m, out, nullptr, g_digest_status[dev], -1, st));
    KVG_CUDA(cudaEventRecord(g_digest_done[dev], st));
    return KVG_OK;
}

// -------------------------------------------------------------------- misc --

extern "C" kvg_status kvg_sync(kvg_cache *c, void *stream, double timeout_s, kvg_graft_report *report) {
    Trace trace_("kvg_sync");
    if (!c) return fail(KVG_ERR_ARG, "null cache");
    DeviceGuard g(c->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const auto t0 = std::chrono::steady_clock::now();
    for (;;) {
        cudaError_t e = cudaStreamQuery(st);
        if (e == cudaSuccess) break;
        if (e != cudaErrorNotReady) return cuda_fail(e, "cudaStreamQuery");
        const double el = std::chrono::duration<double>(std::chrono::steady_clock::now() - t0).count();
        if (el > timeout_s) return fail(KVG_ERR_TIMEOUT, "stream still busy after %.3f s", el);
        std::this_thread::sleep_for(std::chrono::microseconds(50));
    }
    if (report) memset(report, 0, sizeof *report);
    return read_status(c, report);
}

extern "C" kvg_status kvg_selftest_bounded_wait(kvg_cache *c, uint64_t limit_ns, void *stream) {
    if (!c) return fail(KVG_ERR_ARG, "null cache");
    if (limit_ns == 0 || limit_ns > 10000000000ull) return fail(KVG_ERR_ARG, "limit must be in (0, 10 s]");
    DeviceGuard g(c->device);
    KVG_CUDA(launch_wait_selftest(c->status, limit_ns, static_cast<cudaStream_t>(stream)));
    return KVG_OK;
}

extern "C" const char *kvg_status_string(kvg_status s) {
    switch (s) {
        case KVG_OK: return "ok";
        case KVG_ERR_ARG: return "invalid argument";
        case KVG_ERR_OOM: return "out of memory";
        case KVG_ERR_CUDA: return "CUDA error";
        case KVG_ERR_NOT_FOUND: return "block not found";
        case KVG_ERR_CAPACITY: return "capacity exceeded";
        case KVG_ERR_POSITION: return "position out of range";
        case KVG_ERR_DIGEST: return "digest mismatch";
        case KVG_ERR_FORMAT: return "bad block format";
        case KVG_ERR_TIMEOUT: return "timeout";
        case KVG_ERR_DEVICE_CHECK: return "device-side check failed";
    }
    return "unknown status";
}

extern "C" const char *kvg_last_error(void) { return g_last_error.c_str(); }

namespace kvg {
// Read-only views used by noalloc.cu (CacheShape is declared in common.cuh).
bool cache_shape(const kvg_cache *c, CacheShape *out) {
    if (!c || !out) return false;
    *out = CacheShape{c->dims.n_layers, c->dims.n_kv_heads, c->dims.head_dim, c->dims.page_size, c->n_pages,
                      c->max_seqs, c->max_pages, c->device, c->n_sm, c->dims.kv_dtype, c->dims.k_scale,
                      c->dims.v_scale, c->pool, c->page_table, c->page_fill, c->status, &c->pool_map};
    return true;
}
int32_t cache_seq_pages(const kvg_cache *c, int32_t seq) { return (int32_t)c->seq_pages[seq].size(); }
kvg_status cache_plan_decode(const kvg_cache *c, int32_t layer, const int32_t *seq_ids, int32_t B,
                             std::vector<DecodeParams> *plan, int64_t *max_units) {
    return plan_decode(c, layer, seq_ids, B, plan, max_units);
}
void set_last_error(const char *msg) { g_last_error = msg; }
}  // namespace kvg

extern "C" uint32_t kvg_version(void) { return 0x000200u; }

extern "C" uint64_t kvg_launch_count(void) { return kvg::launch_count(); }

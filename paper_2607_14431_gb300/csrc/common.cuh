// common.cuh — internal declarations shared by the libkvg translation units:
// device status word, kernel parameter blocks, inline-PTX helpers for
// mbarriers and bulk (TMA, non-tensor) copies, and the launchers each .cu
// exports to the host runtime.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include <vector>

#include "kvg.h"

namespace kvg {

// ---------------------------------------------------------------- limits --
constexpr int kMaxPagesPerLaunch = 1024;  // page ids carried in kernel params
constexpr int kMaxBatchPerLaunch = 256;   // decode rows carried in kernel params
constexpr int kMaxLayersPerLaunch = 256;  // decode layers carried in kernel params
constexpr int kMaxDevices = 64;           // per-device caches of launch set-up
constexpr int kMaxHalfDim = 128;          // head_dim <= 256
constexpr uint64_t kLeafBytes = KVG_DIGEST_LEAF_BYTES;

// Device status word of a cache (or of a library-level scratch).  Kernels
// record the first error code they see; digest checks count mismatches and
// list the first KVG_REPORT_MAX_PAGES page indices.
struct DevStatus {
    int32_t err;           // 0 or a kvg_status (negative)
    int32_t err_detail;    // kernel-specific detail of the first error
    int32_t n_mismatch;
    int32_t n_checked;
    int32_t seq;
    int32_t pad[3];
    int32_t list[KVG_REPORT_MAX_PAGES];
};

struct PageList {
    int32_t n;
    int32_t pid[kMaxPagesPerLaunch];
};

// ------------------------------------------------------------ graft copy --
// One launch copies n_units = n_layers * 2 * npb pages (block page order
// (l * 2 + kv) * npb + j) from `src` (contiguous block pages) into the pool
// pages named by pids, optionally rotating the valid key rows.
struct GraftParams {
    const uint8_t *src;        // block pages region (device or host-mapped)
    uint8_t *pool;             // cache pool
    uint64_t page_bytes;
    int64_t pool_pages;        // n_pages of the pool (stride between (l,kv) planes)
    int32_t n_layers;
    int32_t npb;               // pages of this launch per (l, kv)
    int32_t page_base;         // block page index of the first page of this launch
    int32_t block_pages;       // block pages per (l, kv) (stride of src planes)
    int32_t chunk_bytes;       // unit of work: divides page_bytes, multiple of 16
    int32_t rotate;            // 0 copy, 1 half-split rotation, 2 interleaved rotation
    int32_t n_kv_heads, page_size, head_dim;
    int64_t n_tokens;          // block tokens (rows >= n_tokens are padding)
    float cosv[kMaxHalfDim];
    float sinv[kMaxHalfDim];
    // metadata written by the same launch
    const int32_t *src_pos;    // block position tags (this launch's tokens start at page_base*P)
    int32_t *dst_pos;          // positions row of the sequence + dst slot of page_base
    int32_t *table_row;        // page_table row + first page index of this launch
    int32_t *fill_row;         // page_fill row + first page index of this launch
    int64_t delta;
    PageList pids;
};

// Position tags (+ delta), page-table entries and fill counts of one graft
// launch's pages, written grid-stride by every thread of the launch.
__device__ __forceinline__ void graft_metadata(const GraftParams &p) {
    const int64_t P = p.page_size;
    const int64_t tok0 = (int64_t)p.page_base * P;
    int64_t n_meta = (int64_t)p.npb * P;
    if (tok0 + n_meta > p.n_tokens) n_meta = p.n_tokens - tok0;
    const int64_t gtid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t gsz = (int64_t)gridDim.x * blockDim.x;
    for (int64_t t = gtid; t < n_meta; t += gsz) p.dst_pos[t] = (int32_t)((int64_t)p.src_pos[t] + p.delta);
    for (int64_t j = gtid; j < p.npb; j += gsz) {
        p.table_row[j] = p.pids.pid[j];
        const int64_t f = p.n_tokens - (tok0 + j * P);
        p.fill_row[j] = (int32_t)(f < P ? f : P);
    }
}

// ------------------------------------------------------------ graft batch --
// One block page of a batched graft: its plane-0 bytes in the store, the
// stride between its (layer, K/V) planes in pages, and its cache page id.
struct GraftJob {
    const uint8_t *src;
    int32_t block_pages;
    int32_t pid;
    int32_t meta;      // the graft this page belongs to
    int32_t page;      // its page index within the block
};
// One graft of a batch: position tags, page-table row and fill row of its
// destination, and its jobs [first_job, first_job + npb).  A graft re-based
// by delta != 0 has the cos/sin table trig (>= 0) of the batch's tables.
struct GraftMeta {
    const int32_t *src_pos;
    int32_t *dst_pos;
    int32_t *table_row;
    int32_t *fill_row;
    int64_t n_tokens;
    int64_t delta;
    int32_t npb;
    int32_t first_job;
    int32_t trig;      // -1: own position (byte copy)
    int32_t pad_;
};
struct GraftBatchParams {
    const GraftJob *jobs;
    const GraftMeta *metas;
    // rotation tables of the re-based grafts: table t holds cos(delta w_i)
    // for i < head_dim / 2, then sin(delta w_i), as fp32
    const float *trig;
    int64_t n_jobs;
    int32_t n_grafts;
    int32_t n_layers, page_size, chunk_bytes;
    int32_t n_kv_heads, head_dim;
    uint64_t page_bytes;
    int64_t pool_pages;
    uint8_t *pool;
};

// ---------------------------------------------------------------- append --
struct AppendParams {
    const uint16_t *k, *v;     // [L][n][Hkv][D]
    const int32_t *pos;        // [n]
    uint8_t *pool;
    int64_t pool_pages;
    int32_t n_layers, n_kv_heads, page_size, head_dim;
    int32_t n;                 // rows of this launch
    int32_t row0;              // first row of this launch within k/v/pos
    int32_t slot0;             // slot of row0
    int32_t page0;             // page index (within the sequence) of pids.pid[0]
    int32_t n_rows_total;      // rows of the whole k/v arrays (their token stride)
    int32_t *pos_row;          // positions row of the sequence
    int32_t *table_row;        // page_table row
    int32_t *fill_row;         // page_fill row
    float k_inv_scale, v_inv_scale;  // fp8 caches: 1/scale (fp32) of the quantizing append
    PageList pids;             // pages touched: page0 .. page0 + n - 1
};

// One new row per sequence (decode step): row b goes to page pid[b], row
// `row[b]` of that page, slot slot[b] of sequence seq[b].
struct AppendBatchParams {
    const uint16_t *k, *v;     // [L][B][Hkv][D]
    const int32_t *pos;        // [B]
    uint8_t *pool;
    int64_t pool_pages;
    int32_t n_layers, n_kv_heads, page_size, head_dim, B, max_pages, max_slots;
    int32_t *page_table, *page_fill, *positions;  // whole-cache arrays
    float k_inv_scale, v_inv_scale;  // fp8 caches: 1/scale (fp32) of the quantizing append
    int32_t seq[kMaxBatchPerLaunch];
    int32_t pid[kMaxBatchPerLaunch];
    int32_t slot[kMaxBatchPerLaunch];
};

// --------------------------------------------------------------- deposit --
struct GatherParams {
    const uint8_t *pool;
    uint8_t *dst;              // block pages region (dst_pids.n == 0), or the pool (dst_pids given)
    uint64_t page_bytes;
    int64_t pool_pages;
    int32_t n_layers, npb, page_base, block_pages;
    int32_t n_kv_heads, page_size, head_dim;
    int64_t n_tokens;          // rows >= n_tokens are written as zero
    const int32_t *src_pos;    // positions row + slot0 (nullable: no position copy)
    int32_t *dst_pos;          // block positions
    PageList pids;             // source pool pages
    PageList dst_pids;         // destination pool pages (pool-resident blocks), n = 0 when unused
};

// Own-position graft by aliasing: page-table entries, fills and position
// tags of a sequence for a block whose pages already sit in the pool.
struct AliasParams {
    const int32_t *src_pos;    // block positions
    int32_t *table_row;        // page_table row + first page index
    int32_t *fill_row;         // page_fill row + first page index
    int32_t *dst_pos;          // positions row + dst slot
    int64_t n_tokens;
    int32_t page_size;
    PageList pids;             // the sequence's pages for the block, in order
};

struct IntsParams {
    int32_t *dst;
    PageList vals;
};

struct HeaderParams {
    uint8_t *dst;
    uint8_t bytes[256];
};

// ---------------------------------------------------------------- digest --
// Address of page p: contiguous (pid == nullptr): base + p * page_bytes;
// cache pages: base + ((p / npb) * plane_pages + pid[p % npb]) * page_bytes.
struct PageSource {
    const uint8_t *base;
    uint64_t page_bytes;
    const int32_t *pid;
    int32_t npb;
    int64_t plane_pages;
    // with pid: leaf digests of page (plane, j) go to page slot
    // plane * out_plane_stride + out_j0 + j of the output (0: plane * npb + j)
    int64_t out_plane_stride = 0;
    int32_t out_j0 = 0;
};

// --------------------------------------------------------------- decode --
// A launch covers Lrun layers x B batch rows x Hkv kv heads ("units").  Unit
// (l, b, g) owns T_b = npages_b * tiles_per_page tiles, in page order; the
// global tile list orders units (l, b, g) with g fastest.  Warp w of W takes
// the contiguous range [w*T/W, (w+1)*T/W) and writes one partial per unit it
// touches, at slot unit + w (unique because both ranges are contiguous).
struct BatchRows {
    int32_t seq[kMaxBatchPerLaunch];
    int32_t tile0[kMaxBatchPerLaunch];  // first tile of the row's pages that is read (window start)
    int32_t lo[kMaxBatchPerLaunch];     // rows of that first tile before the window start
    int32_t pref_tiles[kMaxBatchPerLaunch + 1];  // prefix sums of T_b
};

struct DecodeParams {
    const uint8_t *pool;
    int64_t pool_pages;
    int32_t n_kv_heads, page_size, n_q_heads;
    int32_t n_layers_run, B;
    int16_t layers[kMaxLayersPerLaunch];   // run layer lr -> cache layer
    int16_t qlayers[kMaxLayersPerLaunch];  // run layer lr -> layer index of q and out
    int32_t n_warps;           // W
    int64_t n_tiles;           // T
    const int32_t *page_table;
    const int32_t *page_fill;
    int32_t max_pages;
    const __nv_bfloat16 *q;    // [Lrun][Btot][Hq][D]
    int32_t q_row_stride_b;    // rows of the full batch (B of the whole call)
    int32_t b0;                // first batch row of this launch
    float qscale;              // softmax scale * log2(e) (* k_scale for fp8 keys)
    float vscale;              // 1, or v_scale for fp8 values (applied by the combine)
    float *part_o;             // [U + W][G][D]
    float2 *part_ml;           // [U + W][G]
    __nv_bfloat16 *out;        // [Lrun][Btot][Hq][D] (combine)
    float *state;              // split decode: fp32 [Lrun][Btot][Hq][D + 4] (o, m, l, pad); null otherwise
    int32_t state_merge;       // 1: merge into the state, 0: overwrite it
    DevStatus *status;
    BatchRows rows;
};

// -------------------------------------------------------------- launchers --
// Every launcher counts the kernels it launches (kvg_launch_count()).
void count_launches(uint64_t n);
uint64_t launch_count();
// Integer tuning knob from the environment (read once), e.g. CTAs per SM of
// a grid-stride kernel; `fallback` when unset or not positive.
int env_knob(const char *name, int fallback);

// max_ctas > 0 caps the grid (a copy from host memory needs only enough
// CTAs to keep the host link busy; the rest of the SMs stay free).
// max_ctas > 0: a host-mapped source, read by at most max_ctas CTAs of
// graft_kernel.  Otherwise the shared-memory staged graft runs when the unit
// fits its stages (its bounded waits record into `status`).
cudaError_t launch_graft_copy(const GraftParams &p, int n_sm, cudaStream_t s, int max_ctas = 0,
                              DevStatus *status = nullptr);
// Own-position copies of a batch of grafts in one launch (jobs, metas in device memory).
// rotate: 0 when every graft of the batch is at its own position, else the
// cache's RoPE pairing (1 half-split, 2 interleaved) for its re-based grafts.
cudaError_t launch_graft_batch(const GraftBatchParams &p, int n_sm, cudaStream_t s, int max_ctas = 0,
                               int rotate = 0);
// Bulk append by tensor copies, for appends of at least append_tma_rows()
// rows (16-byte aligned k/v).  Returns cudaErrorNotSupported (nothing
// launched) when the tensor maps cannot be encoded, so the caller can take
// launch_append().
int32_t append_tma_rows(int32_t page_size, int32_t head_dim);
cudaError_t launch_append_tma(const AppendParams &p, DevStatus *status, int n_sm, cudaStream_t s);
// Appends into an fp8 E4M3 cache: bf16 rows quantized with p.k_inv_scale / p.v_inv_scale.
cudaError_t launch_append_e4m3(const AppendParams &p, int n_sm, cudaStream_t s);
cudaError_t launch_append_batch_e4m3(const AppendBatchParams &p, int n_sm, cudaStream_t s);
// Own-position graft (delta 0) fused with the leaf hashes of the copied pages:
// leaf_words[(block page) * leaves_per_page + leaf] gets the leaf's state words.
// ring_ok: a launch of a full wave or more may take the shared-memory ring form.
// split_ok: a small launch may take the two-warp form (not for blocks read
// from pinned host memory, whose loads are too slow for it).
cudaError_t launch_graft_verify(const GraftParams &p, uint32_t *leaf_words, int n_sm, cudaStream_t s,
                                bool ring_ok = true, bool split_ok = true);
cudaError_t launch_append(const AppendParams &p, int n_sm, cudaStream_t s);
cudaError_t launch_append_batch(const AppendBatchParams &p, int n_sm, cudaStream_t s);
cudaError_t launch_gather(const GatherParams &p, int n_sm, cudaStream_t s);
cudaError_t launch_write_header(const HeaderParams &p, cudaStream_t s);
cudaError_t launch_alias(const AliasParams &p, int n_sm, cudaStream_t s);
// One 4-byte load per `stride` bytes of [base, base + bytes) (base 4-byte
// aligned, stride a multiple of 4): resolves the GPU's address translations
// of the pages of a block in pinned host memory ahead of its graft.
cudaError_t launch_touch(const uint8_t *base, uint64_t bytes, uint32_t stride, int n_sm, cudaStream_t s);
// A kernel whose mbarrier nothing completes: its bounded wait gives up after
// limit_ns and records KVG_ERR_DEVICE_CHECK (detail 3) in `status`.
cudaError_t launch_wait_selftest(DevStatus *status, uint64_t limit_ns, cudaStream_t s);
cudaError_t launch_write_ints(const IntsParams &p, cudaStream_t s);
cudaError_t launch_reset_seq(int32_t *table_row, int32_t *fill_row, int32_t max_pages,
                             int32_t *pos_row, int32_t max_slots, cudaStream_t s);

// leaf digests (8 uint32 words per leaf, host order of the hash state)
cudaError_t launch_sha256_leaves(const PageSource &src, int64_t n_pages, uint32_t *leaf_words,
                                 int n_sm, cudaStream_t s);
// page digests from leaf digests; writes out (nullable, 32 bytes per page) and
// compares with expected (nullable), recording mismatches in status.
cudaError_t launch_sha256_pages(const uint32_t *leaf_words, int64_t n_pages, int64_t leaves_per_page,
                                uint8_t *out, const uint8_t *expected, DevStatus *status,
                                int32_t seq, cudaStream_t s);
// SHA-256 of seg0 || seg1 (one thread); expected (nullable) compared like above.
cudaError_t launch_sha256_serial(const uint8_t *seg0, uint64_t n0, const uint8_t *seg1, uint64_t n1,
                                 uint8_t *out, const uint8_t *expected, DevStatus *status,
                                 cudaStream_t s);

// Persistent decode: p.n_warps one-warp CTAs over p.n_tiles tiles, then the
// combine over every (layer, row, query head).  decode_tile_tokens() is the
// tile height TOK of the kernel for that element type (tiles per page =
// ceil(P / TOK); the host plan and the tensor map's box must use the same
// one as the kernel); decode_max_warps() the
// number of co-resident warps the decode kernel can keep on the device.
// Split-decode state -> bf16 output: out[r][d] = o / l (0 where l = 0), for
// n_rows rows of D + 4 floats.
cudaError_t launch_state_finish(const float *state, int64_t n_rows, int head_dim, __nv_bfloat16 *out,
                                cudaStream_t s);
cudaError_t launch_decode(int head_dim, int group, bool fp8, const DecodeParams &p, const CUtensorMap &pool_map,
                          cudaStream_t s);
// Tensor map of a cache pool for the decode kernel: a 2-D bf16 tensor of
// head_dim columns and n_layers*2*n_pages*n_kv_heads*page_size rows, boxes of
// 64 columns x decode_tile_tokens(head_dim, fp8) rows, 128-byte swizzle.
cudaError_t make_pool_tensor_map(CUtensorMap *out, void *pool, int head_dim, bool fp8, uint64_t rows);
// A rank-`rank` bf16 tensor map (no swizzle, zero fill out of bounds): dims
// innermost first, byte strides of dims 1.., box extents per dim.
cudaError_t encode_tensor_map(CUtensorMap *out, int rank, void *base, const cuuint64_t *dims,
                              const cuuint64_t *strides, const cuuint32_t *box);
cudaError_t launch_combine(int head_dim, int group, const DecodeParams &p, cudaStream_t s);
bool decode_supported(int head_dim, int group, bool fp8 = false);
int decode_tile_tokens(int head_dim, bool fp8);
int decode_max_warps(int head_dim, int group, bool fp8, int n_sm);

// ------------------------------------- runtime.cu <-> noalloc.cu interface --
// Read-only view of a cache's geometry and device buffers (runtime.cu fills
// it; noalloc.cu reads it).  One definition here, included by both files.
struct CacheShape {
    int32_t n_layers, n_kv_heads, head_dim, page_size, n_pages, max_seqs, max_pages, device, n_sm;
    int32_t kv_dtype;
    float k_scale, v_scale;
    uint8_t *pool;
    int32_t *page_table, *page_fill;
    DevStatus *status;
    const CUtensorMap *pool_map;
};
bool cache_shape(const kvg_cache *c, CacheShape *out);
int32_t cache_seq_pages(const kvg_cache *c, int32_t seq);
kvg_status cache_plan_decode(const kvg_cache *c, int32_t layer, const int32_t *seq_ids, int32_t B,
                             std::vector<DecodeParams> *plan, int64_t *max_units);
void set_last_error(const char *msg);
// Looks up the device address of the allocation-free decode's static scratch
// on the current device (once per device) and so makes the module that
// holds it resident there; called by kvg_cache_create with the cache's
// device current.  Returns cudaSuccess or the lookup's error.
cudaError_t noalloc_prepare_device(int device);

// ------------------------------------------------------------ PTX helpers --
#ifdef __CUDACC__
__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
                 : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ uint64_t global_timer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Bounded wait on an mbarrier phase: gives up after limit_ns of wall time
// (default ~2 s) and returns false; the caller records KVG_ERR_DEVICE_CHECK
// in its status word and unwinds instead of hanging the GPU.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity,
                                                  uint64_t limit_ns = 2000000000ull) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    for (uint32_t it = 0;; ++it) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((it & 255u) == 255u && global_timer_ns() - t0 > limit_ns) return false;
    }
}

// Bulk (non-tensor) asynchronous copy global -> this CTA's shared memory,
// completing `bytes` of transaction count on `bar`.  dst/src 16-byte aligned,
// bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes,
                                         uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
            "r"(smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

// 2-D tensor copy (TMA) of one box at column x, row y of `map` into this
// CTA's shared memory, completing its bytes on `bar`.  x * 2 bytes must be a
// multiple of 16 (callers use multiples of 64 columns).
__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, int32_t x, int32_t y,
                                            uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
            "r"(smem_addr(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar))
        : "memory");
}

// 4-D tensor copy (TMA) of one box at coordinates (x, y, z, w) of `map`.
// x * element size must be a multiple of 16 bytes (callers pass x = 0).
__device__ __forceinline__ void tma_load_4d(void *dst, const CUtensorMap *map, int32_t x, int32_t y, int32_t z,
                                            int32_t w, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5}], [%6];" ::
            "r"(smem_addr(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(w), "r"(smem_addr(bar))
        : "memory");
}

// Bulk (non-tensor) asynchronous copy of this CTA's shared memory to global
// memory, tracked by the bulk async-group of the issuing thread.  dst/src
// 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_s2g(void *dst, const void *src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(smem_addr(src)),
                 "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// Waits until at most N of the thread's bulk groups still read shared memory.
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
// Waits until at most N of the thread's bulk groups are still incomplete.
template <int N>
__device__ __forceinline__ void bulk_wait() {
    asm volatile("cp.async.bulk.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void fence_proxy_async_shared() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void record_error(DevStatus *st, int32_t code, int32_t detail) {
    if (st && atomicCAS(&st->err, 0, code) == 0) st->err_detail = detail;
}
#endif

}  // namespace kvg

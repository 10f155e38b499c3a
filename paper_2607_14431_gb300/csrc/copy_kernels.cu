// copy_kernels.cu — the byte-moving kernels of the graft path.
//
//  graft_kernel<ROT>: own-position graft (Sec. 3.2) copies block pages into
//    the cache pages a sequence was given; with ROT != 0 the valid key rows
//    are re-based by an offset (Sec. 4.2) on the way.  Work unit = one chunk
//    of one page; the grid strides over all units so a single launch covers
//    every layer, K and V.  Loads and stores are 16-byte vectors with the
//    streaming cache hint (the data is touched once).
//  append_kernel: the "fresh" write of prefill-shaped rows into slots.
//  gather_kernel: deposit, cache pages -> block pages, zeroing padding rows.
#include <atomic>

#include "common.cuh"

namespace kvg {

namespace {

constexpr int kCopyThreads = 512;
constexpr int kCopyUnroll = 8;
constexpr int kRotUnroll = 4;

__device__ __forceinline__ void copy_chunk(uint8_t *__restrict__ dst, const uint8_t *__restrict__ src,
                                           int bytes) {
    const uint4 *s = reinterpret_cast<const uint4 *>(src);
    uint4 *d = reinterpret_cast<uint4 *>(dst);
    const int nvec = bytes >> 4;
    for (int base = threadIdx.x; base < nvec; base += kCopyThreads * kCopyUnroll) {
        uint4 r[kCopyUnroll];
#pragma unroll
        for (int u = 0; u < kCopyUnroll; ++u) {
            const int i = base + u * kCopyThreads;
            if (i < nvec) r[u] = __ldcs(s + i);
        }
#pragma unroll
        for (int u = 0; u < kCopyUnroll; ++u) {
            const int i = base + u * kCopyThreads;
            if (i < nvec) __stcs(d + i, r[u]);
        }
    }
}

__device__ __forceinline__ void unpack8(const uint4 &v, float *f) {
    const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&v);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 t = __bfloat1622float2(h[i]);
        f[2 * i] = t.x;
        f[2 * i + 1] = t.y;
    }
}

__device__ __forceinline__ uint4 pack8(const float *f) {
    uint4 v;
    __nv_bfloat162 *h = reinterpret_cast<__nv_bfloat162 *>(&v);
#pragma unroll
    for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
    return v;
}

// Rotation of the pair (a, b) by the angle whose cosine/sine are (c, s):
// a' = a c - b s, b' = a s + b c, in fp32 with a fixed operation order.
__device__ __forceinline__ void rot(float a, float b, float c, float s, float &ra, float &rb) {
    ra = __fmaf_rn(a, c, __fmul_rn(-b, s));
    rb = __fmaf_rn(a, s, __fmul_rn(b, c));
}

// cos/sin of a re-basing: from the launch's parameters (one graft per
// launch) or from a table in global memory (a batch of grafts).
// load<N>(i0, c, s) gives cos and sin of pairs i0 .. i0 + N - 1 (N = 4 or 8,
// i0 a multiple of N).
struct ParamTrig {
    const GraftParams &p;
    template <int N>
    __device__ __forceinline__ void load(int i0, float *c, float *s) const {
#pragma unroll
        for (int e = 0; e < N; ++e) {
            c[e] = p.cosv[i0 + e];
            s[e] = p.sinv[i0 + e];
        }
    }
};
struct TableTrig {
    const float *cs;  // cos[half] then sin[half], 16-byte aligned, half a multiple of 4
    int half;
    template <int N>
    __device__ __forceinline__ void load(int i0, float *c, float *s) const {
        const float4 *c4 = reinterpret_cast<const float4 *>(cs + i0);
        const float4 *s4 = reinterpret_cast<const float4 *>(cs + half + i0);
#pragma unroll
        for (int q = 0; q < N / 4; ++q) {
            const float4 x = __ldg(c4 + q), y = __ldg(s4 + q);
            c[4 * q] = x.x, c[4 * q + 1] = x.y, c[4 * q + 2] = x.z, c[4 * q + 3] = x.w;
            s[4 * q] = y.x, s[4 * q + 1] = y.y, s[4 * q + 2] = y.z, s[4 * q + 3] = y.w;
        }
    }
};

// Key chunk re-based by delta: rows of head_dim elements; half-split pairs
// (i, i + D/2) live in two 16-byte vectors of the same row, interleaved pairs
// (2i, 2i+1) inside one vector.  Rows whose token index is >= n_tokens are
// padding and are copied unchanged.
template <int ROT, class Trig>
__device__ __forceinline__ void rotate_chunk(uint8_t *__restrict__ dst, const uint8_t *__restrict__ src,
                                             int bytes, int64_t first_row_in_page, int64_t page_token0,
                                             int head_dim, int page_size, int64_t n_tokens, const Trig &trig) {
    const int D = head_dim;
    const int vec_per_row = D >> 3;
    const int rows = bytes / (2 * D);
    const uint4 *s4 = reinterpret_cast<const uint4 *>(src);
    uint4 *d4 = reinterpret_cast<uint4 *>(dst);
    // Rows of the page at or past n_valid are padding (only a block's last
    // page has any); the chunk's rows are (r0 + rr) mod P, rr < rows.
    const int P = page_size;
    const int64_t nv = n_tokens - page_token0;
    const int n_valid = nv < P ? (int)nv : P;
    const int r0 = (int)(first_row_in_page % P);
    if (ROT == 1) {
        // item = (row, pair chunk c < D/16): the 16-byte vectors c and c + D/16
        // of the row; kRotUnroll items per thread loaded before any is stored
        const int half_vecs = vec_per_row >> 1;  // D/16: a power of two
        const int hv_shift = __ffs(half_vecs) - 1;
        const int n_items = rows * half_vecs;
        for (int base = threadIdx.x; base < n_items; base += kCopyThreads * kRotUnroll) {
            uint4 lo[kRotUnroll], hi[kRotUnroll];
#pragma unroll
            for (int u = 0; u < kRotUnroll; ++u) {
                const int it = base + u * kCopyThreads;
                if (it < n_items) {
                    const int rr = it >> hv_shift;
                    const int lo_i = rr * vec_per_row + (it & (half_vecs - 1));
                    lo[u] = __ldcs(s4 + lo_i);
                    hi[u] = __ldcs(s4 + lo_i + half_vecs);
                }
            }
#pragma unroll
            for (int u = 0; u < kRotUnroll; ++u) {
                const int it = base + u * kCopyThreads;
                if (it < n_items) {
                    const int rr = it >> hv_shift;
                    const int c = it & (half_vecs - 1);
                    const int lo_i = rr * vec_per_row + c;
                    if (n_valid == P || (r0 + rr) % P < n_valid) {
                        float a[8], b[8], ra[8], rb[8], cv[8], sv[8];
                        unpack8(lo[u], a);
                        unpack8(hi[u], b);
                        trig.template load<8>(c * 8, cv, sv);
#pragma unroll
                        for (int e = 0; e < 8; ++e) rot(a[e], b[e], cv[e], sv[e], ra[e], rb[e]);
                        __stcs(d4 + lo_i, pack8(ra));
                        __stcs(d4 + lo_i + half_vecs, pack8(rb));
                    } else {
                        __stcs(d4 + lo_i, lo[u]);
                        __stcs(d4 + lo_i + half_vecs, hi[u]);
                    }
                }
            }
        }
    } else {
        const int vr_shift = __ffs(vec_per_row) - 1;  // D/8: a power of two
        const int n_items = rows * vec_per_row;
        for (int it = threadIdx.x; it < n_items; it += kCopyThreads) {
            const int rr = it >> vr_shift;
            const int c = it & (vec_per_row - 1);
            const uint4 x = __ldcs(s4 + it);
            if (n_valid == P || (r0 + rr) % P < n_valid) {
                float f[8], g[8], cv[4], sv[4];
                unpack8(x, f);
                trig.template load<4>(c * 4, cv, sv);
#pragma unroll
                for (int e = 0; e < 4; ++e) rot(f[2 * e], f[2 * e + 1], cv[e], sv[e], g[2 * e], g[2 * e + 1]);
                __stcs(d4 + it, pack8(g));
            } else {
                __stcs(d4 + it, x);
            }
        }
    }
}

template <int ROT>
__global__ void __launch_bounds__(kCopyThreads) graft_kernel(const GraftParams p) {
    const int64_t P = p.page_size;
    graft_metadata(p);
    const uint64_t page_bytes = p.page_bytes;
    const int cpp = (int)(page_bytes / (uint64_t)p.chunk_bytes);
    const int64_t n_units = (int64_t)p.n_layers * 2 * p.npb * cpp;
    const int row_bytes = 2 * p.head_dim;
    for (int64_t unit = blockIdx.x; unit < n_units; unit += gridDim.x) {
        const int64_t page_u = unit / cpp;
        const int chunk = (int)(unit - page_u * cpp);
        const int64_t lkv = page_u / p.npb;
        const int jj = (int)(page_u - lkv * p.npb);
        const uint64_t off = (uint64_t)chunk * (uint64_t)p.chunk_bytes;
        const uint8_t *src = p.src + ((uint64_t)lkv * p.block_pages + p.page_base + jj) * page_bytes + off;
        uint8_t *dst = p.pool + ((uint64_t)lkv * p.pool_pages + p.pids.pid[jj]) * page_bytes + off;
        if (ROT == 0 || (lkv & 1)) {
            copy_chunk(dst, src, p.chunk_bytes);
        } else {
            rotate_chunk<ROT>(dst, src, p.chunk_bytes, (int64_t)(off / row_bytes),
                              (int64_t)(p.page_base + jj) * P, p.head_dim, p.page_size, p.n_tokens, ParamTrig{p});
        }
    }
}

// One warp per (layer, K/V, token) row: the row's Hkv*D*2 source bytes are
// contiguous ([L][n][Hkv][D] input); head h goes to row `row` of head h's
// [P][D] slab in the token's page.  Index arithmetic is per row, not per
// vector; each lane keeps up to kAppendUnroll 16-byte loads in flight.
constexpr int kAppendThreads = 256;
constexpr int kAppendUnroll = 8;

// Position tags, page-table entries and fill counts of one append launch.
__device__ __forceinline__ void append_metadata(const AppendParams &p) {
    const int64_t gtid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t gsz = (int64_t)gridDim.x * blockDim.x;
    const int64_t P = p.page_size;
    for (int64_t t = gtid; t < p.n; t += gsz) p.pos_row[p.slot0 + t] = p.pos[p.row0 + t];
    for (int64_t i = gtid; i < p.pids.n; i += gsz) {
        const int64_t pg = p.page0 + i;
        p.table_row[pg] = p.pids.pid[i];
        const int64_t f = (int64_t)p.slot0 + p.n - pg * P;
        p.fill_row[pg] = (int32_t)(f < P ? f : P);
    }
}

__global__ void __launch_bounds__(kAppendThreads) append_kernel(const AppendParams p) {
    const int64_t gtid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t gsz = (int64_t)gridDim.x * blockDim.x;
    const int64_t P = p.page_size;
    append_metadata(p);
    const int D = p.head_dim;
    const int vpr = D >> 3;                 // 16-byte vectors per head row
    const int vpt = p.n_kv_heads * vpr;     // vectors per token row
    const int lane = threadIdx.x & 31;
    const int64_t warp = gtid >> 5;
    const int64_t n_warps = gsz >> 5;
    const int64_t rows = (int64_t)p.n_layers * 2 * p.n;
    const int64_t head_stride_vec = P * D / 8;  // between heads of one page, in vectors
    for (int64_t r = warp; r < rows; r += n_warps) {
        const int64_t lkv = r / p.n;
        const int t = (int)(r - lkv * p.n);
        const int l = (int)(lkv >> 1), kv = (int)(lkv & 1);
        const uint4 *src = reinterpret_cast<const uint4 *>(
            (kv ? p.v : p.k) + ((int64_t)l * p.n_rows_total + p.row0 + t) * p.n_kv_heads * D);
        const int64_t s = (int64_t)p.slot0 + t;
        const int64_t pg = s / P;
        const int pid = p.pids.pid[pg - p.page0];
        const int64_t row = s - pg * P;
        uint4 *dst = reinterpret_cast<uint4 *>(
            reinterpret_cast<uint16_t *>(p.pool) +
            (((int64_t)lkv * p.pool_pages + pid) * p.n_kv_heads) * P * D + row * D);
        for (int base = lane; base < vpt; base += 32 * kAppendUnroll) {
            uint4 val[kAppendUnroll];
#pragma unroll
            for (int u = 0; u < kAppendUnroll; ++u) {
                const int i = base + 32 * u;
                if (i < vpt) val[u] = __ldcs(src + i);
            }
#pragma unroll
            for (int u = 0; u < kAppendUnroll; ++u) {
                const int i = base + 32 * u;
                if (i < vpt) {
                    const int h = i >> (__ffs(vpr) - 1), c = i & (vpr - 1);  // vpr = D/8, a power of two
                    __stcs(dst + h * head_stride_vec + c, val[u]);
                }
            }
        }
    }
}

// One warp per (layer, K/V, batch row): Hkv*D*2 contiguous source bytes to
// row `row` of each head's slab of the row's page.
// Bulk append with the copy engine of each SM (TMA) instead of its threads.
// A job is (layer, K|V, page, kv head, row chunk): a 4-D tensor copy gathers
// the job's rows of one kv head from k/v [L][n][Hkv][D] (token stride
// Hkv*D) into a shared-memory stage, where they already have the page's
// [rows][D] layout, and one bulk copy writes them to the page.  Lane 0 of
// the one-warp CTA keeps up to kTmaStagesMax stages in flight; the other lanes only
// write the metadata.  The SM's ALUs stay free for concurrent work (hashing).
// kTmaSmemBytes is the largest stage budget (KVG_APPEND_TMA_KB tunes it).
constexpr int kTmaStagesMax = 8;
constexpr uint32_t kTmaSmemBytes = 192 * 1024;

struct TmaJob {
    int32_t lkv, jj, h, row_lo, row_hi;  // rows [row_lo, row_hi) of page jj (launch-relative)
    int64_t tok;                          // source token (row of k/v) of row_lo
};

__device__ __forceinline__ TmaJob tma_job(const AppendParams &p, int64_t J, int chunks, int pbox) {
    TmaJob j;
    const int c = (int)(J % chunks);
    J /= chunks;
    j.h = (int32_t)(J % p.n_kv_heads);
    J /= p.n_kv_heads;
    j.jj = (int32_t)(J % p.pids.n);
    j.lkv = (int32_t)(J / p.pids.n);
    const int64_t P = p.page_size;
    const int64_t pg = p.page0 + j.jj;
    int64_t lo = (int64_t)p.slot0 - pg * P, hi = (int64_t)p.slot0 + p.n - pg * P;
    if (lo < (int64_t)c * pbox) lo = (int64_t)c * pbox;
    if (hi > (int64_t)(c + 1) * pbox) hi = (int64_t)(c + 1) * pbox;
    if (hi > P) hi = P;
    if (hi < lo) hi = lo;
    j.row_lo = (int32_t)lo;
    j.row_hi = (int32_t)hi;
    j.tok = (int64_t)p.row0 + pg * P + lo - p.slot0;
    return j;
}

__global__ void __launch_bounds__(32) append_tma_kernel(const AppendParams p,
                                                        const __grid_constant__ CUtensorMap kmap,
                                                        const __grid_constant__ CUtensorMap vmap,
                                                        DevStatus *status, int32_t pbox, int32_t n_stages,
                                                        uint64_t limit_ns) {
    extern __shared__ __align__(128) uint8_t stage_mem[];
    __shared__ __align__(8) uint64_t bars[kTmaStagesMax];
    append_metadata(p);
    if (threadIdx.x != 0) return;
    const int D = p.head_dim;
    const int64_t P = p.page_size;
    const int chunks = (int)((P + pbox - 1) / pbox);
    const int64_t n_jobs = (int64_t)p.n_layers * 2 * p.pids.n * p.n_kv_heads * chunks;
    if (blockIdx.x >= n_jobs) return;
    const int64_t K = (n_jobs - blockIdx.x + gridDim.x - 1) / gridDim.x;  // this CTA's jobs
    const uint32_t stage_bytes = (uint32_t)pbox * D * 2;
    for (int i = 0; i < n_stages; ++i) mbar_init(&bars[i], 1);
    fence_mbar_init();
    auto job = [&](int64_t k) { return tma_job(p, blockIdx.x + k * gridDim.x, chunks, pbox); };
    auto load = [&](int64_t k) {
        const TmaJob j = job(k);
        const int st = (int)(k % n_stages);
        if (j.row_hi == j.row_lo) {
            mbar_arrive(&bars[st]);
            return;
        }
        mbar_arrive_expect_tx(&bars[st], stage_bytes);
        tma_load_4d(stage_mem + (size_t)st * stage_bytes, (j.lkv & 1) ? &vmap : &kmap, 0, j.h, (int32_t)j.tok,
                    j.lkv >> 1, &bars[st]);
    };
    const int64_t pro = K < n_stages ? K : n_stages;
    for (int64_t k = 0; k < pro; ++k) load(k);
    int64_t loaded = pro;  // jobs [0, loaded) have a load issued
    int64_t k = 0;
    for (; k < K; ++k) {
        const int st = (int)(k % n_stages);
        if (!mbar_wait_bounded(&bars[st], (uint32_t)((k / n_stages) & 1), limit_ns)) {
            record_error(status, KVG_ERR_DEVICE_CHECK, 2);
            break;
        }
        const TmaJob j = job(k);
        if (j.row_hi > j.row_lo) {
            fence_proxy_async_shared();
            uint8_t *dst = p.pool + ((((uint64_t)j.lkv * p.pool_pages + (uint64_t)p.pids.pid[j.jj]) * p.n_kv_heads +
                                      j.h) * P + j.row_lo) * (uint64_t)D * 2;
            bulk_s2g(dst, stage_mem + (size_t)st * stage_bytes, (uint32_t)(j.row_hi - j.row_lo) * D * 2);
        }
        bulk_commit();
        // refill the previous job's stage once its store has read it
        if (k >= 1 && loaded < K) {
            bulk_wait_read<1>();
            load(loaded++);
        }
    }
    if (k < K) {
        // gave up: let the loads still in flight land before the CTA exits
        for (int64_t m = k + 1; m < loaded; ++m)
            mbar_wait_bounded(&bars[m % n_stages], (uint32_t)((m / n_stages) & 1), limit_ns);
    }
    bulk_wait<0>();
}

// ---- appends into an fp8 E4M3 cache (quantized KV blocks) ----------------
// Eight bf16 values -> their E4M3 codes: each value in fp32 times the fp32
// reciprocal of the scale (one rounding), rounded to nearest-even on the E4M3
// grid with saturation at +-448 (cvt.rn.satfinite); code i lands in byte i.
__device__ __forceinline__ uint2 e4m3x8(const uint4 x, float inv_scale) {
    const uint32_t w[4] = {x.x, x.y, x.z, x.w};
    uint32_t h[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float lo = __fmul_rn(__uint_as_float(w[i] << 16), inv_scale);
        const float hi = __fmul_rn(__uint_as_float(w[i] & 0xffff0000u), inv_scale);
        uint16_t c;
        asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(c) : "f"(hi), "f"(lo));
        h[i] = c;
    }
    return make_uint2(h[0] | (h[1] << 16), h[2] | (h[3] << 16));
}

// One warp per (layer, K/V, token) row, like append_kernel; 8 values per lane
// per step (16 bytes in, 8 bytes out).
__global__ void __launch_bounds__(kAppendThreads) append_e4m3_kernel(const AppendParams p) {
    const int64_t gtid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t gsz = (int64_t)gridDim.x * blockDim.x;
    const int64_t P = p.page_size;
    append_metadata(p);
    const int D = p.head_dim;
    const int gpr = D >> 3;               // 8-value groups per head row
    const int gpt = p.n_kv_heads * gpr;   // groups per token row
    const int lane = threadIdx.x & 31;
    const int64_t rows = (int64_t)p.n_layers * 2 * p.n;
    for (int64_t r = gtid >> 5; r < rows; r += gsz >> 5) {
        const int64_t lkv = r / p.n;
        const int t = (int)(r - lkv * p.n);
        const int l = (int)(lkv >> 1), kv = (int)(lkv & 1);
        const float inv = kv ? p.v_inv_scale : p.k_inv_scale;
        const uint4 *src = reinterpret_cast<const uint4 *>(
            (kv ? p.v : p.k) + ((int64_t)l * p.n_rows_total + p.row0 + t) * p.n_kv_heads * D);
        const int64_t s = (int64_t)p.slot0 + t;
        const int64_t pg = s / P;
        const int pid = p.pids.pid[pg - p.page0];
        const int64_t row = s - pg * P;
        uint2 *dst = reinterpret_cast<uint2 *>(p.pool + (((int64_t)lkv * p.pool_pages + pid) * p.n_kv_heads) * P * D +
                                               row * D);
        for (int base = lane; base < gpt; base += 32 * kAppendUnroll) {
            uint4 val[kAppendUnroll];  // the loads first, kAppendUnroll in flight
#pragma unroll
            for (int u = 0; u < kAppendUnroll; ++u)
                if (base + 32 * u < gpt) val[u] = __ldcs(src + base + 32 * u);
#pragma unroll
            for (int u = 0; u < kAppendUnroll; ++u) {
                const int i = base + 32 * u;
                if (i < gpt) {
                    const int h = i >> (__ffs(gpr) - 1), c = i & (gpr - 1);  // gpr = D/8, a power of two
                    __stcs(dst + h * (P * D / 8) + c, e4m3x8(val[u], inv));
                }
            }
        }
    }
}

__global__ void __launch_bounds__(kAppendThreads) append_batch_e4m3_kernel(const AppendBatchParams p) {
    const int64_t gtid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t gsz = (int64_t)gridDim.x * blockDim.x;
    const int64_t P = p.page_size;
    for (int64_t b = gtid; b < p.B; b += gsz) {
        const int64_t s = p.slot[b];
        const int64_t pg = s / P;
        p.positions[(int64_t)p.seq[b] * p.max_slots + s] = p.pos[b];
        p.page_table[(int64_t)p.seq[b] * p.max_pages + pg] = p.pid[b];
        p.page_fill[(int64_t)p.seq[b] * p.max_pages + pg] = (int32_t)(s - pg * P + 1);
    }
    const int D = p.head_dim;
    const int gpr = D >> 3;
    const int gpt = p.n_kv_heads * gpr;
    const int lane = threadIdx.x & 31;
    const int64_t rows = (int64_t)p.n_layers * 2 * p.B;
    for (int64_t r = gtid >> 5; r < rows; r += gsz >> 5) {
        const int64_t lkv = r / p.B;
        const int b = (int)(r - lkv * p.B);
        const int l = (int)(lkv >> 1), kv = (int)(lkv & 1);
        const float inv = kv ? p.v_inv_scale : p.k_inv_scale;
        const uint4 *src = reinterpret_cast<const uint4 *>((kv ? p.v : p.k) + ((int64_t)l * p.B + b) * p.n_kv_heads * D);
        const int64_t s = p.slot[b];
        const int64_t row = s - (s / P) * P;
        uint2 *dst = reinterpret_cast<uint2 *>(p.pool + (((int64_t)lkv * p.pool_pages + p.pid[b]) * p.n_kv_heads) * P * D +
                                               row * D);
        for (int base = lane; base < gpt; base += 32 * kAppendUnroll) {
            uint4 val[kAppendUnroll];  // the loads first, kAppendUnroll in flight
#pragma unroll
            for (int u = 0; u < kAppendUnroll; ++u)
                if (base + 32 * u < gpt) val[u] = __ldcs(src + base + 32 * u);
#pragma unroll
            for (int u = 0; u < kAppendUnroll; ++u) {
                const int i = base + 32 * u;
                if (i < gpt) {
                    const int h = i >> (__ffs(gpr) - 1), c = i & (gpr - 1);  // gpr = D/8, a power of two
                    __stcs(dst + h * (P * D / 8) + c, e4m3x8(val[u], inv));
                }
            }
        }
    }
}

__global__ void __launch_bounds__(kAppendThreads) append_batch_kernel(const AppendBatchParams p) {
    const int64_t gtid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t gsz = (int64_t)gridDim.x * blockDim.x;
    const int64_t P = p.page_size;
    for (int64_t b = gtid; b < p.B; b += gsz) {
        const int64_t s = p.slot[b];
        const int64_t pg = s / P;
        p.positions[(int64_t)p.seq[b] * p.max_slots + s] = p.pos[b];
        p.page_table[(int64_t)p.seq[b] * p.max_pages + pg] = p.pid[b];
        p.page_fill[(int64_t)p.seq[b] * p.max_pages + pg] = (int32_t)(s - pg * P + 1);
    }
    const int D = p.head_dim;
    const int vpr = D >> 3;
    const int vpt = p.n_kv_heads * vpr;
    const int lane = threadIdx.x & 31;
    const int64_t rows = (int64_t)p.n_layers * 2 * p.B;
    const int64_t head_stride_vec = P * D / 8;
    for (int64_t r = gtid >> 5; r < rows; r += gsz >> 5) {
        const int64_t lkv = r / p.B;
        const int b = (int)(r - lkv * p.B);
        const int l = (int)(lkv >> 1), kv = (int)(lkv & 1);
        const uint4 *src = reinterpret_cast<const uint4 *>((kv ? p.v : p.k) + ((int64_t)l * p.B + b) * p.n_kv_heads * D);
        const int64_t s = p.slot[b];
        const int64_t row = s - (s / P) * P;
        uint4 *dst = reinterpret_cast<uint4 *>(reinterpret_cast<uint16_t *>(p.pool) +
                                               (((int64_t)lkv * p.pool_pages + p.pid[b]) * p.n_kv_heads) * P * D +
                                               row * D);
        for (int i = lane; i < vpt; i += 32) {
            const int h = i >> (__ffs(vpr) - 1), c = i & (vpr - 1);  // vpr = D/8, a power of two
            __stcs(dst + h * head_stride_vec + c, __ldcs(src + i));
        }
    }
}

__global__ void __launch_bounds__(256) gather_kernel(const GatherParams p) {
    const int64_t P = p.page_size;
    const int64_t row_bytes = (int64_t)(p.page_bytes / ((uint64_t)p.n_kv_heads * P));
    const int64_t vpp = (int64_t)(p.page_bytes >> 4);
    const int64_t total = (int64_t)p.n_layers * 2 * p.npb * vpp;
    const int64_t gtid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t gsz = (int64_t)gridDim.x * blockDim.x;
    const int64_t tok0 = (int64_t)p.page_base * P;
    int64_t n_meta = (int64_t)p.npb * P;
    if (tok0 + n_meta > p.n_tokens) n_meta = p.n_tokens - tok0;
    if (p.src_pos)
        for (int64_t t = gtid; t < n_meta; t += gsz) p.dst_pos[t] = p.src_pos[t];
    for (int64_t idx = gtid; idx < total; idx += gsz) {
        const int64_t page_u = idx / vpp;
        const int64_t off = idx - page_u * vpp;
        const int64_t lkv = page_u / p.npb;
        const int64_t jj = page_u - lkv * p.npb;
        const int64_t row = ((off * 16) / row_bytes) % P;
        const int64_t tok = (p.page_base + jj) * P + row;
        uint4 val = make_uint4(0, 0, 0, 0);
        if (tok < p.n_tokens) {
            const uint4 *src = reinterpret_cast<const uint4 *>(
                p.pool + ((uint64_t)lkv * p.pool_pages + p.pids.pid[jj]) * p.page_bytes);
            val = __ldcs(src + off);
        }
        uint4 *dst = reinterpret_cast<uint4 *>(
            p.dst_pids.n ? p.dst + ((uint64_t)lkv * p.pool_pages + p.dst_pids.pid[jj]) * p.page_bytes
                         : p.dst + ((uint64_t)lkv * p.block_pages + p.page_base + jj) * p.page_bytes);
        dst[off] = val;
    }
}

__global__ void __launch_bounds__(256) alias_kernel(const AliasParams p) {
    const int64_t gtid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t gsz = (int64_t)gridDim.x * blockDim.x;
    const int64_t P = p.page_size;
    for (int64_t t = gtid; t < p.n_tokens; t += gsz) p.dst_pos[t] = p.src_pos[t];
    for (int64_t j = gtid; j < p.pids.n; j += gsz) {
        p.table_row[j] = p.pids.pid[j];
        const int64_t f = p.n_tokens - j * P;
        p.fill_row[j] = (int32_t)(f < P ? f : P);
    }
}

// One 4-byte load per `stride` bytes of [base, base + bytes): each load makes
// the GPU resolve the address translation of one host page, so a later graft
// that streams the block finds them resolved.  The values are discarded
// (sink is written only if the loads' xor hits a constant, and the launcher
// passes null).
__global__ void __launch_bounds__(256) touch_kernel(const uint8_t *base, uint64_t n_loads, uint32_t stride,
                                                    uint32_t *sink) {
    uint32_t acc = 0;
    for (uint64_t i = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; i < n_loads;
         i += (uint64_t)gridDim.x * blockDim.x)
        acc ^= __ldcv(reinterpret_cast<const uint32_t *>(base + i * stride));
    if (acc == 0x9e3779b9u && sink) *sink = acc;
}

__global__ void wait_selftest_kernel(DevStatus *status, uint64_t limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_mbar_init();
    }
    __syncthreads();
    // no thread arrives and no copy completes: phase 0 never completes
    const bool ok = mbar_wait_bounded(&bar, 0, limit_ns);
    if (!ok && threadIdx.x == 0) record_error(status, KVG_ERR_DEVICE_CHECK, 3);
}

__global__ void write_ints_kernel(const IntsParams p) {
    for (int i = threadIdx.x; i < p.vals.n; i += blockDim.x) p.dst[i] = p.vals.pid[i];
}

__global__ void write_header_kernel(const HeaderParams p) {
    const int i = threadIdx.x;
    if (i < 64) reinterpret_cast<uint32_t *>(p.dst)[i] = reinterpret_cast<const uint32_t *>(p.bytes)[i];
}

__global__ void reset_seq_kernel(int32_t *table_row, int32_t *fill_row, int32_t max_pages,
                                 int32_t *pos_row, int32_t max_slots) {
    const int64_t gtid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t gsz = (int64_t)gridDim.x * blockDim.x;
    for (int64_t j = gtid; j < max_pages; j += gsz) {
        table_row[j] = -1;
        fill_row[j] = 0;
    }
    for (int64_t s = gtid; s < max_slots; s += gsz) pos_row[s] = -1;
}

// ---- graft through shared-memory stages (HBM sources) ---------------------
// A persistent CTA per SM streams its units (chunks of block pages, as in
// graft_kernel) through a ring of shared-memory stages: thread 0 brings a
// unit in with one bulk copy (cp.async.bulk, mbarrier completion), the CTA
// re-rotates the valid key rows in place when the graft relocates, and
// thread 0 writes the stage to the cache page with one bulk copy.  The loads
// of later units are in flight meanwhile, so the copy does not depend on
// registers for its bytes in flight.  Rows, rounding and operation order of
// the rotation are those of rotate_chunk.
constexpr int kTmaGraftThreads = 256;

template <int ROT>
__device__ __forceinline__ void rotate_stage(uint8_t *stage, int bytes, int64_t first_row_in_page,
                                             int64_t page_token0, const GraftParams &p, const float *cs) {
    const int D = p.head_dim;
    const int vec_per_row = D >> 3;
    const int rows = bytes / (2 * D);
    uint4 *v4 = reinterpret_cast<uint4 *>(stage);
    const int P = p.page_size;
    const int64_t nv = p.n_tokens - page_token0;
    const int n_valid = nv < P ? (int)nv : P;
    const int r0 = (int)(first_row_in_page % P);
    if (ROT == 1) {
        const int half_vecs = vec_per_row >> 1;
        const int hv_shift = __ffs(half_vecs) - 1;
        const int n_items = rows * half_vecs;
        for (int it = threadIdx.x; it < n_items; it += blockDim.x) {
            const int rr = it >> hv_shift;
            if (n_valid < P && (r0 + rr) % P >= n_valid) continue;  // padding row: unchanged
            const int c = it & (half_vecs - 1);
            const int lo_i = rr * vec_per_row + c;
            float a[8], b[8], ra[8], rb[8];
            unpack8(v4[lo_i], a);
            unpack8(v4[lo_i + half_vecs], b);
#pragma unroll
            for (int e = 0; e < 8; ++e) rot(a[e], b[e], cs[c * 8 + e], cs[kMaxHalfDim + c * 8 + e], ra[e], rb[e]);
            v4[lo_i] = pack8(ra);
            v4[lo_i + half_vecs] = pack8(rb);
        }
    } else {
        const int vr_shift = __ffs(vec_per_row) - 1;
        const int n_items = rows * vec_per_row;
        for (int it = threadIdx.x; it < n_items; it += blockDim.x) {
            const int rr = it >> vr_shift;
            if (n_valid < P && (r0 + rr) % P >= n_valid) continue;
            const int c = it & (vec_per_row - 1);
            float f[8], g[8];
            unpack8(v4[it], f);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int i = c * 4 + e;
                rot(f[2 * e], f[2 * e + 1], cs[i], cs[kMaxHalfDim + i], g[2 * e], g[2 * e + 1]);
            }
            v4[it] = pack8(g);
        }
    }
}

template <int ROT>
__global__ void __launch_bounds__(kTmaGraftThreads) graft_tma_kernel(const GraftParams p, DevStatus *status,
                                                                     int32_t n_stages, uint64_t limit_ns) {
    extern __shared__ __align__(128) uint8_t stage_mem[];
    __shared__ __align__(8) uint64_t bars[kTmaStagesMax];
    __shared__ float cs[2 * kMaxHalfDim];
    graft_metadata(p);
    const uint64_t page_bytes = p.page_bytes;
    const uint32_t cb = (uint32_t)p.chunk_bytes;
    const int cpp = (int)(page_bytes / cb);
    const int64_t n_units = (int64_t)p.n_layers * 2 * p.npb * cpp;
    if ((int64_t)blockIdx.x >= n_units) return;  // the whole CTA
    const int64_t K = (n_units - blockIdx.x + gridDim.x - 1) / gridDim.x;  // this CTA's units
    if (ROT != 0)
        for (int i = threadIdx.x; i < p.head_dim / 2; i += blockDim.x) {
            cs[i] = p.cosv[i];
            cs[kMaxHalfDim + i] = p.sinv[i];
        }
    if (threadIdx.x == 0) {
        for (int i = 0; i < n_stages; ++i) mbar_init(&bars[i], 1);
        fence_mbar_init();
    }
    __syncthreads();
    struct Unit {
        const uint8_t *src;
        uint8_t *dst;
        int64_t lkv, jj;
        uint64_t off;
    };
    auto unit = [&](int64_t k) {
        const int64_t u = (int64_t)blockIdx.x + k * gridDim.x;
        const int64_t page_u = u / cpp;
        Unit r;
        r.off = (uint64_t)(u - page_u * cpp) * cb;
        r.lkv = page_u / p.npb;
        r.jj = page_u - r.lkv * p.npb;
        r.src = p.src + ((uint64_t)r.lkv * p.block_pages + p.page_base + r.jj) * page_bytes + r.off;
        r.dst = p.pool + ((uint64_t)r.lkv * p.pool_pages + p.pids.pid[r.jj]) * page_bytes + r.off;
        return r;
    };
    auto load = [&](int64_t k) {  // thread 0
        const int st = (int)(k % n_stages);
        mbar_arrive_expect_tx(&bars[st], cb);
        bulk_g2s(stage_mem + (size_t)st * cb, unit(k).src, cb, &bars[st]);
    };
    const int64_t pro = K < n_stages ? K : n_stages;
    if (threadIdx.x == 0)
        for (int64_t k = 0; k < pro; ++k) load(k);
    int64_t loaded = pro;  // thread 0's count of units whose load is issued
    int64_t k = 0;
    for (; k < K; ++k) {
        const int st = (int)(k % n_stages);
        const bool ok = mbar_wait_bounded(&bars[st], (uint32_t)((k / n_stages) & 1), limit_ns);
        if (__syncthreads_or(!ok)) {
            if (threadIdx.x == 0) record_error(status, KVG_ERR_DEVICE_CHECK, 3);
            break;
        }
        const Unit u = unit(k);
        uint8_t *stage = stage_mem + (size_t)st * cb;
        if (ROT != 0 && !(u.lkv & 1)) {
            rotate_stage<ROT>(stage, (int)cb, (int64_t)(u.off / (uint64_t)(2 * p.head_dim)),
                              (int64_t)(p.page_base + u.jj) * p.page_size, p, cs);
            fence_proxy_async_shared();  // this thread's writes, before the bulk copy reads them
            __syncthreads();
        }
        if (threadIdx.x == 0) {
            bulk_s2g(u.dst, stage, cb);
            bulk_commit();
            // refill the previous unit's stage once its store has read it
            if (k >= 1 && loaded < K) {
                bulk_wait_read<1>();
                load(loaded++);
            }
        }
    }
    if (threadIdx.x == 0) {
        if (k < K)  // gave up: let the loads still in flight land before the CTA exits
            for (int64_t m = k; m < loaded; ++m)
                mbar_wait_bounded(&bars[m % n_stages], (uint32_t)((m / n_stages) & 1), limit_ns);
        bulk_wait<0>();
    }
}

int grid_for(int64_t work_items, int per_block, int n_sm, int waves) {
    int64_t g = (work_items + per_block - 1) / per_block;
    const int64_t cap = (int64_t)n_sm * waves;
    if (g > cap) g = cap;
    if (g < 1) g = 1;
    return (int)g;
}

}  // namespace

// A batch of grafts in one launch: every block page of every graft is a job;
// a unit is a chunk of one (job, layer, K/V) page, so the batch keeps every
// SM busy to its end instead of draining after each graft.  ROT > 0: some
// grafts are re-based (their key chunks rotate with their own cos/sin table,
// as the single-graft kernels do; values and own-position grafts copy).
template <int ROT>
__global__ void __launch_bounds__(kCopyThreads) graft_batch_kernel(const GraftBatchParams p) {
    const uint64_t page_bytes = p.page_bytes;
    const int64_t cpp = (int64_t)(page_bytes / (uint64_t)p.chunk_bytes);
    const int64_t per_job = (int64_t)p.n_layers * 2 * cpp;
    const int64_t n_units = p.n_jobs * per_job;
    const int row_bytes = 2 * p.head_dim;
    for (int64_t unit = blockIdx.x; unit < n_units; unit += gridDim.x) {
        const int64_t jb = unit / per_job;
        const int64_t rem = unit - jb * per_job;
        const int64_t lkv = rem / cpp;
        const uint64_t off = (uint64_t)(rem - lkv * cpp) * (uint64_t)p.chunk_bytes;
        const GraftJob job = p.jobs[jb];
        const uint8_t *src = job.src + (uint64_t)lkv * job.block_pages * page_bytes + off;
        uint8_t *dst = p.pool + ((uint64_t)lkv * p.pool_pages + (uint64_t)job.pid) * page_bytes + off;
        const int32_t trig = ROT != 0 && !(lkv & 1) ? p.metas[job.meta].trig : -1;
        if (trig < 0) {
            copy_chunk(dst, src, p.chunk_bytes);
        } else {
            const int half = p.head_dim >> 1;
            rotate_chunk<ROT>(dst, src, p.chunk_bytes, (int64_t)(off / row_bytes), (int64_t)job.page * p.page_size,
                              p.head_dim, p.page_size, p.metas[job.meta].n_tokens,
                              TableTrig{p.trig + (int64_t)trig * 2 * half, half});
        }
    }
    // metadata last: the copies start at once and this fills the tail wave
    const int64_t P = p.page_size;
    const int64_t gtid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t gsz = (int64_t)gridDim.x * blockDim.x;
    for (int32_t g = 0; g < p.n_grafts; ++g) {
        const GraftMeta m = p.metas[g];
        for (int64_t t = gtid; t < m.n_tokens; t += gsz) m.dst_pos[t] = (int32_t)((int64_t)m.src_pos[t] + m.delta);
        for (int64_t j = gtid; j < m.npb; j += gsz) {
            m.table_row[j] = p.jobs[m.first_job + j].pid;
            const int64_t f = m.n_tokens - j * P;
            m.fill_row[j] = (int32_t)(f < P ? f : P);
        }
    }
}

cudaError_t launch_graft_batch(const GraftBatchParams &p, int n_sm, cudaStream_t s, int max_ctas, int rotate) {
    const int64_t units = p.n_jobs * p.n_layers * 2 * (int64_t)(p.page_bytes / p.chunk_bytes);
    int grid = grid_for(units, 1, n_sm, 4);
    if (max_ctas > 0 && grid > max_ctas) grid = max_ctas;
    if (rotate == 0)
        graft_batch_kernel<0><<<grid, kCopyThreads, 0, s>>>(p);
    else if (rotate == 1)
        graft_batch_kernel<1><<<grid, kCopyThreads, 0, s>>>(p);
    else
        graft_batch_kernel<2><<<grid, kCopyThreads, 0, s>>>(p);
    count_launches(1);
    return cudaGetLastError();
}

// Shared-memory stage budget of graft_tma_kernel (KVG_GRAFT_TMA_KB, 0 turns
// the staged graft off).  Three 64 KiB stages measured best: the 31B
// relocation 2.38 ms against 3.08 ms with two, and 32 KiB units (four or six
// stages) 2.51-2.56 ms, 16 KiB units 4.3 ms.
static int graft_tma_budget() {
    static const int kb = [] {
        const char *e = getenv("KVG_GRAFT_TMA_KB");
        return e ? atoi(e) : 192;
    }();
    return kb;
}

// The staged graft for HBM sources: one persistent CTA per SM; -1 if the
// unit does not fit twice in the stage budget (then graft_kernel runs).
static cudaError_t launch_graft_tma(const GraftParams &p, DevStatus *status, int n_sm, cudaStream_t s) {
    const int64_t units = (int64_t)p.n_layers * 2 * p.npb * (int64_t)(p.page_bytes / p.chunk_bytes);
    const uint32_t budget = (uint32_t)std::min(graft_tma_budget(), 200) * 1024u;
    int n_stages = (int)(budget / (uint32_t)p.chunk_bytes);
    if (n_stages > kTmaStagesMax) n_stages = kTmaStagesMax;
    if (n_stages < 2 || units == 0) return cudaErrorNotSupported;
    static std::atomic<bool> attr_set[kMaxDevices][3];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return cudaErrorNotSupported;
    const size_t smem = (size_t)n_stages * p.chunk_bytes;
    const int r = p.rotate;
    if (!attr_set[dev][r].load()) {
        cudaError_t e = r == 0 ? cudaFuncSetAttribute(graft_tma_kernel<0>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                      200 * 1024)
                      : r == 1 ? cudaFuncSetAttribute(graft_tma_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                      200 * 1024)
                               : cudaFuncSetAttribute(graft_tma_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                      200 * 1024);
        if (e != cudaSuccess) return e;
        attr_set[dev][r].store(true);
    }
    const int grid = grid_for(units, 1, n_sm, 1);
    const uint64_t limit_ns = 2000000000ull;
    if (r == 0)
        graft_tma_kernel<0><<<grid, kTmaGraftThreads, smem, s>>>(p, status, n_stages, limit_ns);
    else if (r == 1)
        graft_tma_kernel<1><<<grid, kTmaGraftThreads, smem, s>>>(p, status, n_stages, limit_ns);
    else
        graft_tma_kernel<2><<<grid, kTmaGraftThreads, smem, s>>>(p, status, n_stages, limit_ns);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_graft_copy(const GraftParams &p, int n_sm, cudaStream_t s, int max_ctas, DevStatus *status) {
    // HBM sources go through shared-memory stages; a host-mapped source is
    // read by a capped grid of graft_kernel (the host link bounds it)
    if (max_ctas == 0 && status && graft_tma_budget() > 0) {
        const cudaError_t e = launch_graft_tma(p, status, n_sm, s);
        if (e != cudaErrorNotSupported) return e;
    }
    const int64_t units = (int64_t)p.n_layers * 2 * p.npb * (int64_t)(p.page_bytes / p.chunk_bytes);
    int grid = grid_for(units, 1, n_sm, 4);
    if (max_ctas > 0 && grid > max_ctas) grid = max_ctas;
    if (p.rotate == 0)
        graft_kernel<0><<<grid, kCopyThreads, 0, s>>>(p);
    else if (p.rotate == 1)
        graft_kernel<1><<<grid, kCopyThreads, 0, s>>>(p);
    else
        graft_kernel<2><<<grid, kCopyThreads, 0, s>>>(p);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_append(const AppendParams &p, int n_sm, cudaStream_t s) {
    const int64_t rows = 2ll * p.n_layers * p.n;  // one warp each
    static const int ctas_per_sm = env_knob("KVG_APPEND_CTAS_PER_SM", 2);
    append_kernel<<<grid_for(rows, kAppendThreads / 32, n_sm, ctas_per_sm), kAppendThreads, 0, s>>>(p);
    count_launches(1);
    return cudaGetLastError();
}

// Rows per tensor copy: a page's rows, at most 256 (the box limit) and at
// most 48 KiB of one kv head's rows, so that at least four stages fit.
int32_t append_tma_rows(int32_t page_size, int32_t head_dim) {
    int32_t r = page_size < 256 ? page_size : 256;
    const int32_t cap = 49152 / (2 * head_dim);
    return r < cap ? r : cap;
}

cudaError_t launch_append_tma(const AppendParams &p, DevStatus *status, int n_sm, cudaStream_t s) {
    const int pbox = append_tma_rows(p.page_size, p.head_dim);
    const int D = p.head_dim;
    const uint32_t stage_bytes = (uint32_t)pbox * D * 2;
    // 96 KiB of stages per SM keeps HBM busy (6.5 TB/s alone) while leaving
    // room beside it for concurrent hashing; 192 KiB starves a concurrent
    // graft + verify of bandwidth, 64 KiB starves the append.
    static const uint32_t smem_budget =
        (uint32_t)std::min(std::max(env_knob("KVG_APPEND_TMA_KB", 96), 16), 192) * 1024u;
    int n_stages = (int)(smem_budget / stage_bytes);
    if (n_stages > kTmaStagesMax) n_stages = kTmaStagesMax;
    if (n_stages < 2) return cudaErrorNotSupported;
    // k and v: 4-D bf16 tensors (D, Hkv, n_rows_total, L); box (D, 1, pbox, 1)
    CUtensorMap maps[2];
    const cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)p.n_kv_heads, (cuuint64_t)p.n_rows_total,
                                (cuuint64_t)p.n_layers};
    const cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)p.n_kv_heads * D * 2,
                                   (cuuint64_t)p.n_rows_total * p.n_kv_heads * D * 2};
    const cuuint32_t box[4] = {(cuuint32_t)D, 1, (cuuint32_t)pbox, 1};
    const uint16_t *src[2] = {p.k, p.v};
    for (int i = 0; i < 2; ++i)
        if (encode_tensor_map(&maps[i], 4, const_cast<uint16_t *>(src[i]), dims, strides, box) != cudaSuccess)
            return cudaErrorNotSupported;
    // the shared-memory attribute is per device
    static std::atomic<bool> attr_set[kMaxDevices];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return cudaErrorNotSupported;
    if (!attr_set[dev].load()) {
        cudaError_t e = cudaFuncSetAttribute(append_tma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)kTmaSmemBytes);
        if (e != cudaSuccess) return e;
        attr_set[dev].store(true);
    }
    const int chunks = (p.page_size + pbox - 1) / pbox;
    const int64_t jobs = 2ll * p.n_layers * p.pids.n * p.n_kv_heads * chunks;
    const int grid = grid_for(jobs, 1, n_sm, 1);
    append_tma_kernel<<<grid, 32, (size_t)n_stages * stage_bytes, s>>>(p, maps[0], maps[1], status, pbox, n_stages,
                                                                      2000000000ull);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_append_e4m3(const AppendParams &p, int n_sm, cudaStream_t s) {
    const int64_t rows = 2ll * p.n_layers * p.n;  // one warp each
    static const int ctas_per_sm = env_knob("KVG_APPEND_CTAS_PER_SM", 2);
    append_e4m3_kernel<<<grid_for(rows, kAppendThreads / 32, n_sm, ctas_per_sm), kAppendThreads, 0, s>>>(p);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_append_batch_e4m3(const AppendBatchParams &p, int n_sm, cudaStream_t s) {
    const int64_t rows = 2ll * p.n_layers * p.B;
    append_batch_e4m3_kernel<<<grid_for(rows, kAppendThreads / 32, n_sm, 8), kAppendThreads, 0, s>>>(p);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_append_batch(const AppendBatchParams &p, int n_sm, cudaStream_t s) {
    const int64_t rows = 2ll * p.n_layers * p.B;
    append_batch_kernel<<<grid_for(rows, kAppendThreads / 32, n_sm, 8), kAppendThreads, 0, s>>>(p);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_gather(const GatherParams &p, int n_sm, cudaStream_t s) {
    const int64_t items = 2ll * p.n_layers * p.npb * (int64_t)(p.page_bytes / 16);
    gather_kernel<<<grid_for(items, 256, n_sm, 8), 256, 0, s>>>(p);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_alias(const AliasParams &p, int n_sm, cudaStream_t s) {
    alias_kernel<<<grid_for(p.n_tokens > p.pids.n ? p.n_tokens : p.pids.n, 256, n_sm, 1), 256, 0, s>>>(p);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_touch(const uint8_t *base, uint64_t bytes, uint32_t stride, int n_sm, cudaStream_t s) {
    const uint64_t n_loads = bytes / stride + (bytes % stride >= 4 ? 1 : 0);  // every load fits in [base, +bytes)
    if (n_loads == 0) return cudaSuccess;
    touch_kernel<<<grid_for((int64_t)n_loads, 256, n_sm, 2), 256, 0, s>>>(base, n_loads, stride, nullptr);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_wait_selftest(DevStatus *status, uint64_t limit_ns, cudaStream_t s) {
    wait_selftest_kernel<<<1, 32, 0, s>>>(status, limit_ns);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_write_ints(const IntsParams &p, cudaStream_t s) {
    write_ints_kernel<<<1, 256, 0, s>>>(p);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_write_header(const HeaderParams &p, cudaStream_t s) {
    write_header_kernel<<<1, 64, 0, s>>>(p);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_reset_seq(int32_t *table_row, int32_t *fill_row, int32_t max_pages,
                             int32_t *pos_row, int32_t max_slots, cudaStream_t s) {
    const int64_t items = max_pages > max_slots ? max_pages : max_slots;
    reset_seq_kernel<<<grid_for(items, 256, 152, 1), 256, 0, s>>>(table_row, fill_row, max_pages,
                                                                   pos_row, max_slots);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace kvg

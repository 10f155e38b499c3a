// attn_kernels.cu — paged GQA decode attention (Sec. 3.2 / Sec. 4.3: one new
// query token attends to every row of the grafted context).
//
// Persistent, load-balanced ("stream-K") design.  The work of a call is a
// global list of tiles: unit (layer, batch row, kv head) owns its sequence's
// pages in logical order, each page split into ceil(P / TOK) tiles of TOK
// rows.  The kernel launches W one-warp CTAs, all co-resident; warp w takes
// the contiguous range [w*T/W, (w+1)*T/W) of the T tiles, so every warp gets
// the same share and there is no tail wave.  A warp is an independent
// pipeline: lane 0 issues bulk asynchronous copies (cp.async.bulk, completion
// on an mbarrier, bounded wait) of the K and V rows of a tile into a
// STAGES-deep shared-memory ring, STAGES-1 tiles ahead, across unit
// boundaries; the 32 lanes consume them:
//   - lanes form 4 groups of 8; a group owns every 4th row of the tile and
//     each lane 8*D/64 dimensions in 16-byte chunks j, j+8, ... (a group's 8
//     lanes read one contiguous 128-byte span: no bank conflicts);
//   - q.k partial sums are all-reduced over the group with 3 xor shuffles;
//   - each group keeps an online-softmax state (running max m, sum l, fp32
//     output o) for all G query heads of the kv head (K/V read once) and
//     rescales o only when the running max grows (the skipped factor is
//     exactly 1);
//   - when the warp leaves a unit it merges its 4 groups in a fixed order and
//     writes the unit's partial (o, m, l) to slot unit + w.
// The combine kernel merges, for each unit, the partials of the warps that
// covered it, in warp order.  Every reduction order is a function of logical
// token indices and of (T, W) only — never of physical page ids — so results
// are bitwise reproducible and identical for grafted and freshly written rows.
// G = 2 fills 2 of 16 rows of an MMA tile; at ~2 flop per byte the CUDA cores
// keep up with HBM, so the contraction stays on the FMA pipe.
#include <math.h>

#include "common.cuh"

namespace kvg {

namespace {

template <int D>
struct TileShape;
template <>
struct TileShape<64> {
    static constexpr int TOK = 32, STAGES = 3;
};
template <>
struct TileShape<128> {
    static constexpr int TOK = 32, STAGES = 2;
};
template <>
struct TileShape<256> {
    static constexpr int TOK = 16, STAGES = 2;
};

template <int D>
struct Cfg {
    static constexpr int TOK = TileShape<D>::TOK;
    static constexpr int STAGES = TileShape<D>::STAGES;
    static constexpr int NCH = D / 64;              // 16-byte chunks per lane per row
    static constexpr int TILE_BYTES = TOK * D * 2;  // one K (or V) tile
    static constexpr int STAGE_BYTES = 2 * TILE_BYTES;
    static constexpr int RING_BYTES = STAGES * STAGE_BYTES;
    static constexpr int SMEM = RING_BYTES + STAGES * (8 + 4);
};

__device__ __forceinline__ void unpack8(const uint4 &v, float *f) {
    const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&v);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 t = __bfloat1622float2(h[i]);
        f[2 * i] = t.x;
        f[2 * i + 1] = t.y;
    }
}

// Weighted sum x*a + y*b with an operation order that is symmetric in the two
// operands, so both partners of a shuffle merge compute identical bits.
__device__ __forceinline__ float wsum(float x, float a, float y, float b) {
    return __fadd_rn(__fmul_rn(x, a), __fmul_rn(y, b));
}

// Position of global tile t: unit (lr, b, g) and tile index within the unit.
struct TilePos {
    int lr, b, g;
    int64_t unit;
    int tile;
};

__device__ __forceinline__ TilePos locate(const DecodeParams &p, int64_t t) {
    const int64_t sumT = p.rows.pref_tiles[p.B];
    const int64_t per_layer = (int64_t)p.n_kv_heads * sumT;
    TilePos r;
    r.lr = (int)(t / per_layer);
    const int64_t rem = t - (int64_t)r.lr * per_layer;
    int lo = 0, hi = p.B - 1;  // largest b with Hkv * pref[b] <= rem
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if ((int64_t)p.n_kv_heads * p.rows.pref_tiles[mid] <= rem)
            lo = mid;
        else
            hi = mid - 1;
    }
    r.b = lo;
    const int64_t r2 = rem - (int64_t)p.n_kv_heads * p.rows.pref_tiles[lo];
    const int Tb = p.rows.pref_tiles[lo + 1] - p.rows.pref_tiles[lo];
    r.g = (int)(r2 / Tb);
    r.tile = (int)(r2 - (int64_t)r.g * Tb);
    r.unit = ((int64_t)r.lr * p.B + r.b) * p.n_kv_heads + r.g;
    return r;
}

__device__ __forceinline__ int64_t warp_start(int64_t w, int64_t T, int64_t W) { return w * T / W; }

template <int D, int G>
__global__ void __launch_bounds__(32) decode_kernel(const DecodeParams p) {
    using C = Cfg<D>;
    constexpr int TOK = C::TOK, STAGES = C::STAGES, NCH = C::NCH;
    constexpr int TPG = TOK / 4;  // rows per lane group per tile
    extern __shared__ __align__(128) uint8_t smem[];

    const int lane = threadIdx.x;
    const int grp = lane >> 3, lj = lane & 7;
    const int64_t w = blockIdx.x;
    const int64_t t0 = warp_start(w, p.n_tiles, p.n_warps);
    const int64_t t1 = warp_start(w + 1, p.n_tiles, p.n_warps);
    const int P = p.page_size;
    const int tpp = (P + TOK - 1) / TOK;

    uint8_t *ring = smem;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + C::RING_BYTES);
    int *vrs = reinterpret_cast<int *>(smem + C::RING_BYTES + STAGES * 8);
    if (lane == 0) {
#pragma unroll
        for (int s = 0; s < STAGES; ++s) mbar_init(&bars[s], 1);
        fence_mbar_init();
    }
    __syncwarp();

    const int64_t plane_elems = p.pool_pages * (int64_t)p.n_kv_heads * P * D;
    const __nv_bfloat16 *poolh = reinterpret_cast<const __nv_bfloat16 *>(p.pool);

    auto issue = [&](int64_t t, int stg) {  // lane 0
        const TilePos tp = locate(p, t);
        const int seq = p.rows.seq[tp.b];
        const int jj = tp.tile / tpp;
        const int k = tp.tile - jj * tpp;
        const int fill = p.page_fill[(int64_t)seq * p.max_pages + jj];
        const int pid = p.page_table[(int64_t)seq * p.max_pages + jj];
        int vr = fill - k * TOK;
        vr = vr < 0 ? 0 : (vr > TOK ? TOK : vr);
        if (vr > 0 && (pid < 0 || pid >= p.pool_pages)) {
            record_error(p.status, KVG_ERR_DEVICE_CHECK, 1);
            vr = 0;
        }
        vrs[stg] = vr;
        uint64_t *bar = &bars[stg];
        if (vr > 0) {
            const uint32_t bytes = (uint32_t)vr * D * 2;
            mbar_arrive_expect_tx(bar, 2 * bytes);
            const int l = p.layer0 + tp.lr;
            const __nv_bfloat16 *ks = poolh + (int64_t)(2 * l) * plane_elems +
                                      ((int64_t)pid * p.n_kv_heads + tp.g) * P * D + (int64_t)k * TOK * D;
            uint8_t *dst = ring + stg * C::STAGE_BYTES;
            bulk_g2s(dst, ks, bytes, bar);
            bulk_g2s(dst + C::TILE_BYTES, ks + plane_elems, bytes, bar);
        } else {
            mbar_arrive(bar);
        }
    };

    float qf[G][NCH][8];
    float m[G], lsum[G], o[G][NCH][8];
    int64_t cur_unit = -1;

    auto flush = [&](int64_t unit) {
        // merge the 4 lane groups: (0,1),(2,3) then (01,23)
#pragma unroll
        for (int off = 8; off <= 16; off <<= 1) {
#pragma unroll
            for (int h = 0; h < G; ++h) {
                const float mo = __shfl_xor_sync(0xffffffffu, m[h], off);
                const float lo = __shfl_xor_sync(0xffffffffu, lsum[h], off);
                const float mn = fmaxf(m[h], mo);
                const float a = m[h] == -INFINITY ? 0.f : exp2f(m[h] - mn);
                const float bb = mo == -INFINITY ? 0.f : exp2f(mo - mn);
                lsum[h] = wsum(lsum[h], a, lo, bb);
#pragma unroll
                for (int c = 0; c < NCH; ++c)
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const float oo = __shfl_xor_sync(0xffffffffu, o[h][c][e], off);
                        o[h][c][e] = wsum(o[h][c][e], a, oo, bb);
                    }
                m[h] = mn;
            }
        }
        const int64_t slot = unit + w;
        if (lane < 8) {
#pragma unroll
            for (int h = 0; h < G; ++h) {
                float *dst = p.part_o + (slot * G + h) * D;
#pragma unroll
                for (int c = 0; c < NCH; ++c) {
                    float4 *d4 = reinterpret_cast<float4 *>(dst + 8 * (lj + 8 * c));
                    d4[0] = make_float4(o[h][c][0], o[h][c][1], o[h][c][2], o[h][c][3]);
                    d4[1] = make_float4(o[h][c][4], o[h][c][5], o[h][c][6], o[h][c][7]);
                }
            }
            if (lane == 0)
#pragma unroll
                for (int h = 0; h < G; ++h) p.part_ml[slot * G + h] = make_float2(m[h], lsum[h]);
        }
    };

    auto begin = [&](const TilePos &tp) {
        const __nv_bfloat16 *qrow =
            p.q + ((int64_t)(tp.lr * p.q_row_stride_b + p.b0 + tp.b) * p.n_q_heads + tp.g * G) * D;
#pragma unroll
        for (int h = 0; h < G; ++h) {
            m[h] = -INFINITY;
            lsum[h] = 0.f;
#pragma unroll
            for (int c = 0; c < NCH; ++c) {
                const uint4 v = *reinterpret_cast<const uint4 *>(qrow + h * D + 8 * (lj + 8 * c));
                unpack8(v, qf[h][c]);
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    qf[h][c][e] *= p.qscale;
                    o[h][c][e] = 0.f;
                }
            }
        }
    };

    if (lane == 0) {
        for (int i = 0; i < STAGES && t0 + i < t1; ++i) issue(t0 + i, i);
    }

    bool alive = true;
    int64_t unit_end = t0;  // first tile past the current unit
    for (int64_t t = t0; t < t1; ++t) {
        const int64_t i = t - t0;
        const int stg = (int)(i % STAGES);
        const uint32_t par = (uint32_t)((i / STAGES) & 1);
        if (t >= unit_end) {
            const TilePos tp = locate(p, t);
            if (cur_unit >= 0) flush(cur_unit);
            begin(tp);
            cur_unit = tp.unit;
            unit_end = t - tp.tile + (p.rows.pref_tiles[tp.b + 1] - p.rows.pref_tiles[tp.b]);
        }
        const bool ok = mbar_wait_bounded(&bars[stg], par);
        if (!__all_sync(0xffffffffu, ok)) {
            if (lane == 0) record_error(p.status, KVG_ERR_DEVICE_CHECK, 2);
            alive = false;
            break;
        }
        const int vr = vrs[stg];
        if (vr > 0) {
            const __nv_bfloat16 *Ks = reinterpret_cast<const __nv_bfloat16 *>(ring + stg * C::STAGE_BYTES);
            const __nv_bfloat16 *Vs = Ks + TOK * D;
            float s[TPG][G];
#pragma unroll
            for (int i4 = 0; i4 < TPG; ++i4) {
                const int ti = i4 * 4 + grp;
                float acc[G];
#pragma unroll
                for (int h = 0; h < G; ++h) acc[h] = 0.f;
                if (ti < vr) {
#pragma unroll
                    for (int c = 0; c < NCH; ++c) {
                        const uint4 kv = *reinterpret_cast<const uint4 *>(Ks + ti * D + 8 * (lj + 8 * c));
                        float kf[8];
                        unpack8(kv, kf);
#pragma unroll
                        for (int h = 0; h < G; ++h)
#pragma unroll
                            for (int e = 0; e < 8; ++e) acc[h] = fmaf(qf[h][c][e], kf[e], acc[h]);
                    }
                }
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    acc[h] += __shfl_xor_sync(0xffffffffu, acc[h], 4);
                    acc[h] += __shfl_xor_sync(0xffffffffu, acc[h], 2);
                    acc[h] += __shfl_xor_sync(0xffffffffu, acc[h], 1);
                    s[i4][h] = ti < vr ? acc[h] : -INFINITY;
                }
            }
#pragma unroll
            for (int h = 0; h < G; ++h) {
                float mt = s[0][h];
#pragma unroll
                for (int i4 = 1; i4 < TPG; ++i4) mt = fmaxf(mt, s[i4][h]);
                if (mt > m[h]) {
                    const float alpha = exp2f(m[h] - mt);
                    lsum[h] *= alpha;
#pragma unroll
                    for (int c = 0; c < NCH; ++c)
#pragma unroll
                        for (int e = 0; e < 8; ++e) o[h][c][e] *= alpha;
                    m[h] = mt;
                }
            }
#pragma unroll
            for (int i4 = 0; i4 < TPG; ++i4) {
                const int ti = i4 * 4 + grp;
                if (ti < vr) {
                    float pw[G];
#pragma unroll
                    for (int h = 0; h < G; ++h) {
                        pw[h] = exp2f(s[i4][h] - m[h]);
                        lsum[h] += pw[h];
                    }
#pragma unroll
                    for (int c = 0; c < NCH; ++c) {
                        const uint4 vv = *reinterpret_cast<const uint4 *>(Vs + ti * D + 8 * (lj + 8 * c));
                        float vf[8];
                        unpack8(vv, vf);
#pragma unroll
                        for (int h = 0; h < G; ++h)
#pragma unroll
                            for (int e = 0; e < 8; ++e) o[h][c][e] = fmaf(pw[h], vf[e], o[h][c][e]);
                    }
                }
            }
        }
        __syncwarp();
        if (lane == 0 && t + STAGES < t1) issue(t + STAGES, stg);
    }
    if (!alive) {
        // a copy never completed: wait (bounded) on every stage once more so
        // no copy is left writing this CTA's shared memory, then record an
        // empty partial for the unit in progress
        if (lane == 0)
            for (int s = 0; s < STAGES; ++s) (void)mbar_wait_bounded(&bars[s], 0);
#pragma unroll
        for (int h = 0; h < G; ++h) {
            m[h] = -INFINITY;
            lsum[h] = 0.f;
#pragma unroll
            for (int c = 0; c < NCH; ++c)
#pragma unroll
                for (int e = 0; e < 8; ++e) o[h][c][e] = 0.f;
        }
    }
    if (cur_unit >= 0) flush(cur_unit);
}

// Largest warp index whose range starts at or before tile t.
__device__ __forceinline__ int64_t warp_of(int64_t t, int64_t T, int64_t W) { return ((t + 1) * W - 1) / T; }

template <int D>
__global__ void __launch_bounds__(D) combine_kernel(const DecodeParams p) {
    const int h = blockIdx.x, b = blockIdx.y, lr = blockIdx.z;
    const int G = p.n_q_heads / p.n_kv_heads;
    const int g = h / G, hh = h - g * G;
    const int d = threadIdx.x;
    const int64_t unit = ((int64_t)lr * p.B + b) * p.n_kv_heads + g;
    const int64_t sumT = p.rows.pref_tiles[p.B];
    const int64_t Tb = p.rows.pref_tiles[b + 1] - p.rows.pref_tiles[b];
    float L = 0.f, O = 0.f;
    if (Tb > 0) {
        const int64_t T = p.n_tiles, W = p.n_warps;
        const int64_t first = (int64_t)lr * p.n_kv_heads * sumT + (int64_t)p.n_kv_heads * p.rows.pref_tiles[b] +
                              (int64_t)g * Tb;
        const int64_t last = first + Tb - 1;
        const int64_t wa = warp_of(first, T, W), wb = warp_of(last, T, W);
        float M = -INFINITY;
        for (int64_t w = wa; w <= wb; ++w) {
            if (warp_start(w + 1, T, W) == warp_start(w, T, W)) continue;  // empty range
            M = fmaxf(M, p.part_ml[(unit + w) * G + hh].x);
        }
        for (int64_t w = wa; w <= wb; ++w) {
            if (warp_start(w + 1, T, W) == warp_start(w, T, W)) continue;
            const float2 ml = p.part_ml[(unit + w) * G + hh];
            if (ml.x == -INFINITY) continue;
            const float sc = exp2f(ml.x - M);
            L = __fmaf_rn(ml.y, sc, L);
            O = __fmaf_rn(p.part_o[((unit + w) * G + hh) * D + d], sc, O);
        }
    }
    const float r = L > 0.f ? __fdiv_rn(O, L) : 0.f;
    p.out[((int64_t)(lr * p.q_row_stride_b + p.b0 + b) * p.n_q_heads + h) * D + d] = __float2bfloat16_rn(r);
}

template <int D, int G>
struct DecodeLaunch {
    static int max_blocks_per_sm() {
        static int cached = -1;
        if (cached < 0) {
            if (cudaFuncSetAttribute(decode_kernel<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     Cfg<D>::SMEM) != cudaSuccess)
                return 0;
            int n = 0;
            if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, decode_kernel<D, G>, 32, Cfg<D>::SMEM) !=
                cudaSuccess)
                return 0;
            cached = n;
        }
        return cached;
    }
    static cudaError_t run(const DecodeParams &p, cudaStream_t s) {
        if (max_blocks_per_sm() <= 0) return cudaErrorInvalidConfiguration;
        if (p.n_warps <= 0 || p.n_tiles <= 0) return cudaSuccess;
        decode_kernel<D, G><<<p.n_warps, 32, Cfg<D>::SMEM, s>>>(p);
        count_launches(1);
        return cudaGetLastError();
    }
};

}  // namespace

bool decode_supported(int head_dim, int group) {
    if (head_dim != 64 && head_dim != 128 && head_dim != 256) return false;
    if (group != 1 && group != 2 && group != 4 && group != 8) return false;
    return head_dim * group <= 512;
}

int decode_tile_tokens(int head_dim) {
    switch (head_dim) {
        case 64: return Cfg<64>::TOK;
        case 128: return Cfg<128>::TOK;
        case 256: return Cfg<256>::TOK;
    }
    return 0;
}

#define KVG_DECODE_CASES(X) \
    X(64, 1) X(64, 2) X(64, 4) X(64, 8) X(128, 1) X(128, 2) X(128, 4) X(256, 1) X(256, 2)

int decode_max_warps(int head_dim, int group, int n_sm) {
#define KVG_CASE(DD, GG) \
    if (head_dim == DD && group == GG) return DecodeLaunch<DD, GG>::max_blocks_per_sm() * n_sm;
    KVG_DECODE_CASES(KVG_CASE)
#undef KVG_CASE
    return 0;
}

cudaError_t launch_decode(int head_dim, int group, const DecodeParams &p, cudaStream_t s) {
#define KVG_CASE(DD, GG) \
    if (head_dim == DD && group == GG) return DecodeLaunch<DD, GG>::run(p, s);
    KVG_DECODE_CASES(KVG_CASE)
#undef KVG_CASE
    return cudaErrorInvalidValue;
}

cudaError_t launch_combine(int head_dim, int group, const DecodeParams &p, cudaStream_t s) {
    (void)group;
    dim3 grid(p.n_q_heads, p.B, p.n_layers_run);
    switch (head_dim) {
        case 64: combine_kernel<64><<<grid, 64, 0, s>>>(p); count_launches(1); break;
        case 128: combine_kernel<128><<<grid, 128, 0, s>>>(p); count_launches(1); break;
        case 256: combine_kernel<256><<<grid, 256, 0, s>>>(p); count_launches(1); break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace kvg

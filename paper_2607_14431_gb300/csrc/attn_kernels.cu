// attn_kernels.cu — split-K paged GQA decode attention (Sec. 3.2 / Sec. 4.3:
// one new query token attends to every row of the grafted context).
//
// Grid (split, kv head g, layer x batch row).  A CTA owns a contiguous range
// of the sequence's logical pages for one (layer, sequence, kv head) and all
// G = Hq / Hkv query heads that read that kv head, so every K/V byte is read
// from HBM once per step.  Each warp is an independent pipeline: its lane 0
// issues bulk asynchronous copies (cp.async.bulk, completion on an mbarrier)
// of TOK-row K and V tiles into the warp's own STAGES-deep shared-memory ring,
// and all 32 lanes consume them:
//   - lanes form 4 groups of 8; a group owns TOK/4 rows of the tile and each
//     lane of the group 8*NCH of the D dimensions (16-byte chunks j, j+8, ...
//     so a group's 8 lanes read one contiguous 128-byte span: no bank
//     conflicts);
//   - q.k partial sums are all-reduced over the group with 3 xor shuffles;
//   - each group keeps its own online-softmax state (running max m, sum l,
//     output o in fp32) and rescales o only when the running max grows
//     (multiplying by exp2(0) = 1 would change nothing, so this is exact);
//   - at the end the 4 groups, then the warps, then the splits are merged in a
//     fixed order.
// Every reduction order depends only on logical token indices, never on the
// physical page ids, so the output is bitwise reproducible and identical for
// grafted and freshly written rows.  G = 2 (the workloads here) fills 2 of 16
// rows of an MMA tile; at ~2 flop per byte the CUDA cores keep up with HBM.
#include <math.h>

#include "common.cuh"

namespace kvg {

namespace {

template <int D>
struct TileShape;
template <>
struct TileShape<64> {
    static constexpr int TOK = 32, STAGES = 3, WARPS = 4;
};
template <>
struct TileShape<128> {
    static constexpr int TOK = 32, STAGES = 3, WARPS = 4;
};
template <>
struct TileShape<256> {
    static constexpr int TOK = 16, STAGES = 3, WARPS = 4;
};

template <int D>
struct Cfg {
    static constexpr int TOK = TileShape<D>::TOK;
    static constexpr int STAGES = TileShape<D>::STAGES;
    static constexpr int WARPS = TileShape<D>::WARPS;
    static constexpr int NCH = D / 64;            // 16-byte chunks per lane per row
    static constexpr int TILE_BYTES = TOK * D * 2;  // one K (or V) tile
    static constexpr int STAGE_BYTES = 2 * TILE_BYTES;
    static constexpr int RING_BYTES = WARPS * STAGES * STAGE_BYTES;
    static constexpr int SMEM = RING_BYTES + WARPS * STAGES * (8 + 4);
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

template <int D, int G>
__global__ void __launch_bounds__(Cfg<D>::WARPS * 32, 1) decode_split_kernel(const DecodeParams p) {
    using C = Cfg<D>;
    constexpr int TOK = C::TOK, STAGES = C::STAGES, WARPS = C::WARPS, NCH = C::NCH;
    constexpr int TPG = TOK / 4;  // rows per lane group per tile
    extern __shared__ __align__(128) uint8_t smem[];

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int grp = lane >> 3, lj = lane & 7;
    const int split = blockIdx.x, g = blockIdx.y;
    const int lr = blockIdx.z / p.B, b = blockIdx.z - lr * p.B;
    const int l = p.layer0 + lr;
    const int seq = p.rows.seq[b];
    const int np = p.rows.npages[b];
    const int P = p.page_size;
    const int tpp = (P + TOK - 1) / TOK;
    const int j0 = split * p.pages_per_split;
    int j1 = j0 + p.pages_per_split;
    if (j1 > np) j1 = np;
    const int ntiles = j1 > j0 ? (j1 - j0) * tpp : 0;
    const int my_n = warp < ntiles ? (ntiles - warp + WARPS - 1) / WARPS : 0;

    uint8_t *ring = smem + warp * STAGES * C::STAGE_BYTES;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + C::RING_BYTES) + warp * STAGES;
    int *vrs = reinterpret_cast<int *>(smem + C::RING_BYTES + WARPS * STAGES * 8) + warp * STAGES;

    if (lane == 0) {
#pragma unroll
        for (int s = 0; s < STAGES; ++s) mbar_init(&bars[s], 1);
        fence_mbar_init();
    }
    __syncwarp();

    const int64_t plane_elems = p.pool_pages * (int64_t)p.n_kv_heads * P * D;
    const __nv_bfloat16 *poolh = reinterpret_cast<const __nv_bfloat16 *>(p.pool);
    const int32_t *trow = p.page_table + (int64_t)seq * p.max_pages;
    const int32_t *frow = p.page_fill + (int64_t)seq * p.max_pages;

    auto issue = [&](int i) {  // lane 0: tile i of this warp's sequence
        const int t = warp + i * WARPS;
        const int jj = j0 + t / tpp;
        const int k = t - (t / tpp) * tpp;
        const int stg = i % STAGES;
        const int fill = frow[jj];
        const int pid = trow[jj];
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
            const __nv_bfloat16 *ks = poolh + (int64_t)(2 * l) * plane_elems +
                                      ((int64_t)pid * p.n_kv_heads + g) * P * D + (int64_t)k * TOK * D;
            uint8_t *dst = ring + stg * C::STAGE_BYTES;
            bulk_g2s(dst, ks, bytes, bar);
            bulk_g2s(dst + C::TILE_BYTES, ks + plane_elems, bytes, bar);
        } else {
            mbar_arrive(bar);
        }
    };

    // query rows of this kv head's group, pre-scaled by scale*log2(e)
    float qf[G][NCH][8];
    {
        const __nv_bfloat16 *qrow =
            p.q + ((int64_t)(lr * p.q_row_stride_b + p.b0 + b) * p.n_q_heads + g * G) * D;
#pragma unroll
        for (int h = 0; h < G; ++h)
#pragma unroll
            for (int c = 0; c < NCH; ++c) {
                const uint4 v = *reinterpret_cast<const uint4 *>(qrow + h * D + 8 * (lj + 8 * c));
                unpack8(v, qf[h][c]);
#pragma unroll
                for (int e = 0; e < 8; ++e) qf[h][c][e] *= p.qscale;
            }
    }

    float m[G], lsum[G], o[G][NCH][8];
#pragma unroll
    for (int h = 0; h < G; ++h) {
        m[h] = -INFINITY;
        lsum[h] = 0.f;
#pragma unroll
        for (int c = 0; c < NCH; ++c)
#pragma unroll
            for (int e = 0; e < 8; ++e) o[h][c][e] = 0.f;
    }

    if (lane == 0) {
        const int pre = my_n < STAGES ? my_n : STAGES;
        for (int i = 0; i < pre; ++i) issue(i);
    }

    bool alive = true;
    for (int i = 0; i < my_n; ++i) {
        const int stg = i % STAGES;
        const uint32_t par = (uint32_t)((i / STAGES) & 1);
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
        if (lane == 0 && i + STAGES < my_n) issue(i + STAGES);
    }
    if (!alive) {
        // drain this warp's copies still in flight (bounded) before the CTA
        // can exit, then report an empty partial
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

    // merge the 4 lane groups of the warp: (0,1),(2,3) then (01,23)
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

    // merge the warps through shared memory (ring no longer in use), in order
    __syncthreads();
    float *red_o = reinterpret_cast<float *>(smem);                    // [WARPS][G][D]
    float2 *red_ml = reinterpret_cast<float2 *>(smem + WARPS * G * D * 4);  // [WARPS][G]
    if (lane < 8) {
#pragma unroll
        for (int h = 0; h < G; ++h)
#pragma unroll
            for (int c = 0; c < NCH; ++c)
#pragma unroll
                for (int e = 0; e < 8; ++e) red_o[(warp * G + h) * D + 8 * (lj + 8 * c) + e] = o[h][c][e];
        if (lane == 0)
#pragma unroll
            for (int h = 0; h < G; ++h) red_ml[warp * G + h] = make_float2(m[h], lsum[h]);
    }
    __syncthreads();
    const int64_t unit = ((int64_t)lr * p.B + b) * p.n_kv_heads + g;
    for (int idx = threadIdx.x; idx < G * D; idx += WARPS * 32) {
        const int h = idx / D, d = idx - h * D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < WARPS; ++w) M = fmaxf(M, red_ml[w * G + h].x);
        float L = 0.f, O = 0.f;
#pragma unroll
        for (int w = 0; w < WARPS; ++w) {
            const float2 ml = red_ml[w * G + h];
            const float sc = ml.x == -INFINITY ? 0.f : exp2f(ml.x - M);
            L = __fmaf_rn(ml.y, sc, L);
            O = __fmaf_rn(red_o[(w * G + h) * D + d], sc, O);
        }
        const int64_t part = (unit * p.n_splits + split) * G + h;
        p.part_o[part * D + d] = O;
        if (d == 0) p.part_ml[part] = make_float2(M, L);
    }
}

template <int D>
__global__ void __launch_bounds__(D) combine_kernel(const CombineParams p) {
    const int h = blockIdx.x, b = blockIdx.y, lr = blockIdx.z;
    const int G = p.n_q_heads / p.n_kv_heads;
    const int g = h / G, hh = h - g * G;
    const int d = threadIdx.x;
    const int64_t unit = ((int64_t)lr * p.B + b) * p.n_kv_heads + g;
    float M = -INFINITY;
    for (int s = 0; s < p.n_splits; ++s) M = fmaxf(M, p.part_ml[(unit * p.n_splits + s) * G + hh].x);
    float L = 0.f, O = 0.f;
    for (int s = 0; s < p.n_splits; ++s) {
        const int64_t part = (unit * p.n_splits + s) * G + hh;
        const float2 ml = p.part_ml[part];
        if (ml.x == -INFINITY) continue;
        const float sc = exp2f(ml.x - M);
        L = __fmaf_rn(ml.y, sc, L);
        O = __fmaf_rn(p.part_o[part * D + d], sc, O);
    }
    const float r = L > 0.f ? __fdiv_rn(O, L) : 0.f;
    p.out[((int64_t)(lr * p.q_row_stride_b + p.b0 + b) * p.n_q_heads + h) * D + d] = __float2bfloat16_rn(r);
}

template <int D, int G>
cudaError_t launch_decode_t(const DecodeParams &p, cudaStream_t s) {
    static bool configured = false;  // attribute set once per instantiation
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(decode_split_kernel<D, G>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<D>::SMEM);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    dim3 grid(p.n_splits, p.n_kv_heads, p.n_layers_run * p.B);
    decode_split_kernel<D, G><<<grid, Cfg<D>::WARPS * 32, Cfg<D>::SMEM, s>>>(p);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace

bool decode_supported(int head_dim, int group) {
    if (head_dim != 64 && head_dim != 128 && head_dim != 256) return false;
    if (group != 1 && group != 2 && group != 4 && group != 8) return false;
    return head_dim * group <= 512;
}

size_t decode_smem_bytes(int head_dim) {
    switch (head_dim) {
        case 64: return Cfg<64>::SMEM;
        case 128: return Cfg<128>::SMEM;
        case 256: return Cfg<256>::SMEM;
    }
    return 0;
}

cudaError_t launch_decode(int head_dim, int group, const DecodeParams &p, cudaStream_t s) {
#define KVG_CASE(DD, GG) \
    if (head_dim == DD && group == GG) return launch_decode_t<DD, GG>(p, s);
    KVG_CASE(64, 1) KVG_CASE(64, 2) KVG_CASE(64, 4) KVG_CASE(64, 8)
    KVG_CASE(128, 1) KVG_CASE(128, 2) KVG_CASE(128, 4)
    KVG_CASE(256, 1) KVG_CASE(256, 2)
#undef KVG_CASE
    return cudaErrorInvalidValue;
}

cudaError_t launch_combine(int head_dim, int group, const CombineParams &p, int n_layers_run, int B,
                           cudaStream_t s) {
    (void)group;
    dim3 grid(p.n_q_heads, B, n_layers_run);
    switch (head_dim) {
        case 64: combine_kernel<64><<<grid, 64, 0, s>>>(p); count_launches(1); break;
        case 128: combine_kernel<128><<<grid, 128, 0, s>>>(p); count_launches(1); break;
        case 256: combine_kernel<256><<<grid, 256, 0, s>>>(p); count_launches(1); break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace kvg

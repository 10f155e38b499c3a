// attn_kernels.cu — paged GQA decode attention (Sec. 3.2 / Sec. 4.3: one new
// query token attends to every row of the grafted context).
//
// Persistent, load-balanced ("stream-K") design.  The work of a call is a
// global list of tiles: unit (layer, batch row, kv head) owns its sequence's
// pages in logical order, each page split into ceil(P / TOK) tiles of TOK
// rows.  The kernel launches W one-warp CTAs, all co-resident; warp w takes
// the contiguous range [w*T/W, (w+1)*T/W) of the T tiles, so every warp gets
// the same share and there is no tail wave.  A warp is an independent
// pipeline over a STAGES-deep shared-memory ring: for each tile lane 0 issues
// 2-D tensor copies (TMA, cp.async.bulk.tensor, completion on an mbarrier,
// bounded wait) of the K and V rows as boxes of 64 columns x TOK rows with the
// 128-byte swizzle, so the 8-row ldmatrix reads below hit 8 different bank
// groups; value rows past the page's fill are zeroed after arrival and the
// scores of those rows are masked; on a sliding-window layer the unit starts
// at the window's first tile and the rows before the window are masked too.
//
// The contractions run on the tensor cores with mma.sync m16n8k16 (bf16 in,
// fp32 accumulate).  Each tile is bandwidth-bound (~2 flop per byte at G = 2),
// so the point is not FLOPs but instruction count: a 16-row sub-tile costs
// D/16 MMAs for q.k and D/16 for p.v instead of ~1,400 scalar instructions.
//   S[16 tok][8] = K[16][D] . Q^T[D][8]  (A = K rows, B = the G query heads of
//                                          the kv head, padded with zeros)
//   O^T[D][8] += V^T[D][16] . P^T[16][8] (A = V rows, transposed by ldmatrix;
//                                          B = the bf16-rounded weights P)
// The online softmax is per head in fp32: scores are scaled by scale*log2(e),
// the running max m is reduced across the 8 lanes holding a head's column, O
// is rescaled only when m grows (the skipped factor is exactly 1), and the
// running sum l adds the same bf16-rounded weights the MMA uses.  When the
// warp leaves a unit it writes that unit's partial (o, m, l) to slot unit + w;
// the combine kernel merges, for each unit, the partials of the warps that
// covered it, in warp order.  Every order of operations is a function of
// logical token indices and of (T, W) only — never of physical page ids — so
// results are bitwise reproducible and identical for grafted and freshly
// written rows.
#include <cuda_fp16.h>
#include <math.h>

#include <atomic>

#include "common.cuh"

namespace kvg {

namespace {

template <int D>
struct TileShape;
template <>
struct TileShape<64> {
    static constexpr int TOK = 64, STAGES = 3;
};
// Tile rows and ring stages per head_dim (compile-time knobs, measured on
// the GB300 decode of the 31B and 12B shapes): head_dim 128, 64 rows x 2
// stages, 3 warps per SM (7.11 ms for batch 8 x 65,536 rows x 12 layers,
// against 7.36 with 32 x 3 and 7.22 with 16 x 2); head_dim 256, 16 rows x 3
// stages, 4 warps per SM (32 x 2 ties; 16 x 2, 16 x 4, 32 x 3, 64 x 2 slower).
#ifndef KVG_DEC128_TOK
#define KVG_DEC128_TOK 64
#endif
#ifndef KVG_DEC128_STAGES
#define KVG_DEC128_STAGES 2
#endif
#ifndef KVG_DEC256_TOK
#define KVG_DEC256_TOK 16
#endif
#ifndef KVG_DEC256_STAGES
#define KVG_DEC256_STAGES 3
#endif
template <>
struct TileShape<128> {
    static constexpr int TOK = KVG_DEC128_TOK, STAGES = KVG_DEC128_STAGES;
};
template <>
struct TileShape<256> {
    static constexpr int TOK = KVG_DEC256_TOK, STAGES = KVG_DEC256_STAGES;
};

// fp8 tiles (knobs for head_dim 128 and 256).
#ifndef KVG_FP8_128_TOK
#define KVG_FP8_128_TOK 32
#endif
#ifndef KVG_FP8_256_TOK
#define KVG_FP8_256_TOK 16
#endif
#ifndef KVG_FP8_STAGES
#define KVG_FP8_STAGES 2
#endif
template <int D>
struct Fp8TileShape {
    static constexpr int TOK = D == 256 ? KVG_FP8_256_TOK : (D == 128 ? KVG_FP8_128_TOK : 64);
    static constexpr int STAGES = KVG_FP8_STAGES;
};

// FP8: the pool holds E4M3 codes; TMA brings boxes of 128 one-byte columns.
// Keys go from the fp8 tile straight into MMA fragments; values are expanded
// into a 16-bit staging tile with the bf16 layout (for ldmatrix.trans).
// fp8 tiles carry half the bytes; two stages per warp leave room for 8
// warps per SM (the decode is latency-bound per warp: more warps, not deeper
// rings, keep HBM busy; three stages gave 0.77 of the copy peak, two 0.97)
template <int D, bool FP8 = false>
struct Cfg {
    static constexpr int TOK = FP8 ? Fp8TileShape<D>::TOK : TileShape<D>::TOK;
    static constexpr int STAGES = FP8 ? Fp8TileShape<D>::STAGES : TileShape<D>::STAGES;
    static constexpr int NB = D / 64;                  // 64-column 16-bit boxes per K (or V) tile
    static constexpr int BOX = TOK * 128;              // bytes of one box (TOK rows x 128 B)
    static constexpr int NB8 = FP8 ? D / 128 : 0;      // 128-column fp8 boxes per K (or V) tile
    static constexpr int STAGE_BYTES = FP8 ? 2 * NB8 * BOX : 2 * NB * BOX;  // K boxes then V boxes
    static constexpr int RING_BYTES = STAGES * STAGE_BYTES;
    static constexpr int STAGING_BYTES = FP8 ? NB * BOX : 0;  // the current tile's values, expanded
    static constexpr int SMEM = RING_BYTES + STAGING_BYTES + STAGES * (8 + 4 + 4) + 1024;  // + alignment slack
    static constexpr int KS = D / 16;                  // k-steps of q.k, m-tiles of p.v
    static constexpr int SUB = TOK / 16;               // 16-row sub-tiles per tile
    static_assert(BOX % 1024 == 0, "a swizzle atom is 8 rows of 128 bytes");
    static_assert(!FP8 || D % 128 == 0, "fp8 tiles are whole 128-byte boxes");
};

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

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// D += A(16x16, row) . B(16x8, col), bf16 (F16: fp16) inputs, fp32 accumulators.
template <bool F16>
__device__ __forceinline__ void mma16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                      uint32_t b0, uint32_t b1) {
    if constexpr (F16)
        asm volatile(
            "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
            "{%0,%1,%2,%3};"
            : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
            : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
    else
        asm volatile(
            "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
            "{%0,%1,%2,%3};"
            : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
            : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Two floats rounded (RNE) to the MMA's 16-bit type, low half first.
template <bool F16>
__device__ __forceinline__ uint32_t pack16(float lo, float hi) {
    if constexpr (F16) {
        const __half2 v = __floats2half2_rn(lo, hi);
        return *reinterpret_cast<const uint32_t *>(&v);
    } else {
        const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
        return *reinterpret_cast<const uint32_t *>(&v);
    }
}

// The two values of a packed 16-bit pair, as floats.
template <bool F16>
__device__ __forceinline__ float lo16(uint32_t x) {
    if constexpr (F16)
        return __low2float(*reinterpret_cast<const __half2 *>(&x));
    else
        return __uint_as_float(x << 16);
}
template <bool F16>
__device__ __forceinline__ float hi16(uint32_t x) {
    if constexpr (F16)
        return __high2float(*reinterpret_cast<const __half2 *>(&x));
    else
        return __uint_as_float(x & 0xffff0000u);
}

// Two E4M3 codes (low byte first) -> two fp16 values (exact: every E4M3
// value is an fp16 value).
__device__ __forceinline__ uint32_t e4m3x2_to_f16x2(uint32_t two_codes) {
    uint32_t d;
    const uint16_t a = (uint16_t)two_codes;
    asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(d) : "h"(a));
    return d;
}

template <int D, int G, bool FP8>
__global__ void __launch_bounds__(32) decode_kernel(const DecodeParams p, const __grid_constant__ CUtensorMap pool_map) {
    using C = Cfg<D, FP8>;
    constexpr int TOK = C::TOK, STAGES = C::STAGES, KS = C::KS, SUB = C::SUB, NB = C::NB, BOX = C::BOX;
    constexpr int NB8 = C::NB8;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    // swizzled boxes must start on a 1024-byte boundary
    uint8_t *smem = smem_raw + ((1024 - (smem_addr(smem_raw) & 1023)) & 1023);

    const int lane = threadIdx.x;
    const int gq = lane >> 2, tq = lane & 3;  // mma fragment coordinates
    const int64_t w = blockIdx.x;
    const int64_t t0 = warp_start(w, p.n_tiles, p.n_warps);
    const int64_t t1 = warp_start(w + 1, p.n_tiles, p.n_warps);
    const int P = p.page_size;
    const int tpp = (P + TOK - 1) / TOK;

    uint8_t *ring = smem;
    uint8_t *staging = smem + C::RING_BYTES;  // fp8: the current tile's values expanded to fp16
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + C::RING_BYTES + C::STAGING_BYTES);
    int *vrs = reinterpret_cast<int *>(smem + C::RING_BYTES + C::STAGING_BYTES + STAGES * 8);  // valid rows [los, vrs)
    int *los = vrs + STAGES;
    if (lane == 0) {
#pragma unroll
        for (int s = 0; s < STAGES; ++s) mbar_init(&bars[s], 1);
        fence_mbar_init();
    }
    __syncwarp();

    const int64_t plane_rows = p.pool_pages * (int64_t)p.n_kv_heads * P;  // rows per (layer, K/V)

    // Lane 0's cursor over the tiles it copies: tiles are issued in order, so
    // the position advances by one; it is re-located only at a unit boundary.
    struct Cursor {
        int64_t t, end;  // next tile to issue; first tile past its unit
        int lr, b, g, seq, jj, k;
        int lo;          // rows before the window start in the next tile (its unit's first only)
    } cur;
    cur.t = t0;
    cur.end = t0;
    auto advance_to_unit = [&]() {
        const TilePos tp = locate(p, cur.t);
        cur.lr = tp.lr;
        cur.b = tp.b;
        cur.g = tp.g;
        cur.seq = p.rows.seq[tp.b];
        const int tile = tp.tile + p.rows.tile0[tp.b];
        cur.jj = tile / tpp;
        cur.k = tile - cur.jj * tpp;
        cur.lo = tp.tile == 0 ? p.rows.lo[tp.b] : 0;
        cur.end = cur.t - tp.tile + (p.rows.pref_tiles[tp.b + 1] - p.rows.pref_tiles[tp.b]);
    };

    // The page-table entry and fill of the next tile to issue are loaded one
    // issue ahead (lane 0's registers), so their latency hides behind a
    // tile's compute instead of stalling the warp at the issue.
    struct PageAhead {
        int seq = -1, jj = -1, fill = 0, pid = -1;
    } ahead;
    // lane 0: arm the stage's barrier and copy the next tile's K and V boxes
    auto issue = [&](int stg) {
        if (cur.t >= cur.end) advance_to_unit();
        const int seq = cur.seq, jj = cur.jj, k = cur.k, lo = cur.lo;
        struct { int lr, g; } tp{cur.lr, cur.g};
        ++cur.t;
        cur.lo = 0;
        if (++cur.k == tpp) {
            cur.k = 0;
            ++cur.jj;
        }
        int fill, pid;
        if (!FP8 && ahead.seq == seq && ahead.jj == jj) {
            fill = ahead.fill;
            pid = ahead.pid;
        } else {
            fill = p.page_fill[(int64_t)seq * p.max_pages + jj];
            pid = p.page_table[(int64_t)seq * p.max_pages + jj];
        }
        // the next tile of this unit (same page, or the next one); the fp8
        // kernel issues in mid-tile and measured no faster with it
        if constexpr (!FP8) {
            if (cur.t < cur.end && cur.jj != jj) {
                ahead.seq = cur.seq;
                ahead.jj = cur.jj;
                ahead.fill = p.page_fill[(int64_t)cur.seq * p.max_pages + cur.jj];
                ahead.pid = p.page_table[(int64_t)cur.seq * p.max_pages + cur.jj];
            } else if (cur.jj == jj) {
                ahead.seq = seq;
                ahead.jj = jj;
                ahead.fill = fill;
                ahead.pid = pid;
            }
        }
        int vr = fill - k * TOK;
        vr = vr < 0 ? 0 : (vr > TOK ? TOK : vr);
        if (lo >= vr) vr = 0;
        if (vr > 0 && (pid < 0 || pid >= p.pool_pages)) {
            record_error(p.status, KVG_ERR_DEVICE_CHECK, 1);
            vr = 0;
        }
        vrs[stg] = vr;
        los[stg] = lo;
        uint64_t *bar = &bars[stg];
        if (vr > 0) {
            mbar_arrive_expect_tx(bar, (uint32_t)C::STAGE_BYTES);
            const int l = p.layers[tp.lr];
            const int32_t row_k = (int32_t)((2 * l) * plane_rows + ((int64_t)pid * p.n_kv_heads + tp.g) * P +
                                            (int64_t)k * TOK);
            const int32_t row_v = (int32_t)(row_k + plane_rows);
            uint8_t *dst = ring + stg * C::STAGE_BYTES;
            if constexpr (FP8) {
#pragma unroll
                for (int b = 0; b < NB8; ++b) {
                    tma_load_2d(dst + b * BOX, &pool_map, 128 * b, row_k, bar);
                    tma_load_2d(dst + (NB8 + b) * BOX, &pool_map, 128 * b, row_v, bar);
                }
            } else {
#pragma unroll
                for (int b = 0; b < NB; ++b) {
                    tma_load_2d(dst + b * BOX, &pool_map, 64 * b, row_k, bar);
                    tma_load_2d(dst + (NB + b) * BOX, &pool_map, 64 * b, row_v, bar);
                }
            }
        } else {
            mbar_arrive(bar);
        }
    };

    uint32_t qb[KS][2];   // B fragments of q (heads gq < G), per k-step
    float o[KS][4];       // O^T accumulators: dims 16*mt + gq (+8), heads 2*tq (+1)
    float m[2], lsum[2];  // running max / partial sum of heads 2*tq, 2*tq+1
    int64_t cur_unit = -1;

    auto flush = [&](int64_t unit) {
        float lt[2];
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            float v = lsum[e];
            v += __shfl_xor_sync(0xffffffffu, v, 4);
            v += __shfl_xor_sync(0xffffffffu, v, 8);
            v += __shfl_xor_sync(0xffffffffu, v, 16);
            lt[e] = v;
        }
        const int64_t slot = unit + w;
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int h = 2 * tq + e;
            if (h < G) {
                float *dst = p.part_o + (slot * G + h) * D;
#pragma unroll
                for (int mt = 0; mt < KS; ++mt) {
                    dst[16 * mt + gq] = o[mt][e];
                    dst[16 * mt + gq + 8] = o[mt][2 + e];
                }
                if (gq == 0) p.part_ml[slot * G + h] = make_float2(m[e], lt[e]);
            }
        }
    };

    auto begin = [&](const TilePos &tp) {
        const __nv_bfloat16 *qrow =
            p.q + ((int64_t)(p.qlayers[tp.lr] * p.q_row_stride_b + p.b0 + tp.b) * p.n_q_heads + tp.g * G) * D;
#pragma unroll
        for (int ks = 0; ks < KS; ++ks) {
            if (gq < G) {
                if constexpr (FP8) {
                    // fp16 MMAs over permuted dims: within each 16-dim step the
                    // MMA's k = 2tq, 2tq+1, 2tq+8, 2tq+9 are dims 4tq .. 4tq+3, so a
                    // key row's 4 consecutive codes fill a lane's two registers
                    const uint32_t *q32 = reinterpret_cast<const uint32_t *>(qrow + gq * D + 16 * ks + 4 * tq);
                    qb[ks][0] = pack16<true>(lo16<false>(q32[0]), hi16<false>(q32[0]));
                    qb[ks][1] = pack16<true>(lo16<false>(q32[1]), hi16<false>(q32[1]));
                } else {
                    const uint32_t *q32 = reinterpret_cast<const uint32_t *>(qrow + gq * D + 16 * ks + 2 * tq);
                    qb[ks][0] = q32[0];
                    qb[ks][1] = q32[4];  // dims + 8
                }
            } else {
                qb[ks][0] = qb[ks][1] = 0u;
            }
#pragma unroll
            for (int c = 0; c < 4; ++c) o[ks][c] = 0.f;
        }
        m[0] = m[1] = -INFINITY;
        lsum[0] = lsum[1] = 0.f;
    };

    if (lane == 0)
        for (int i = 0; i < STAGES && t0 + i < t1; ++i) issue(i);

    const uint32_t ring_s = smem_addr(ring);
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
        const int vr = vrs[stg], lo = los[stg];
        bool zeroed = false;
        if constexpr (FP8) {
            if (vr > 0) {
                // expand the value codes into the fp16 staging tile (the swizzled
                // box layout of a bf16 tile); rows outside [lo, vr) become zeros.
                // All loads first, then the conversions and stores.
                constexpr int GPR = D / 8;             // 8-value groups per row
                constexpr int ITEMS = TOK * GPR / 32;  // per lane
                const uint8_t *v8 = ring + stg * C::STAGE_BYTES + NB8 * BOX;
                uint2 w[ITEMS];
#pragma unroll
                for (int i = 0; i < ITEMS; ++i) {
                    const int item = i * 32 + lane, r = item / GPR, g = item % GPR;
                    w[i] = make_uint2(0, 0);
                    if (r >= lo && r < vr)
                        w[i] = *reinterpret_cast<const uint2 *>(v8 + (g >> 4) * BOX + r * 128 +
                                                                ((((g & 15) >> 1) ^ (r & 7)) << 4) + (g & 1) * 8);
                }
#pragma unroll
                for (int i = 0; i < ITEMS; ++i) {
                    const int item = i * 32 + lane, r = item / GPR, g = item % GPR;
                    *reinterpret_cast<uint4 *>(staging + (g >> 3) * BOX + r * 128 + (((g & 7) ^ (r & 7)) << 4)) =
                        make_uint4(e4m3x2_to_f16x2(w[i].x), e4m3x2_to_f16x2(w[i].x >> 16), e4m3x2_to_f16x2(w[i].y),
                                   e4m3x2_to_f16x2(w[i].y >> 16));
                }
                __syncwarp();
            } else if (lane == 0 && t + STAGES < t1) {
                issue(stg);  // an empty tile: nothing to read from the stage
            }
        } else if (vr > 0 && (vr < TOK || lo > 0)) {
            // value rows past the fill hold whatever the pool had there, and
            // rows before a window's start are outside the attention: zero
            // both so their zero weights contribute exactly 0
            uint4 *vz = reinterpret_cast<uint4 *>(ring + stg * C::STAGE_BYTES + NB * BOX);
            const int n_out = TOK - vr + lo;  // rows [0, lo) and [vr, TOK)
            for (int idx = lane; idx < NB * n_out * 8; idx += 32) {
                const int b = idx / (n_out * 8);
                const int rem = idx - b * n_out * 8;
                const int r = rem / 8 < lo ? rem / 8 : vr + (rem / 8 - lo);
                vz[(b * BOX + r * 128) / 16 + (rem & 7)] = make_uint4(0, 0, 0, 0);
            }
            fence_proxy_async_shared();
            zeroed = true;
            __syncwarp();
        }
        if (vr > 0) {
            const uint32_t ks_base = ring_s + stg * C::STAGE_BYTES;
            const uint32_t vs_base = FP8 ? smem_addr(staging) : ks_base + NB * BOX;
            // ---- scores S[16 rows][8 heads] per sub-tile
            float sc[SUB][4];
#pragma unroll
            for (int sb = 0; sb < SUB; ++sb) {
                float acc0[4] = {0.f, 0.f, 0.f, 0.f}, acc1[4] = {0.f, 0.f, 0.f, 0.f};
                if constexpr (FP8) {
                    // rows gq and gq+8 of the sub-tile, 4 codes at dims 16ks + 4tq of
                    // each (swizzle: chunk ^ (row & 7), the same for both rows)
                    const uint8_t *k0 = ring + stg * C::STAGE_BYTES + (16 * sb + gq) * 128 + 4 * tq;
#pragma unroll
                    for (int ks = 0; ks < KS; ++ks) {
                        const int off = (ks >> 3) * BOX + (((ks & 7) ^ gq) << 4);
                        const uint32_t w0 = *reinterpret_cast<const uint32_t *>(k0 + off);
                        const uint32_t w1 = *reinterpret_cast<const uint32_t *>(k0 + off + 8 * 128);
                        const uint32_t a0 = e4m3x2_to_f16x2(w0), a2 = e4m3x2_to_f16x2(w0 >> 16);
                        const uint32_t a1 = e4m3x2_to_f16x2(w1), a3 = e4m3x2_to_f16x2(w1 >> 16);
                        if (ks & 1)
                            mma16<true>(acc1, a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
                        else
                            mma16<true>(acc0, a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
                    }
                } else {
                    // lane -> row of its 8x8 matrix (rows +8 for matrices 1,3) and
                    // 16-byte chunk (+1 for matrices 2,3), swizzled: chunk ^ (row & 7)
                    const uint32_t a_row = ks_base + (16 * sb + (lane & 7) + ((lane >> 3) & 1) * 8) * 128;
                    const int a_hi = (lane >> 4) & 1;
#pragma unroll
                    for (int ks = 0; ks < KS; ++ks) {
                        uint32_t a0, a1, a2, a3;
                        const int chunk = ((ks & 3) << 1) + a_hi;
                        ldsm_x4(a_row + (ks >> 2) * BOX + ((chunk ^ (lane & 7)) << 4), a0, a1, a2, a3);
                        if (ks & 1)
                            mma16<false>(acc1, a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
                        else
                            mma16<false>(acc0, a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
                    }
                }
                const int r0 = 16 * sb + gq, r1 = r0 + 8;
                const bool in0 = r0 >= lo && r0 < vr, in1 = r1 >= lo && r1 < vr;
                sc[sb][0] = in0 ? (acc0[0] + acc1[0]) * p.qscale : -INFINITY;
                sc[sb][1] = in0 ? (acc0[1] + acc1[1]) * p.qscale : -INFINITY;
                sc[sb][2] = in1 ? (acc0[2] + acc1[2]) * p.qscale : -INFINITY;
                sc[sb][3] = in1 ? (acc0[3] + acc1[3]) * p.qscale : -INFINITY;
            }
            if constexpr (FP8) {
                // the keys have been read: the stage can take the next tile
                __syncwarp();
                if (lane == 0 && t + STAGES < t1) issue(stg);
            }
            // ---- online softmax for heads 2*tq (e = 0) and 2*tq+1 (e = 1)
            float mt_[2] = {-INFINITY, -INFINITY};
#pragma unroll
            for (int sb = 0; sb < SUB; ++sb) {
                mt_[0] = fmaxf(mt_[0], fmaxf(sc[sb][0], sc[sb][2]));
                mt_[1] = fmaxf(mt_[1], fmaxf(sc[sb][1], sc[sb][3]));
            }
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                mt_[e] = fmaxf(mt_[e], __shfl_xor_sync(0xffffffffu, mt_[e], 4));
                mt_[e] = fmaxf(mt_[e], __shfl_xor_sync(0xffffffffu, mt_[e], 8));
                mt_[e] = fmaxf(mt_[e], __shfl_xor_sync(0xffffffffu, mt_[e], 16));
                if (mt_[e] > m[e]) {
                    const float alpha = exp2f(m[e] - mt_[e]);
                    lsum[e] *= alpha;
#pragma unroll
                    for (int mt = 0; mt < KS; ++mt) {
                        o[mt][e] *= alpha;
                        o[mt][2 + e] *= alpha;
                    }
                    m[e] = mt_[e];
                }
            }
#pragma unroll
            for (int sb = 0; sb < SUB; ++sb) {
                // weights, rounded to the MMA's 16-bit type exactly as it consumes them
                const uint32_t p01 = pack16<FP8>(exp2f(sc[sb][0] - m[0]), exp2f(sc[sb][1] - m[1]));
                const uint32_t p23 = pack16<FP8>(exp2f(sc[sb][2] - m[0]), exp2f(sc[sb][3] - m[1]));
                lsum[0] += lo16<FP8>(p01) + lo16<FP8>(p23);
                lsum[1] += hi16<FP8>(p01) + hi16<FP8>(p23);
                // B fragment of P^T for this lane: tokens 2*tq, 2*tq+1 (+8) of head gq,
                // held by lanes 4*token + gq/2 in half gq%2 of p01 (p23 for +8)
                const int src0 = 4 * (2 * tq) + (gq >> 1), src1 = src0 + 4;
                const uint32_t x0 = __shfl_sync(0xffffffffu, p01, src0);
                const uint32_t x1 = __shfl_sync(0xffffffffu, p01, src1);
                const uint32_t y0 = __shfl_sync(0xffffffffu, p23, src0);
                const uint32_t y1 = __shfl_sync(0xffffffffu, p23, src1);
                const uint32_t sel = (gq & 1) ? 0x7632u : 0x5410u;
                uint32_t b0 = __byte_perm(x0, x1, sel);
                uint32_t b1 = __byte_perm(y0, y1, sel);
                if (gq >= G) b0 = b1 = 0u;
                // ---- O^T[D][8] += V^T[D][16 rows] . P^T[16][8]
                const uint32_t v_row = vs_base + (16 * sb + (lane & 7) + ((lane >> 4) & 1) * 8) * 128;
                const int v_hi = (lane >> 3) & 1;
#pragma unroll
                for (int mt = 0; mt < KS; ++mt) {
                    uint32_t a0, a1, a2, a3;
                    const int chunk = ((mt & 3) << 1) + v_hi;
                    ldsm_x4_t(v_row + (mt >> 2) * BOX + ((chunk ^ (lane & 7)) << 4), a0, a1, a2, a3);
                    mma16<FP8>(o[mt], a0, a1, a2, a3, b0, b1);
                }
            }
        }
        __syncwarp();
        (void)zeroed;
        if (!FP8 && lane == 0 && t + STAGES < t1) issue(stg);
    }
    if (!alive) {
        // a copy never completed: wait (bounded) on every stage once more so
        // no copy is left writing this CTA's shared memory, then record an
        // empty partial for the unit in progress
        for (int s = 0; s < STAGES; ++s) (void)mbar_wait_bounded(&bars[s], 0);
#pragma unroll
        for (int mt = 0; mt < KS; ++mt)
#pragma unroll
            for (int c = 0; c < 4; ++c) o[mt][c] = 0.f;
        m[0] = m[1] = -INFINITY;
        lsum[0] = lsum[1] = 0.f;
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
    const float r = L > 0.f ? __fdiv_rn(O, L) * p.vscale : 0.f;
    p.out[((int64_t)(p.qlayers[lr] * p.q_row_stride_b + p.b0 + b) * p.n_q_heads + h) * D + d] =
        __float2bfloat16_rn(r);
}

// The same merge for a split decode: the unit's partials give (M, L, O) for
// this call's rows, scaled by vscale, and the result is stored as the state
// (o, m, l) of query head h, or merged into the state already there:
// m' = max(m0, M), o' = o0 2^(m0 - m') + O 2^(M - m'), l' likewise (a side
// with l = 0 holds no rows and is left out).
template <int D>
__global__ void __launch_bounds__(D) combine_state_kernel(const DecodeParams p) {
    const int h = blockIdx.x, b = blockIdx.y, lr = blockIdx.z;
    const int G = p.n_q_heads / p.n_kv_heads;
    const int g = h / G, hh = h - g * G;
    const int d = threadIdx.x;
    const int64_t unit = ((int64_t)lr * p.B + b) * p.n_kv_heads + g;
    const int64_t sumT = p.rows.pref_tiles[p.B];
    const int64_t Tb = p.rows.pref_tiles[b + 1] - p.rows.pref_tiles[b];
    float L = 0.f, O = 0.f, M = -INFINITY;
    if (Tb > 0) {
        const int64_t T = p.n_tiles, W = p.n_warps;
        const int64_t first = (int64_t)lr * p.n_kv_heads * sumT + (int64_t)p.n_kv_heads * p.rows.pref_tiles[b] +
                              (int64_t)g * Tb;
        const int64_t last = first + Tb - 1;
        const int64_t wa = warp_of(first, T, W), wb = warp_of(last, T, W);
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
        O = __fmul_rn(O, p.vscale);
    }
    float *st = p.state + ((int64_t)(p.qlayers[lr] * p.q_row_stride_b + p.b0 + b) * p.n_q_heads + h) * (D + 4);
    if (p.state_merge) {
        const float m0 = st[D], l0 = st[D + 1], o0 = st[d];
        __syncthreads();  // every thread has read (m0, l0) before thread 0 rewrites them
        if (l0 > 0.f) {
            if (L > 0.f) {
                const float mm = fmaxf(m0, M);
                const float a = exp2f(m0 - mm), c = exp2f(M - mm);
                O = __fmaf_rn(o0, a, __fmul_rn(O, c));
                L = __fmaf_rn(l0, a, __fmul_rn(L, c));
                M = mm;
            } else {
                O = o0;
                L = l0;
                M = m0;
            }
        }
    }
    if (L == 0.f) {
        O = 0.f;
        M = -INFINITY;
    }
    st[d] = O;
    if (d == 0) {
        st[D] = M;
        st[D + 1] = L;
        st[D + 2] = 0.f;
        st[D + 3] = 0.f;
    }
}

__global__ void state_finish_kernel(const float *__restrict__ state, int64_t n_rows, int D,
                                    __nv_bfloat16 *__restrict__ out) {
    const int64_t n = n_rows * D;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / D;
        const int d = (int)(i - r * D);
        const float *st = state + r * (D + 4);
        const float l = st[D + 1];
        out[i] = __float2bfloat16_rn(l > 0.f ? __fdiv_rn(st[d], l) : 0.f);
    }
}

template <int D, int G, bool FP8>
struct DecodeLaunch {
    // The shared-memory attribute is per device: set and cached per device.
    static int max_blocks_per_sm() {
        static std::atomic<int> cached[kMaxDevices];  // 0 = not yet known
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 0;
        int n = cached[dev].load();
        if (n > 0) return n;
        if (cudaFuncSetAttribute(decode_kernel<D, G, FP8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 Cfg<D, FP8>::SMEM) != cudaSuccess)
            return 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, decode_kernel<D, G, FP8>, 32, Cfg<D, FP8>::SMEM) !=
                cudaSuccess ||
            n <= 0)
            return 0;
        cached[dev].store(n);
        return n;
    }
    static cudaError_t run(const DecodeParams &p, const CUtensorMap &map, cudaStream_t s) {
        if (max_blocks_per_sm() <= 0) return cudaErrorInvalidConfiguration;
        if (p.n_warps <= 0 || p.n_tiles <= 0) return cudaSuccess;
        decode_kernel<D, G, FP8><<<p.n_warps, 32, Cfg<D, FP8>::SMEM, s>>>(p, map);
        count_launches(1);
        return cudaGetLastError();
    }
};

}  // namespace

namespace {
typedef CUresult (*EncodeTiled)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// The driver's tensor-map encoder, looked up once (thread-safe static init).
EncodeTiled tensor_map_encoder() {
    static const EncodeTiled fn = []() -> EncodeTiled {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return nullptr;
        return reinterpret_cast<EncodeTiled>(f);
    }();
    return fn;
}
}  // namespace

cudaError_t encode_tensor_map(CUtensorMap *out, int rank, void *base, const cuuint64_t *dims,
                              const cuuint64_t *strides, const cuuint32_t *box) {
    const EncodeTiled encode = tensor_map_encoder();
    if (!encode) return cudaErrorSymbolNotFound;
    const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    const CUresult r = encode(out, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, base, dims, strides, box, estr,
                              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t make_pool_tensor_map(CUtensorMap *out, void *pool, int head_dim, bool fp8, uint64_t rows) {
    const EncodeTiled encode = tensor_map_encoder();
    if (!encode) return cudaErrorSymbolNotFound;
    if (fp8 && head_dim % 128) {  // no fp8 decode for this head_dim: nothing to map
        memset(out, 0, sizeof *out);
        return cudaSuccess;
    }
    const int tok = decode_tile_tokens(head_dim, fp8);  // the box height the kernel for this element type expects
    if (tok == 0 || rows == 0 || rows > 0x7fffffffull) return cudaErrorInvalidValue;
    // 128-byte rows per box: 64 bf16 columns, or 128 fp8 columns
    const cuuint64_t dims[2] = {(cuuint64_t)head_dim, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)head_dim * (fp8 ? 1 : 2)};
    const cuuint32_t box[2] = {fp8 ? 128u : 64u, (cuuint32_t)tok};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = encode(out, fp8 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, pool,
                              dims, strides, box, estr,
                              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

bool decode_supported(int head_dim, int group, bool fp8) {
    if (head_dim != 64 && head_dim != 128 && head_dim != 256) return false;
    if (fp8 && head_dim == 64) return false;
    if (group != 1 && group != 2 && group != 4 && group != 8) return false;
    return head_dim * group <= 512;
}

int decode_tile_tokens(int head_dim, bool fp8) {
    switch (head_dim) {
        case 64: return fp8 ? 0 : Cfg<64>::TOK;
        case 128: return fp8 ? Cfg<128, true>::TOK : Cfg<128>::TOK;
        case 256: return fp8 ? Cfg<256, true>::TOK : Cfg<256>::TOK;
    }
    return 0;
}

#define KVG_DECODE_CASES(X)                                                                              \
    X(64, 1, false) X(64, 2, false) X(64, 4, false) X(64, 8, false) X(128, 1, false) X(128, 2, false)   \
    X(128, 4, false) X(256, 1, false) X(256, 2, false) X(128, 1, true) X(128, 2, true) X(128, 4, true) \
    X(256, 1, true) X(256, 2, true)

int decode_max_warps(int head_dim, int group, bool fp8, int n_sm) {
#define KVG_CASE(DD, GG, FF) \
    if (head_dim == DD && group == GG && fp8 == FF) return DecodeLaunch<DD, GG, FF>::max_blocks_per_sm() * n_sm;
    KVG_DECODE_CASES(KVG_CASE)
#undef KVG_CASE
    return 0;
}

cudaError_t launch_decode(int head_dim, int group, bool fp8, const DecodeParams &p, const CUtensorMap &pool_map,
                          cudaStream_t s) {
#define KVG_CASE(DD, GG, FF) \
    if (head_dim == DD && group == GG && fp8 == FF) return DecodeLaunch<DD, GG, FF>::run(p, pool_map, s);
    KVG_DECODE_CASES(KVG_CASE)
#undef KVG_CASE
    return cudaErrorInvalidValue;
}

cudaError_t launch_combine(int head_dim, int group, const DecodeParams &p, cudaStream_t s) {
    (void)group;
    dim3 grid(p.n_q_heads, p.B, p.n_layers_run);
    if (p.state) {
        switch (head_dim) {
            case 64: combine_state_kernel<64><<<grid, 64, 0, s>>>(p); break;
            case 128: combine_state_kernel<128><<<grid, 128, 0, s>>>(p); break;
            case 256: combine_state_kernel<256><<<grid, 256, 0, s>>>(p); break;
            default: return cudaErrorInvalidValue;
        }
        count_launches(1);
        return cudaGetLastError();
    }
    switch (head_dim) {
        case 64: combine_kernel<64><<<grid, 64, 0, s>>>(p); count_launches(1); break;
        case 128: combine_kernel<128><<<grid, 128, 0, s>>>(p); count_launches(1); break;
        case 256: combine_kernel<256><<<grid, 256, 0, s>>>(p); count_launches(1); break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

cudaError_t launch_state_finish(const float *state, int64_t n_rows, int head_dim, __nv_bfloat16 *out,
                                cudaStream_t s) {
    const int64_t n = n_rows * head_dim;
    if (n == 0) return cudaSuccess;
    int64_t grid = (n + 255) / 256;
    if (grid > 65535) grid = 65535;
    state_finish_kernel<<<(int)grid, 256, 0, s>>>(state, n_rows, head_dim, out);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace kvg

// sha256_kernels.cu — SHA-256 (FIPS 180-4) on the GPU for page digests.
//
// The digest of a page is SHA-256 over the concatenated SHA-256 digests of its
// consecutive 4096-byte leaves.  A leaf is a serial Merkle-Damgard chain, so
// the natural mapping is one thread per leaf (65 compressions for a 4 KB
// leaf); a second kernel hashes each page's leaf digests with one thread per
// page.  Integer-ALU bound: ~1.7k simple integer ops per 64-byte block.
#include "common.cuh"

namespace kvg {

namespace {

// FIPS 180-4 sec. 4.2.2 round constants and sec. 5.3.3 initial hash value.
__constant__ uint32_t kK[64] = {
    0x428a2f98u, 0x71374491u, 0xb5c0fbcfu, 0xe9b5dba5u, 0x3956c25bu, 0x59f111f1u, 0x923f82a4u,
    0xab1c5ed5u, 0xd807aa98u, 0x12835b01u, 0x243185beu, 0x550c7dc3u, 0x72be5d74u, 0x80deb1feu,
    0x9bdc06a7u, 0xc19bf174u, 0xe49b69c1u, 0xefbe4786u, 0x0fc19dc6u, 0x240ca1ccu, 0x2de92c6fu,
    0x4a7484aau, 0x5cb0a9dcu, 0x76f988dau, 0x983e5152u, 0xa831c66du, 0xb00327c8u, 0xbf597fc7u,
    0xc6e00bf3u, 0xd5a79147u, 0x06ca6351u, 0x14292967u, 0x27b70a85u, 0x2e1b2138u, 0x4d2c6dfcu,
    0x53380d13u, 0x650a7354u, 0x766a0abbu, 0x81c2c92eu, 0x92722c85u, 0xa2bfe8a1u, 0xa81a664bu,
    0xc24b8b70u, 0xc76c51a3u, 0xd192e819u, 0xd6990624u, 0xf40e3585u, 0x106aa070u, 0x19a4c116u,
    0x1e376c08u, 0x2748774cu, 0x34b0bcb5u, 0x391c0cb3u, 0x4ed8aa4au, 0x5b9cca4fu, 0x682e6ff3u,
    0x748f82eeu, 0x78a5636fu, 0x84c87814u, 0x8cc70208u, 0x90befffau, 0xa4506cebu, 0xbef9a3f7u,
    0xc67178f2u};
__constant__ uint32_t kH0[8] = {0x6a09e667u, 0xbb67ae85u, 0x3c6ef372u, 0xa54ff53au,
                                0x510e527fu, 0x9b05688cu, 0x1f83d9abu, 0x5be0cd19u};

__device__ __forceinline__ uint32_t rotr(uint32_t x, int n) { return __funnelshift_r(x, x, n); }

// The integer ALU pipe is this kernel's bottleneck while the FMA pipe idles.
// Additions written as a*one + b and right shifts written as the high word of
// a*2^(32-n) execute as IMAD on the FMA pipe.  `one` is a kernel argument
// (always 1) so the compiler cannot fold the multiply back into an add.
// FMA = false: plain additions and shifts (the compiler fuses them into
// 3-input IADD3 on the ALU pipe) for a serial chain, where the dependency
// chain's latency, not pipe throughput, sets the pace.
template <bool FMA = true>
__device__ __forceinline__ uint32_t fadd(uint32_t a, uint32_t b, uint32_t one) {
    if (!FMA) return a + b;
    uint32_t d;
    asm("mad.lo.u32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(one), "r"(b));
    return d;
}
template <int N, bool FMA = true>
__device__ __forceinline__ uint32_t fshr(uint32_t x, uint32_t one) {
    if (!FMA) return x >> N;
    uint32_t d;
    asm("mul.hi.u32 %0, %1, %2;" : "=r"(d) : "r"(x), "r"(one << (32 - N)));
    return d;
}

__device__ __forceinline__ uint32_t bswap(uint32_t x) { return __byte_perm(x, 0, 0x0123); }

// One compression of the 16-word block w (FIPS 180-4 sec. 6.2.2), with the
// message schedule kept as a rolling 16-word window.  Rotations and logic
// stay on the ALU pipe; additions and the schedule's plain shifts go to the
// FMA pipe (fadd/fshr), balancing the two.
template <bool FMA = true>
__device__ __forceinline__ void compress(uint32_t st[8], uint32_t w[16], uint32_t one) {
    uint32_t a = st[0], b = st[1], c = st[2], d = st[3], e = st[4], f = st[5], g = st[6], h = st[7];
#pragma unroll
    for (int t = 0; t < 64; ++t) {
        uint32_t wt;
        if (t < 16) {
            wt = w[t];
        } else {
            const uint32_t w15 = w[(t - 15) & 15], w2 = w[(t - 2) & 15];
            const uint32_t s0 = rotr(w15, 7) ^ rotr(w15, 18) ^ fshr<3, FMA>(w15, one);
            const uint32_t s1 = rotr(w2, 17) ^ rotr(w2, 19) ^ fshr<10, FMA>(w2, one);
            wt = w[t & 15] = fadd<FMA>(fadd<FMA>(w[t & 15], s0, one), fadd<FMA>(w[(t - 7) & 15], s1, one), one);
        }
        const uint32_t S1 = rotr(e, 6) ^ rotr(e, 11) ^ rotr(e, 25);
        const uint32_t ch = (e & f) ^ (~e & g);
        const uint32_t T1 = fadd<FMA>(fadd<FMA>(h, S1, one), fadd<FMA>(fadd<FMA>(ch, kK[t], one), wt, one), one);
        const uint32_t S0 = rotr(a, 2) ^ rotr(a, 13) ^ rotr(a, 22);
        const uint32_t maj = (a & b) ^ (a & c) ^ (b & c);
        h = g;
        g = f;
        f = e;
        e = fadd<FMA>(d, T1, one);
        d = c;
        c = b;
        b = a;
        a = fadd<FMA>(T1, fadd<FMA>(S0, maj, one), one);
    }
    st[0] += a;
    st[1] += b;
    st[2] += c;
    st[3] += d;
    st[4] += e;
    st[5] += f;
    st[6] += g;
    st[7] += h;
}

__device__ __forceinline__ void init_state(uint32_t st[8]) {
#pragma unroll
    for (int i = 0; i < 8; ++i) st[i] = kH0[i];
}

// Final block(s) for a message whose last `rem` (< 64) bytes start at `tail`
// and whose total length is `total_bytes`.
__device__ void finish(uint32_t st[8], const uint8_t *tail, int rem, uint64_t total_bytes, uint32_t one) {
    uint32_t w[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) w[i] = 0;
    for (int k = 0; k < rem; ++k) w[k >> 2] |= (uint32_t)tail[k] << (24 - 8 * (k & 3));
    w[rem >> 2] |= 0x80u << (24 - 8 * (rem & 3));
    const uint64_t bits = total_bytes * 8ull;
    if (rem < 56) {
        w[14] = (uint32_t)(bits >> 32);
        w[15] = (uint32_t)bits;
        compress(st, w, one);
    } else {
        compress(st, w, one);
#pragma unroll
        for (int i = 0; i < 16; ++i) w[i] = 0;
        w[14] = (uint32_t)(bits >> 32);
        w[15] = (uint32_t)bits;
        compress(st, w, one);
    }
}

__device__ __forceinline__ const uint8_t *page_addr(const PageSource &s, int64_t p) {
    if (!s.pid) return s.base + (uint64_t)p * s.page_bytes;
    const int64_t plane = p / s.npb;
    const int64_t j = p - plane * s.npb;
    return s.base + ((uint64_t)plane * s.plane_pages + (uint64_t)s.pid[j]) * s.page_bytes;
}

// 16-byte asynchronous copy global -> this thread's shared memory (LDGSTS,
// L1 bypassed); completion is tracked by the thread's cp.async groups.
__device__ __forceinline__ void cp_async16(void *smem_dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(smem_dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// SHA-256 of one leaf that is also copied to `copy_to`, from the same
// registers that are hashed, so the bytes written are exactly the bytes whose
// digest is checked.  The leaf's next R 64-byte blocks are in flight through
// a ring of this thread's shared memory (ring: R x 64 contiguous bytes), not
// held in registers, so their latency (long when other kernels keep HBM
// busy) hides behind the compressions without costing registers.  (A layout
// with the 32 lanes' vectors side by side, free of bank conflicts, measured
// slower in the 12b step: 6.05 against 5.94 ms.)
template <int R>
__device__ __forceinline__ void hash_leaf_ring(const uint8_t *leaf, uint64_t len, uint8_t *copy_to, uint32_t st[8],
                                               uint32_t one, uint4 *ring) {
    const uint4 *v = reinterpret_cast<const uint4 *>(leaf);
    uint4 *o = reinterpret_cast<uint4 *>(copy_to);
    init_state(st);
    const int nfull = (int)(len >> 6);
#pragma unroll
    for (int b = 0; b < R; ++b) {
        if (b < nfull)
#pragma unroll
            for (int q = 0; q < 4; ++q) cp_async16(ring + 4 * b + q, v + 4 * b + q);
        cp_async_commit();  // one group per block, empty or not, so the count stays uniform
    }
    for (int blk = 0; blk < nfull; ++blk) {
        cp_async_wait<R - 1>();  // block blk has landed
        const int slot = blk % R;
        uint32_t w[16];
        uint4 x[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) x[q] = ring[4 * slot + q];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            w[4 * q + 0] = bswap(x[q].x);
            w[4 * q + 1] = bswap(x[q].y);
            w[4 * q + 2] = bswap(x[q].z);
            w[4 * q + 3] = bswap(x[q].w);
        }
        // the slot is free once its words are in registers: refill it
        if (blk + R < nfull)
#pragma unroll
            for (int q = 0; q < 4; ++q) cp_async16(ring + 4 * slot + q, v + 4 * (blk + R) + q);
        cp_async_commit();
#pragma unroll
        for (int q = 0; q < 4; ++q) __stcs(o + 4 * blk + q, x[q]);
        compress(st, w, one);
    }
    cp_async_wait<0>();
    const int rem = (int)(len & 63);
    if (rem == 0) {
        uint32_t w[16];
#pragma unroll
        for (int q = 0; q < 16; ++q) w[q] = 0;
        w[0] = 0x80000000u;
        const uint64_t bits = len * 8ull;
        w[14] = (uint32_t)(bits >> 32);
        w[15] = (uint32_t)bits;
        compress(st, w, one);
    } else {
        for (int q = 0; q < rem / 16; ++q) o[4 * nfull + q] = v[4 * nfull + q];
        finish(st, leaf + (len & ~63ull), rem, len, one);
    }
}

// SHA-256 of one leaf of `len` bytes (16-byte aligned).  With COPY the leaf
// is also written to `copy_to`, from the same registers that are hashed, so
// the bytes written are exactly the bytes whose digest is checked.
template <bool COPY>
__device__ __forceinline__ void hash_leaf(const uint8_t *leaf, uint64_t len, uint8_t *copy_to, uint32_t st[8],
                                          uint32_t one) {
    const uint4 *v = reinterpret_cast<const uint4 *>(leaf);
    uint4 *o = reinterpret_cast<uint4 *>(copy_to);
    init_state(st);
    const int nfull = (int)(len >> 6);
    // The next two 64-byte blocks are in flight while the current one is
    // compressed, so their memory latency (long when other kernels keep HBM
    // busy) hides behind ~3.4k ALU ops.
    uint4 n1[4], n2[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        if (nfull > 0) n1[q] = __ldg(v + q);
        if (nfull > 1) n2[q] = __ldg(v + 4 + q);
    }
    for (int blk = 0; blk < nfull; ++blk) {
        uint32_t w[16];
        uint4 x[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            x[q] = n1[q];
            n1[q] = n2[q];
        }
        if (blk + 2 < nfull) {
#pragma unroll
            for (int q = 0; q < 4; ++q) n2[q] = __ldg(v + 4 * (blk + 2) + q);
        }
        if (COPY) {
#pragma unroll
            for (int q = 0; q < 4; ++q) __stcs(o + 4 * blk + q, x[q]);
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            w[4 * q + 0] = bswap(x[q].x);
            w[4 * q + 1] = bswap(x[q].y);
            w[4 * q + 2] = bswap(x[q].z);
            w[4 * q + 3] = bswap(x[q].w);
        }
        compress(st, w, one);
    }
    const int rem = (int)(len & 63);
    if (rem == 0) {
        uint32_t w[16];
#pragma unroll
        for (int q = 0; q < 16; ++q) w[q] = 0;
        w[0] = 0x80000000u;
        const uint64_t bits = len * 8ull;
        w[14] = (uint32_t)(bits >> 32);
        w[15] = (uint32_t)bits;
        compress(st, w, one);
    } else {
        if (COPY)
            for (int q = 0; q < rem / 16; ++q) o[4 * nfull + q] = v[4 * nfull + q];
        finish(st, leaf + (len & ~63ull), rem, len, one);
    }
}

__device__ __forceinline__ void store_state(uint32_t *out, const uint32_t st[8]) {
    uint4 *o = reinterpret_cast<uint4 *>(out);
    o[0] = make_uint4(st[0], st[1], st[2], st[3]);
    o[1] = make_uint4(st[4], st[5], st[6], st[7]);
}

// ---- two-warp form, for launches too small to fill the GPU ---------------
// When there are few chains, each one's latency decides, and a thread that
// both expands the message schedule and runs the rounds issues ~27
// instructions a round from one warp.  Here a 64-thread CTA works on 32
// chains (lane c of both warps on chain c): warp 1 loads each chain's next
// 64-byte block, expands its schedule and leaves K[t] + W[t] in shared
// memory; warp 0 runs the 64 rounds from there.  The rounds' warp then
// issues ~18 instructions a round on its own scheduler: ~1,775 cycles per
// block against ~2,480 (a probe over 256 blocks per chain, same digests).
// Two buffers change hands through named barriers: 1 + b (buffer b full,
// warp 1 arrives, warp 0 waits) and 3 + b (buffer b free again, warp 0
// arrives, warp 1 waits).  Both warps run the same number of blocks, with
// every lane taking part (lanes past the last chain hash zeros and store
// nothing), so every arrival meets its wait.
constexpr int kSplitChains = 32;

__device__ __forceinline__ void bar_sync_pair(int id) { asm volatile("bar.sync %0, 64;" ::"r"(id) : "memory"); }
__device__ __forceinline__ void bar_arrive_pair(int id) { asm volatile("bar.arrive %0, 64;" ::"r"(id) : "memory"); }

// Warp 1: the message schedule of block w plus the round constants, into
// column `lane` of kw[64][32] (plain ALU arithmetic: this warp's scheduler
// has nothing else to issue).
__device__ __forceinline__ void split_expand(uint32_t (*kw)[kSplitChains], uint32_t w[16], int lane) {
#pragma unroll
    for (int t = 0; t < 64; ++t) {
        uint32_t wt;
        if (t < 16) {
            wt = w[t];
        } else {
            const uint32_t w15 = w[(t - 15) & 15], w2 = w[(t - 2) & 15];
            const uint32_t s0 = rotr(w15, 7) ^ rotr(w15, 18) ^ (w15 >> 3);
            const uint32_t s1 = rotr(w2, 17) ^ rotr(w2, 19) ^ (w2 >> 10);
            wt = w[t & 15] = w[t & 15] + s0 + w[(t - 7) & 15] + s1;
        }
        kw[t][lane] = wt + kK[t];
    }
}

// Warp 0: the 64 rounds of one block from kw (FIPS 180-4 sec. 6.2.2 step 3,
// with h + K[t] + W[t] taken whole from shared memory) and the feed-forward.
// The additions off the last step go to the FMA pipe (fadd), so the ALU pipe
// carries the rotations and logic.
__device__ __forceinline__ void split_rounds(uint32_t st[8], const uint32_t (*kw)[kSplitChains], int lane,
                                             uint32_t one) {
    uint32_t a = st[0], b = st[1], c = st[2], d = st[3], e = st[4], f = st[5], g = st[6], h = st[7];
#pragma unroll
    for (int t = 0; t < 64; ++t) {
        const uint32_t k = kw[t][lane];
        const uint32_t S1 = rotr(e, 6) ^ rotr(e, 11) ^ rotr(e, 25);
        const uint32_t ch = (e & f) ^ (~e & g);
        const uint32_t S0 = rotr(a, 2) ^ rotr(a, 13) ^ rotr(a, 22);
        const uint32_t maj = (a & b) ^ (a & c) ^ (b & c);
        const uint32_t hkc = fadd(fadd(h, k, one), ch, one);  // h + K[t] + W[t] + Ch
        const uint32_t T1 = fadd(hkc, S1, one);
        const uint32_t ne = fadd(fadd(d, hkc, one), S1, one);  // d + T1
        h = g;
        g = f;
        f = e;
        e = ne;
        d = c;
        c = b;
        b = a;
        a = T1 + S0 + maj;
    }
    st[0] += a;
    st[1] += b;
    st[2] += c;
    st[3] += d;
    st[4] += e;
    st[5] += f;
    st[6] += g;
    st[7] += h;
}

// Warp 0's side of a chain of n_blocks blocks: state from H0 to the digest.
__device__ __forceinline__ void split_consume(uint32_t st[8], uint32_t (*kw)[64][kSplitChains], int n_blocks,
                                              int lane, uint32_t one) {
    init_state(st);
    for (int blk = 0; blk < n_blocks; ++blk) {
        const int buf = blk & 1;
        bar_sync_pair(1 + buf);
        split_rounds(st, kw[buf], lane, one);
        if (blk + 2 < n_blocks) bar_arrive_pair(3 + buf);
    }
}

// Warp 1 hands over block blk (its 16 words in w) through buffer blk & 1.
__device__ __forceinline__ void split_hand_over(uint32_t (*kw)[64][kSplitChains], uint32_t w[16], int blk, int lane) {
    const int buf = blk & 1;
    if (blk >= 2) bar_sync_pair(3 + buf);
    split_expand(kw[buf], w, lane);
    __threadfence_block();
    bar_arrive_pair(1 + buf);
}

// The padding block of a message of `bytes` bytes (a multiple of 64).
__device__ __forceinline__ void padding_block(uint32_t w[16], uint64_t bytes) {
#pragma unroll
    for (int q = 0; q < 16; ++q) w[q] = 0;
    w[0] = 0x80000000u;
    const uint64_t bits = bytes * 8ull;
    w[14] = (uint32_t)(bits >> 32);
    w[15] = (uint32_t)bits;
}

// Warp 1's side of a whole 4 KiB leaf at v (nullptr: zeros), also written to
// o when COPY (the bytes written are the bytes hashed): 64 data blocks, the
// next two in flight, then the padding block.
template <bool COPY>
__device__ __forceinline__ void split_produce_leaf(uint32_t (*kw)[64][kSplitChains], const uint4 *v, uint4 *o,
                                                   int lane) {
    constexpr int kData = (int)(kLeafBytes / 64);
    uint4 n1[4], n2[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        n1[q] = v ? __ldg(v + q) : make_uint4(0, 0, 0, 0);
        n2[q] = v ? __ldg(v + 4 + q) : make_uint4(0, 0, 0, 0);
    }
    for (int blk = 0; blk < kData; ++blk) {
        uint4 x[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            x[q] = n1[q];
            n1[q] = n2[q];
        }
        if (v && blk + 2 < kData) {
#pragma unroll
            for (int q = 0; q < 4; ++q) n2[q] = __ldg(v + 4 * (blk + 2) + q);
        }
        if (COPY && o) {
#pragma unroll
            for (int q = 0; q < 4; ++q) __stcs(o + 4 * blk + q, x[q]);
        }
        uint32_t w[16];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            w[4 * q + 0] = bswap(x[q].x);
            w[4 * q + 1] = bswap(x[q].y);
            w[4 * q + 2] = bswap(x[q].z);
            w[4 * q + 3] = bswap(x[q].w);
        }
        split_hand_over(kw, w, blk, lane);
    }
    uint32_t w[16];
    padding_block(w, kLeafBytes);
    split_hand_over(kw, w, kData, lane);
}

constexpr int kSplitLeafBlocks = (int)(kLeafBytes / 64) + 1;

// graft_verify_kernel's work in the two-warp form, for pages made of whole
// 4 KiB leaves and launches of at most one such CTA per SM.
__global__ void __launch_bounds__(64) graft_verify_split_kernel(const GraftParams p, int64_t leaves_per_page,
                                                                uint32_t *__restrict__ out, uint32_t one) {
    __shared__ __align__(16) uint32_t kw[2][64][kSplitChains];
    graft_metadata(p);
    const int lane = threadIdx.x & 31;
    const uint64_t page_bytes = p.page_bytes;
    const int64_t n_leaves = (int64_t)p.n_layers * 2 * p.npb * leaves_per_page;
    const int64_t idx = (int64_t)blockIdx.x * kSplitChains + lane;
    const bool valid = idx < n_leaves;
    const int64_t page_u = idx / leaves_per_page;
    const int64_t i = idx - page_u * leaves_per_page;
    const int64_t lkv = page_u / p.npb;
    const int64_t jj = page_u - lkv * p.npb;
    const int64_t block_page = lkv * p.block_pages + p.page_base + jj;
    if (threadIdx.x >= 32) {
        const uint64_t off = (uint64_t)i * kLeafBytes;
        const uint4 *v = valid ? reinterpret_cast<const uint4 *>(p.src + (uint64_t)block_page * page_bytes + off)
                               : nullptr;
        uint4 *o = valid ? reinterpret_cast<uint4 *>(p.pool + ((uint64_t)lkv * p.pool_pages +
                                                               (uint64_t)p.pids.pid[jj]) * page_bytes + off)
                         : nullptr;
        split_produce_leaf<true>(kw, v, o, lane);
    } else {
        uint32_t st[8];
        split_consume(st, kw, kSplitLeafBlocks, lane, one);
        if (valid) store_state(out + (block_page * leaves_per_page + i) * 8, st);
    }
}

// sha256_leaves_kernel's work in the two-warp form (whole 4 KiB leaves).
__global__ void __launch_bounds__(64) sha256_leaves_split_kernel(const PageSource src, int64_t n_pages,
                                                                 int64_t leaves_per_page,
                                                                 uint32_t *__restrict__ out, uint32_t one) {
    __shared__ __align__(16) uint32_t kw[2][64][kSplitChains];
    const int lane = threadIdx.x & 31;
    const int64_t idx = (int64_t)blockIdx.x * kSplitChains + lane;
    const bool valid = idx < n_pages * leaves_per_page;
    const int64_t p = idx / leaves_per_page;
    const int64_t i = idx - p * leaves_per_page;
    bool in_range = valid;
    if (valid && src.pid) {  // page ids come from a device page table: never read outside the pool
        const int32_t pid = src.pid[p - (p / src.npb) * src.npb];
        in_range = pid >= 0 && pid < src.plane_pages;
    }
    if (threadIdx.x >= 32) {
        const uint4 *v = in_range ? reinterpret_cast<const uint4 *>(page_addr(src, p) + (uint64_t)i * kLeafBytes)
                                  : nullptr;
        split_produce_leaf<false>(kw, v, nullptr, lane);
    } else {
        uint32_t st[8];
        split_consume(st, kw, kSplitLeafBlocks, lane, one);
        if (!valid) return;
        if (!in_range) {
#pragma unroll
            for (int w = 0; w < 8; ++w) st[w] = 0u;  // no digest of any page: reported as a mismatch
        }
        int64_t po = p;
        if (src.pid && src.out_plane_stride) {
            const int64_t plane = p / src.npb;
            po = plane * src.out_plane_stride + src.out_j0 + (p - plane * src.npb);
        }
        store_state(out + (po * leaves_per_page + i) * 8, st);
    }
}

__global__ void __launch_bounds__(128) sha256_leaves_kernel(const PageSource src, int64_t n_pages,
                                                            int64_t leaves_per_page,
                                                            uint32_t *__restrict__ out, uint32_t one) {
    const int64_t n_leaves = n_pages * leaves_per_page;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < n_leaves;
         idx += (int64_t)gridDim.x * blockDim.x) {
        const int64_t p = idx / leaves_per_page;
        const int64_t i = idx - p * leaves_per_page;
        uint64_t len = src.page_bytes - (uint64_t)i * kLeafBytes;
        if (len > kLeafBytes) len = kLeafBytes;
        uint32_t st[8];
        bool in_range = true;
        if (src.pid) {  // page ids come from a device page table: never read outside the pool
            const int32_t pid = src.pid[p - (p / src.npb) * src.npb];
            in_range = pid >= 0 && pid < src.plane_pages;
        }
        if (in_range) {
            hash_leaf<false>(page_addr(src, p) + (uint64_t)i * kLeafBytes, len, nullptr, st, one);
        } else {
#pragma unroll
            for (int w = 0; w < 8; ++w) st[w] = 0u;  // no digest of any page: reported as a mismatch
        }
        int64_t po = p;
        if (src.pid && src.out_plane_stride) {
            const int64_t plane = p / src.npb;
            po = plane * src.out_plane_stride + src.out_j0 + (p - plane * src.npb);
        }
        store_state(out + (po * leaves_per_page + i) * 8, st);
    }
}

// graft_verify_kernel with each thread keeping its leaf's next
// kGraftVerifyRing blocks in flight through its own slots of shared memory
// instead of two blocks in registers; the registers that frees let five CTAs
// of 128 threads stay resident per SM (96 registers).  Used for launches of
// at least one full wave of it (five CTAs on every SM): beside a concurrent
// append the 12b step's window shortens (step 5.94 against 6.01 ms; alone
// the same 3.12 ms; rings of two or four blocks, or six CTAs at 80
// registers, measured slower in the step).  For smaller launches each leaf's
// chain latency decides: the register form is faster there (the tiny
// verified graft 0.099 against 0.133 ms), and the two-warp form faster still
// for launches of up to 64 leaves per SM (0.071 ms).
constexpr int kGraftVerifyRing = 3;
__global__ void __launch_bounds__(128, 5) graft_verify_ring_kernel(const GraftParams p, int64_t leaves_per_page,
                                                                   uint32_t *__restrict__ out, uint32_t one) {
    constexpr int R = kGraftVerifyRing;
    extern __shared__ __align__(16) uint4 ring_mem[];
    graft_metadata(p);
    const uint64_t page_bytes = p.page_bytes;
    const int64_t n_leaves = (int64_t)p.n_layers * 2 * p.npb * leaves_per_page;
    uint4 *ring = ring_mem + threadIdx.x * 4 * R;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < n_leaves;
         idx += (int64_t)gridDim.x * blockDim.x) {
        const int64_t page_u = idx / leaves_per_page;
        const int64_t i = idx - page_u * leaves_per_page;
        const int64_t lkv = page_u / p.npb;
        const int64_t jj = page_u - lkv * p.npb;
        const uint64_t off = (uint64_t)i * kLeafBytes;
        uint64_t len = page_bytes - off;
        if (len > kLeafBytes) len = kLeafBytes;
        const int64_t block_page = lkv * p.block_pages + p.page_base + jj;
        const uint8_t *src = p.src + (uint64_t)block_page * page_bytes + off;
        uint8_t *dst = p.pool + ((uint64_t)lkv * p.pool_pages + (uint64_t)p.pids.pid[jj]) * page_bytes + off;
        uint32_t st[8];
        hash_leaf_ring<R>(src, len, dst, st, one, ring);
        store_state(out + (block_page * leaves_per_page + i) * 8, st);
    }
}

// Own-position graft with the verification folded into the copy: one thread
// per 4 KiB leaf reads it from the block once, writes it to its cache page and
// hashes it (leaf order of a page digest, Sec. 3.2's integrity check).
__global__ void __launch_bounds__(128) graft_verify_kernel(const GraftParams p, int64_t leaves_per_page,
                                                           uint32_t *__restrict__ out, uint32_t one) {
    graft_metadata(p);
    const uint64_t page_bytes = p.page_bytes;
    const int64_t n_leaves = (int64_t)p.n_layers * 2 * p.npb * leaves_per_page;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < n_leaves;
         idx += (int64_t)gridDim.x * blockDim.x) {
        const int64_t page_u = idx / leaves_per_page;
        const int64_t i = idx - page_u * leaves_per_page;
        const int64_t lkv = page_u / p.npb;
        const int64_t jj = page_u - lkv * p.npb;
        const uint64_t off = (uint64_t)i * kLeafBytes;
        uint64_t len = page_bytes - off;
        if (len > kLeafBytes) len = kLeafBytes;
        const int64_t block_page = lkv * p.block_pages + p.page_base + jj;
        const uint8_t *src = p.src + (uint64_t)block_page * page_bytes + off;
        uint8_t *dst = p.pool + ((uint64_t)lkv * p.pool_pages + (uint64_t)p.pids.pid[jj]) * page_bytes + off;
        uint32_t st[8];
        hash_leaf<true>(src, len, dst, st, one);
        store_state(out + (block_page * leaves_per_page + i) * 8, st);
    }
}

// Page p's digest (the state words, big-endian) written to out and/or
// compared with expected; a mismatch is recorded in the status word.
__device__ __forceinline__ void page_verdict(int64_t p, const uint32_t st[8], uint8_t *__restrict__ out,
                                             const uint8_t *__restrict__ expected, DevStatus *status, int32_t seq) {
    uint8_t dg[32];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        dg[4 * k + 0] = (uint8_t)(st[k] >> 24);
        dg[4 * k + 1] = (uint8_t)(st[k] >> 16);
        dg[4 * k + 2] = (uint8_t)(st[k] >> 8);
        dg[4 * k + 3] = (uint8_t)st[k];
    }
    if (out) {
#pragma unroll
        for (int k = 0; k < 32; ++k) out[p * 32 + k] = dg[k];
    }
    if (expected) {
        bool same = true;
#pragma unroll
        for (int k = 0; k < 32; ++k) same &= dg[k] == expected[p * 32 + k];
        if (!same) {
            const int slot = atomicAdd(&status->n_mismatch, 1);
            if (slot < KVG_REPORT_MAX_PAGES) status->list[slot] = (int32_t)p;
            status->seq = seq;
            atomicCAS(&status->err, 0, (int32_t)KVG_ERR_DIGEST);
        }
    }
}

// Page digest from its leaf digests: the message is the leaf digests' bytes,
// i.e. (big-endian) exactly the 8 state words of each leaf in order.
__global__ void __launch_bounds__(128) sha256_pages_kernel(const uint32_t *__restrict__ leaf_words,
                                                           int64_t n_pages, int64_t m,
                                                           uint8_t *__restrict__ out,
                                                           const uint8_t *__restrict__ expected,
                                                           DevStatus *status, int32_t seq, uint32_t one) {
    const int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (p >= n_pages) return;
    const uint32_t *lw = leaf_words + p * m * 8;
    uint32_t st[8];
    init_state(st);
    const int64_t nwords = m * 8;
    const int64_t nfull = nwords / 16;
    for (int64_t blk = 0; blk < nfull; ++blk) {
        uint32_t w[16];
        const uint4 *v = reinterpret_cast<const uint4 *>(lw + blk * 16);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint4 x = v[q];
            w[4 * q + 0] = x.x;
            w[4 * q + 1] = x.y;
            w[4 * q + 2] = x.z;
            w[4 * q + 3] = x.w;
        }
        compress<false>(st, w, one);
    }
    {
        uint32_t w[16];
#pragma unroll
        for (int q = 0; q < 16; ++q) w[q] = 0;
        const int remw = (int)(nwords - nfull * 16);  // 0 or 8
        for (int q = 0; q < remw; ++q) w[q] = lw[nfull * 16 + q];
        w[remw] = 0x80000000u;
        const uint64_t bits = (uint64_t)m * 32ull * 8ull;
        w[14] = (uint32_t)(bits >> 32);
        w[15] = (uint32_t)bits;
        compress<false>(st, w, one);
    }
    page_verdict(p, st, out, expected, status, seq);
}

// sha256_pages_kernel in the two-warp form: warp 1 feeds each page's leaf
// digests (already big-endian words) and the final block.
__global__ void __launch_bounds__(64) sha256_pages_split_kernel(const uint32_t *__restrict__ leaf_words,
                                                                int64_t n_pages, int64_t m,
                                                                uint8_t *__restrict__ out,
                                                                const uint8_t *__restrict__ expected,
                                                                DevStatus *status, int32_t seq, uint32_t one) {
    __shared__ __align__(16) uint32_t kw[2][64][kSplitChains];
    const int lane = threadIdx.x & 31;
    const int64_t p = (int64_t)blockIdx.x * kSplitChains + lane;
    const bool valid = p < n_pages;
    const int64_t nwords = m * 8;
    const int nfull = (int)(nwords / 16);
    const int remw = (int)(nwords - (int64_t)nfull * 16);  // 0 or 8
    if (threadIdx.x >= 32) {
        const uint32_t *lw = leaf_words + (valid ? p : 0) * m * 8;
        uint4 nx[4];
#pragma unroll
        for (int q = 0; q < 4; ++q)
            nx[q] = valid && nfull > 0 ? reinterpret_cast<const uint4 *>(lw)[q] : make_uint4(0, 0, 0, 0);
        for (int blk = 0; blk < nfull; ++blk) {
            uint4 x[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) x[q] = nx[q];
            if (valid && blk + 1 < nfull) {
#pragma unroll
                for (int q = 0; q < 4; ++q) nx[q] = reinterpret_cast<const uint4 *>(lw + (blk + 1) * 16)[q];
            }
            uint32_t w[16];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                w[4 * q + 0] = x[q].x;
                w[4 * q + 1] = x[q].y;
                w[4 * q + 2] = x[q].z;
                w[4 * q + 3] = x[q].w;
            }
            split_hand_over(kw, w, blk, lane);
        }
        uint32_t w[16];
#pragma unroll
        for (int q = 0; q < 16; ++q) w[q] = 0;
        for (int q = 0; q < remw; ++q) w[q] = valid ? lw[nfull * 16 + q] : 0u;
        w[remw] = 0x80000000u;
        const uint64_t bits = (uint64_t)m * 32ull * 8ull;
        w[14] = (uint32_t)(bits >> 32);
        w[15] = (uint32_t)bits;
        split_hand_over(kw, w, nfull, lane);
    } else {
        uint32_t st[8];
        split_consume(st, kw, nfull + 1, lane, one);
        if (valid) page_verdict(p, st, out, expected, status, seq);
    }
}

// Streaming single-thread hasher for seg0 || seg1 of arbitrary lengths.
struct Stream {
    uint32_t one;
    uint32_t st[8];
    uint32_t w[16];
    int fill;  // bytes in w
    uint64_t total;

    __device__ void init(uint32_t one_) {
        one = one_;
        init_state(st);
        fill = 0;
        total = 0;
#pragma unroll
        for (int i = 0; i < 16; ++i) w[i] = 0;
    }
    __device__ void byte(uint8_t x) {
        w[fill >> 2] |= (uint32_t)x << (24 - 8 * (fill & 3));
        if (++fill == 64) {
            compress<false>(st, w, one);
            fill = 0;
#pragma unroll
            for (int i = 0; i < 16; ++i) w[i] = 0;
        }
    }
    __device__ void feed(const uint8_t *ptr, uint64_t n) {
        total += n;
        uint64_t k = 0;
        while (k < n && (fill != 0 || (reinterpret_cast<uintptr_t>(ptr + k) & 3))) byte(ptr[k++]);
        while (n - k >= 64) {
            const uint32_t *q = reinterpret_cast<const uint32_t *>(ptr + k);
#pragma unroll
            for (int i = 0; i < 16; ++i) w[i] = bswap(q[i]);
            compress<false>(st, w, one);
#pragma unroll
            for (int i = 0; i < 16; ++i) w[i] = 0;
            k += 64;
        }
        while (k < n) byte(ptr[k++]);
    }
    __device__ void final(uint8_t out[32]) {
        const uint64_t bits = total * 8ull;
        byte(0x80);
        while (fill != 56) byte(0);
        for (int i = 7; i >= 0; --i) byte((uint8_t)(bits >> (8 * i)));
        for (int k = 0; k < 8; ++k) {
            out[4 * k + 0] = (uint8_t)(st[k] >> 24);
            out[4 * k + 1] = (uint8_t)(st[k] >> 16);
            out[4 * k + 2] = (uint8_t)(st[k] >> 8);
            out[4 * k + 3] = (uint8_t)st[k];
        }
    }
};

// SHA-256 of seg0 || seg1: one serial chain, run by lane 0 of one warp.
// When both segments are 4-byte aligned and seg0's length is a multiple of 4
// (a block's position tags and page digests are), the 32 lanes load the next
// 2 KiB of the message (coalesced 4-byte words) while lane 0 compresses the
// current 2 KiB from shared memory, so the chain never waits on a load;
// otherwise (any byte alignment) lane 0 streams the bytes itself.
constexpr int kSerialChunkWords = 512;  // 2 KiB = 32 blocks per chunk

__device__ __forceinline__ uint32_t msg_word(const uint8_t *seg0, uint64_t n0, const uint8_t *seg1, uint64_t i) {
    const uint64_t off = 4 * i;
    return off < n0 ? *reinterpret_cast<const uint32_t *>(seg0 + off)
                    : *reinterpret_cast<const uint32_t *>(seg1 + (off - n0));
}

__global__ void __launch_bounds__(32) sha256_serial_kernel(const uint8_t *seg0, uint64_t n0, const uint8_t *seg1,
                                                           uint64_t n1, uint8_t *out, const uint8_t *expected,
                                                           DevStatus *status, uint32_t one) {
    __shared__ uint32_t buf[2][kSerialChunkWords];
    const int lane = threadIdx.x;
    if (blockIdx.x != 0) return;
    const uint64_t total = n0 + n1;
    const bool fast = !((reinterpret_cast<uintptr_t>(seg0) | reinterpret_cast<uintptr_t>(seg1) | n0) & 3);
    const uint64_t n_chunks = fast ? total / (4 * kSerialChunkWords) : 0;
    Stream s;
    if (lane == 0) s.init(one);
    if (n_chunks) {
        for (int k = 0; k < kSerialChunkWords / 32; ++k)
            buf[0][lane + 32 * k] = msg_word(seg0, n0, seg1, lane + 32 * k);
        __syncwarp();
        for (uint64_t c = 0; c < n_chunks; ++c) {
            uint32_t nxt[kSerialChunkWords / 32];
            const bool more = c + 1 < n_chunks;
            if (more) {
#pragma unroll
                for (int k = 0; k < kSerialChunkWords / 32; ++k)
                    nxt[k] = msg_word(seg0, n0, seg1, (c + 1) * kSerialChunkWords + lane + 32 * k);
            }
            if (lane == 0) {
                const uint32_t *cur = buf[c & 1];
                for (int b = 0; b < kSerialChunkWords / 16; ++b) {
                    uint32_t w[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) w[i] = bswap(cur[16 * b + i]);
                    compress<false>(s.st, w, one);
                }
            }
            __syncwarp();
            if (more) {
#pragma unroll
                for (int k = 0; k < kSerialChunkWords / 32; ++k) buf[(c + 1) & 1][lane + 32 * k] = nxt[k];
            }
            __syncwarp();
        }
    }
    if (lane != 0) return;
    // the rest of the message (and all of it on the byte path)
    const uint64_t done = n_chunks * 4 * kSerialChunkWords;
    s.total = done;
    if (done < n0) s.feed(seg0 + done, n0 - done);
    const uint64_t d1 = done > n0 ? done - n0 : 0;
    if (d1 < n1) s.feed(seg1 + d1, n1 - d1);
    uint8_t dg[32];
    s.final(dg);
    if (out)
        for (int k = 0; k < 32; ++k) out[k] = dg[k];
    if (expected) {
        bool same = true;
        for (int k = 0; k < 32; ++k) same &= dg[k] == expected[k];
        if (!same) {
            atomicAdd(&status->n_mismatch, 1);
            atomicCAS(&status->err, 0, (int32_t)KVG_ERR_DIGEST);
        }
    }
}

// sha256_serial_kernel's whole 64-byte blocks in the two-warp form: every
// lane of both warps runs the same chain (lane 0's result is kept), warp 1
// reads the message two blocks ahead, warp 0 runs the rounds; lane 0 of
// warp 0 then finishes the tail and the padding with the byte-wise hasher.
// For 4-byte aligned segments with seg0's length a multiple of 4.
__global__ void __launch_bounds__(64) sha256_serial_split_kernel(const uint8_t *seg0, uint64_t n0, const uint8_t *seg1,
                                                                 uint64_t n1, int32_t n_blocks, uint8_t *out,
                                                                 const uint8_t *expected, DevStatus *status,
                                                                 uint32_t one) {
    __shared__ __align__(16) uint32_t kw[2][64][kSplitChains];
    const int lane = threadIdx.x & 31;
    if (blockIdx.x != 0) return;
    if (threadIdx.x >= 32) {
        uint32_t n1w[16], n2w[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            n1w[i] = n_blocks > 0 ? msg_word(seg0, n0, seg1, (uint64_t)i) : 0u;
            n2w[i] = n_blocks > 1 ? msg_word(seg0, n0, seg1, 16ull + i) : 0u;
        }
        for (int blk = 0; blk < n_blocks; ++blk) {
            uint32_t w[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                w[i] = bswap(n1w[i]);
                n1w[i] = n2w[i];
            }
            if (blk + 2 < n_blocks) {
#pragma unroll
                for (int i = 0; i < 16; ++i) n2w[i] = msg_word(seg0, n0, seg1, 16ull * (blk + 2) + i);
            }
            split_hand_over(kw, w, blk, lane);
        }
        return;
    }
    uint32_t st[8];
    split_consume(st, kw, n_blocks, lane, one);
    if (lane != 0) return;
    Stream s;
    s.init(one);
#pragma unroll
    for (int i = 0; i < 8; ++i) s.st[i] = st[i];
    const uint64_t done = 64ull * (uint64_t)n_blocks;
    s.total = done;
    if (done < n0) s.feed(seg0 + done, n0 - done);
    const uint64_t d1 = done > n0 ? done - n0 : 0;
    if (d1 < n1) s.feed(seg1 + d1, n1 - d1);
    uint8_t dg[32];
    s.final(dg);
    if (out)
        for (int k = 0; k < 32; ++k) out[k] = dg[k];
    if (expected) {
        bool same = true;
        for (int k = 0; k < 32; ++k) same &= dg[k] == expected[k];
        if (!same) {
            atomicAdd(&status->n_mismatch, 1);
            atomicCAS(&status->err, 0, (int32_t)KVG_ERR_DIGEST);
        }
    }
}

}  // namespace

// The two-warp form is used for pages of whole 4 KiB leaves when a launch has
// at most two of its 32-chain CTAs per SM (leaves) or four (page digests,
// which read their input from L2); beyond that the one-warp forms keep more
// chains going per SM.  KVG_SHA_NO_SPLIT=1 turns it off.
static bool split_off() {
    static const bool off = env_knob("KVG_SHA_NO_SPLIT", 0) > 0;
    return off;
}

// Leaves per SM up to which a leaf-hashing launch takes the two-warp form:
// two of its CTAs per SM (four warps, one per scheduler).  A verified graft
// of 16 to 64 leaves per SM took 0.082-0.083 ms in it against 0.117 in the
// one-warp form; at 96 and 128 leaves per SM 0.130-0.137 against 0.118-0.121.
// A verified graft from pinned host memory keeps the one-warp form: its leaf
// loads outlast the rounds of a block in the two-warp form (the last chunk of
// the 12B block's host-store graft, 40 leaves per SM, made the e2e step
// 15.73-15.83 ms instead of 15.63-15.71).
static int split_leaves_per_sm() {
    static const int v = env_knob("KVG_SHA_SPLIT_LEAVES_PER_SM", 2 * kSplitChains);
    return v;
}

static int current_sm_count() {
    static int cache[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    if (!cache[dev]) cudaDeviceGetAttribute(&cache[dev], cudaDevAttrMultiProcessorCount, dev);
    return cache[dev];
}

cudaError_t launch_sha256_leaves(const PageSource &src, int64_t n_pages, uint32_t *leaf_words,
                                 int n_sm, cudaStream_t s) {
    const int64_t m = (int64_t)((src.page_bytes + kLeafBytes - 1) / kLeafBytes);
    const int64_t n = n_pages * m;
    if (n == 0) return cudaSuccess;
    if (!split_off() && src.page_bytes % kLeafBytes == 0 && n <= (int64_t)n_sm * split_leaves_per_sm()) {
        sha256_leaves_split_kernel<<<(int)((n + kSplitChains - 1) / kSplitChains), 64, 0, s>>>(src, n_pages, m,
                                                                                             leaf_words, 1u);
        count_launches(1);
        return cudaGetLastError();
    }
    int64_t grid = (n + 127) / 128;
    // One CTA per 128 leaves (no grid-stride cap by default): 4 CTAs of
    // 125 registers are resident per SM and the rest queue, which measured
    // 2-3% faster than a capped, striding grid.
    static const int ctas_per_sm = env_knob("KVG_SHA_CTAS_PER_SM", 0);
    if (ctas_per_sm > 0 && grid > (int64_t)n_sm * ctas_per_sm) grid = (int64_t)n_sm * ctas_per_sm;
    sha256_leaves_kernel<<<(int)grid, 128, 0, s>>>(src, n_pages, m, leaf_words, 1u);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_graft_verify(const GraftParams &p, uint32_t *leaf_words, int n_sm, cudaStream_t s, bool ring_ok,
                                bool split_ok) {
    const int64_t m = (int64_t)((p.page_bytes + kLeafBytes - 1) / kLeafBytes);
    const int64_t n = (int64_t)p.n_layers * 2 * p.npb * m;
    if (n == 0) return cudaSuccess;
    if (split_ok && !split_off() && p.page_bytes % kLeafBytes == 0 && n <= (int64_t)n_sm * split_leaves_per_sm()) {
        graft_verify_split_kernel<<<(int)((n + kSplitChains - 1) / kSplitChains), 64, 0, s>>>(p, m, leaf_words, 1u);
        count_launches(1);
        return cudaGetLastError();
    }
    int64_t grid = (n + 127) / 128;
    // One CTA per 128 leaves (no grid-stride cap by default): four CTAs of
    // the register form (125 registers) or five of the ring form (96) are
    // resident per SM and the rest queue.
    static const int ctas_per_sm = env_knob("KVG_SHA_CTAS_PER_SM", 0);
    if (ctas_per_sm > 0 && grid > (int64_t)n_sm * ctas_per_sm) grid = (int64_t)n_sm * ctas_per_sm;
    // a full wave of the ring form (five CTAs on every SM) or more, where the
    // caller allows it: the ring form; otherwise the register form (see
    // graft_verify_ring_kernel).  KVG_SHA_REGISTER_FORM=1 keeps the register
    // form for every size.
    static const bool regs_only = env_knob("KVG_SHA_REGISTER_FORM", 0) > 0;
    if (ring_ok && !regs_only && n >= (int64_t)n_sm * 5 * 128 && grid > (int64_t)n_sm * 4) {
        const size_t smem = (size_t)128 * kGraftVerifyRing * 64;  // 24 KiB of ring slots per CTA
        graft_verify_ring_kernel<<<(int)grid, 128, smem, s>>>(p, m, leaf_words, 1u);
    } else {
        graft_verify_kernel<<<(int)grid, 128, 0, s>>>(p, m, leaf_words, 1u);
    }
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_sha256_pages(const uint32_t *leaf_words, int64_t n_pages, int64_t leaves_per_page,
                                uint8_t *out, const uint8_t *expected, DevStatus *status,
                                int32_t seq, cudaStream_t s) {
    if (n_pages == 0) return cudaSuccess;
    if (!split_off() && n_pages <= (int64_t)current_sm_count() * 4 * kSplitChains) {
        sha256_pages_split_kernel<<<(int)((n_pages + kSplitChains - 1) / kSplitChains), 64, 0, s>>>(
            leaf_words, n_pages, leaves_per_page, out, expected, status, seq, 1u);
        count_launches(1);
        return cudaGetLastError();
    }
    sha256_pages_kernel<<<(int)((n_pages + 127) / 128), 128, 0, s>>>(leaf_words, n_pages,
                                                                     leaves_per_page, out,
                                                                     expected, status, seq, 1u);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_sha256_serial(const uint8_t *seg0, uint64_t n0, const uint8_t *seg1, uint64_t n1,
                                 uint8_t *out, const uint8_t *expected, DevStatus *status,
                                 cudaStream_t s) {
    const bool aligned = !((reinterpret_cast<uintptr_t>(seg0) | reinterpret_cast<uintptr_t>(seg1) | n0) & 3);
    const uint64_t n_blocks = (n0 + n1) / 64;
    if (!split_off() && aligned && n_blocks >= 1 && n_blocks < (1ull << 30)) {
        sha256_serial_split_kernel<<<1, 64, 0, s>>>(seg0, n0, seg1, n1, (int32_t)n_blocks, out, expected, status, 1u);
    } else {
        sha256_serial_kernel<<<1, 32, 0, s>>>(seg0, n0, seg1, n1, out, expected, status, 1u);
    }
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace kvg

/*
 * kvg_oracle.c — plain, slow, obviously-correct CPU oracle for the KV-state
 * graft hot path of "Byte-Exact KV-State Grafting" (arxiv 2607.14431).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product library links, loads or
 * calls this file; only the test-suite, the smoke check and the benchmark's
 * CPU-baseline leg do.  It shares no code, header, table or constant with the
 * CUDA path: every constant below is derived here from its published
 * definition.
 *
 * Contents (each function cites the passage it follows):
 *   - SHA-256 exactly as FIPS 180-4 defines it (the paper's digest, Sec. 3.2
 *     eq. for byte-exactness and Sec. 4.11 block digests).  The round
 *     constants K and initial hash H0 are computed from their definition
 *     (fractional parts of cube / square roots of the first primes) with
 *     exact integer roots, not typed in.
 *   - The two-level page digest: SHA-256 over the concatenated SHA-256 digests
 *     of consecutive 4096-byte leaves of a page.  The paper keeps its hashing
 *     scheme closed (Sec. 3.1); this leaf/page reading is ours.
 *   - bf16 round-to-nearest-even of an fp64 value (a single correct rounding).
 *   - Rotary position embedding rotation by an offset (Su et al.; the paper's
 *     relocation analysis, Sec. 4.2), in fp64.
 *   - Softmax attention for one decode query per head, in fp64 with
 *     max-subtraction (the decode step on top of a grafted prefix, Sec. 3.2 /
 *     Sec. 4.3).
 *
 * Parity pins for every function live in tests/test_oracle_pins.py.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>
#include <stdlib.h>
#include <fenv.h>

/* ------------------------------------------------------------------------ */
/* SHA-256 (FIPS 180-4)                                                     */
/* ------------------------------------------------------------------------ */

static uint32_t K256[64];
static uint32_t H256[8];
static int sha_ready = 0;

/* floor(cuberoot(x)) for x < 2^120, by bisection on 128-bit integers. */
static unsigned __int128 icbrt128(unsigned __int128 x) {
    unsigned __int128 lo = 0, hi = ((unsigned __int128)1) << 41;
    while (hi - lo > 1) {
        unsigned __int128 mid = (lo + hi) / 2;
        if (mid * mid * mid <= x) lo = mid; else hi = mid;
    }
    return lo;
}

/* floor(sqrt(x)) for x < 2^120, by bisection. */
static unsigned __int128 isqrt128(unsigned __int128 x) {
    unsigned __int128 lo = 0, hi = ((unsigned __int128)1) << 61;
    while (hi - lo > 1) {
        unsigned __int128 mid = (lo + hi) / 2;
        if (mid * mid <= x) lo = mid; else hi = mid;
    }
    return lo;
}

/* FIPS 180-4 sec. 4.2.2: K[t] = first 32 bits of the fractional part of the
 * cube root of the t-th prime; sec. 5.3.3: H0[i] = first 32 bits of the
 * fractional part of the square root of the i-th prime.
 * floor(frac(cbrt(p)) * 2^32) = floor(cbrt(p * 2^96)) mod 2^32. */
static void sha256_init_constants(void) {
    int primes[64];
    int n = 0;
    for (int c = 2; n < 64; ++c) {
        int is_p = 1;
        for (int d = 2; d * d <= c; ++d) if (c % d == 0) { is_p = 0; break; }
        if (is_p) primes[n++] = c;
    }
    for (int t = 0; t < 64; ++t) {
        unsigned __int128 x = ((unsigned __int128)primes[t]) << 96;
        K256[t] = (uint32_t)(icbrt128(x) & 0xffffffffu);
    }
    for (int i = 0; i < 8; ++i) {
        unsigned __int128 x = ((unsigned __int128)primes[i]) << 64;
        H256[i] = (uint32_t)(isqrt128(x) & 0xffffffffu);
    }
    sha_ready = 1;
}

static uint32_t rotr(uint32_t x, int n) { return (x >> n) | (x << (32 - n)); }

/* FIPS 180-4 sec. 6.2.2: one compression of a 64-byte message block. */
static void sha256_compress(uint32_t h[8], const uint8_t blk[64]) {
    uint32_t W[64];
    for (int t = 0; t < 16; ++t)
        W[t] = ((uint32_t)blk[4 * t] << 24) | ((uint32_t)blk[4 * t + 1] << 16) |
               ((uint32_t)blk[4 * t + 2] << 8) | (uint32_t)blk[4 * t + 3];
    for (int t = 16; t < 64; ++t) {
        uint32_t s0 = rotr(W[t - 15], 7) ^ rotr(W[t - 15], 18) ^ (W[t - 15] >> 3);
        uint32_t s1 = rotr(W[t - 2], 17) ^ rotr(W[t - 2], 19) ^ (W[t - 2] >> 10);
        W[t] = s1 + W[t - 7] + s0 + W[t - 16];
    }
    uint32_t a = h[0], b = h[1], c = h[2], d = h[3];
    uint32_t e = h[4], f = h[5], g = h[6], hh = h[7];
    for (int t = 0; t < 64; ++t) {
        uint32_t S1 = rotr(e, 6) ^ rotr(e, 11) ^ rotr(e, 25);
        uint32_t ch = (e & f) ^ ((~e) & g);
        uint32_t T1 = hh + S1 + ch + K256[t] + W[t];
        uint32_t S0 = rotr(a, 2) ^ rotr(a, 13) ^ rotr(a, 22);
        uint32_t maj = (a & b) ^ (a & c) ^ (b & c);
        uint32_t T2 = S0 + maj;
        hh = g; g = f; f = e; e = d + T1;
        d = c; c = b; b = a; a = T1 + T2;
    }
    h[0] += a; h[1] += b; h[2] += c; h[3] += d;
    h[4] += e; h[5] += f; h[6] += g; h[7] += hh;
}

/* FIPS 180-4 sec. 5.1.1 padding + sec. 6.2 hash computation. */
void ora_sha256(const uint8_t *msg, uint64_t n, uint8_t out[32]) {
    if (!sha_ready) sha256_init_constants();
    uint32_t h[8];
    memcpy(h, H256, sizeof h);
    uint64_t full = n / 64;
    for (uint64_t i = 0; i < full; ++i) sha256_compress(h, msg + 64 * i);
    uint8_t tail[128];
    uint64_t rem = n - 64 * full;
    memset(tail, 0, sizeof tail);
    if (rem) memcpy(tail, msg + 64 * full, rem);
    tail[rem] = 0x80;
    uint64_t tail_len = (rem + 1 + 8 <= 64) ? 64 : 128;
    uint64_t bits = n * 8;
    for (int i = 0; i < 8; ++i) tail[tail_len - 1 - i] = (uint8_t)(bits >> (8 * i));
    for (uint64_t off = 0; off < tail_len; off += 64) sha256_compress(h, tail + off);
    for (int i = 0; i < 8; ++i) {
        out[4 * i] = (uint8_t)(h[i] >> 24);
        out[4 * i + 1] = (uint8_t)(h[i] >> 16);
        out[4 * i + 2] = (uint8_t)(h[i] >> 8);
        out[4 * i + 3] = (uint8_t)h[i];
    }
}

/* Copies of the derived constants, so the tests can compare them with the
 * FIPS 180-4 definition independently. */
void ora_sha256_constants(uint32_t k_out[64], uint32_t h_out[8]) {
    if (!sha_ready) sha256_init_constants();
    memcpy(k_out, K256, sizeof K256);
    memcpy(h_out, H256, sizeof H256);
}

/* Two-level page digest (reading of the paper's per-block SHA-256, Sec. 4.11,
 * applied per page): leaf i = bytes [i*leaf, min((i+1)*leaf, page_bytes)) of
 * the page (the last leaf may be shorter);
 * digest = SHA-256( SHA-256(leaf_0) || ... || SHA-256(leaf_{m-1}) ),
 * m = ceil(page_bytes / leaf_bytes). */
int ora_page_digest(const uint8_t *page, uint64_t page_bytes, uint64_t leaf_bytes,
                    uint8_t out[32]) {
    if (leaf_bytes == 0 || page_bytes == 0) return -1;
    uint64_t m = (page_bytes + leaf_bytes - 1) / leaf_bytes;
    uint8_t *cat = (uint8_t *)malloc(32 * m);
    if (!cat) return -2;
    for (uint64_t i = 0; i < m; ++i) {
        uint64_t len = page_bytes - i * leaf_bytes;
        if (len > leaf_bytes) len = leaf_bytes;
        ora_sha256(page + i * leaf_bytes, len, cat + 32 * i);
    }
    ora_sha256(cat, 32 * m, out);
    free(cat);
    return 0;
}

/* Page digests of n_pages consecutive pages (independent, so optionally in
 * parallel across pages; each page's arithmetic is the serial definition). */
int ora_page_digests(const uint8_t *pages, uint64_t n_pages, uint64_t page_bytes,
                     uint64_t leaf_bytes, uint8_t *out) {
    int bad = 0;
    if (!sha_ready) sha256_init_constants();
#pragma omp parallel for schedule(static) reduction(| : bad)
    for (int64_t p = 0; p < (int64_t)n_pages; ++p)
        bad |= ora_page_digest(pages + (uint64_t)p * page_bytes, page_bytes, leaf_bytes,
                               out + 32 * (uint64_t)p) != 0;
    return bad ? -1 : 0;
}

/* ------------------------------------------------------------------------ */
/* bf16                                                                     */
/* ------------------------------------------------------------------------ */

/* Value of a bf16 bit pattern: the top 16 bits of an IEEE binary32. */
double ora_bf16_to_f64(uint16_t b) {
    uint32_t u = ((uint32_t)b) << 16;
    float f;
    memcpy(&f, &u, 4);
    return (double)f;
}

/* Correct round-to-nearest-even of a finite fp64 value to bf16 (8 exponent
 * bits, 7 stored mantissa bits, binary32 exponent range).  With e the binary
 * exponent of |x| (clamped at the smallest normal exponent -126), the bf16
 * quantum is 2^(e-7); x / quantum is exact in fp64, nearbyint() rounds it to
 * the nearest integer with ties to even, and the product is the rounded
 * value, exactly representable in binary32. */
uint16_t ora_bf16_rne(double x) {
    if (x == 0.0) {
        uint32_t u;
        float f = (float)x; /* keeps the sign of zero */
        memcpy(&u, &f, 4);
        return (uint16_t)(u >> 16);
    }
    int e;
    frexp(x, &e); /* |x| = m * 2^e, m in [0.5, 1) -> binary exponent e-1 */
    int be = e - 1;
    if (be < -126) be = -126;
    double q = ldexp(1.0, be - 7);
    double r = nearbyint(x / q) * q;
    float f = (float)r; /* exact: r has at most 8 significant bits */
    uint32_t u;
    memcpy(&u, &f, 4);
    return (uint16_t)(u >> 16);
}

void ora_bf16_rne_array(const double *x, uint64_t n, uint16_t *out) {
    for (uint64_t i = 0; i < n; ++i) out[i] = ora_bf16_rne(x[i]);
}

/* ------------------------------------------------------------------------ */
/* RoPE rotation by an offset (Sec. 4.2; Su et al.)                          */
/* ------------------------------------------------------------------------ */

/* Rotates one head row x[D] (bf16 bits) by the angle offset `delta` positions:
 * pair (a, b) of dimension index i < D/2 is rotated by delta * w_i,
 * w_i = theta^(-2i/D), as the complex product (x_a + i x_b) * exp(i delta w_i).
 * style 0 (half-split, "NeoX"): a = i, b = i + D/2.
 * style 1 (interleaved, "GPT-J"): a = 2i, b = 2i + 1.
 * Output y[D] in fp64. */
int ora_rope_rotate_row(const uint16_t *x, int D, double delta, double theta, int style,
                        double *y) {
    if (D <= 0 || D % 2) return -1;
    int half = D / 2;
    for (int i = 0; i < half; ++i) {
        int a = style == 0 ? i : 2 * i;
        int b = style == 0 ? i + half : 2 * i + 1;
        double w = pow(theta, -2.0 * (double)i / (double)D);
        double ang = delta * w;
        double c = cos(ang), s = sin(ang);
        double xa = ora_bf16_to_f64(x[a]), xb = ora_bf16_to_f64(x[b]);
        y[a] = xa * c - xb * s;
        y[b] = xa * s + xb * c;
    }
    return 0;
}

/* Same rotation on an fp64 row (used to check composition R(a)R(b) = R(a+b)). */
int ora_rope_rotate_row_f64(const double *x, int D, double delta, double theta, int style,
                            double *y) {
    if (D <= 0 || D % 2) return -1;
    int half = D / 2;
    for (int i = 0; i < half; ++i) {
        int a = style == 0 ? i : 2 * i;
        int b = style == 0 ? i + half : 2 * i + 1;
        double w = pow(theta, -2.0 * (double)i / (double)D);
        double ang = delta * w;
        double c = cos(ang), s = sin(ang);
        double xa = x[a], xb = x[b];
        y[a] = xa * c - xb * s;
        y[b] = xa * s + xb * c;
    }
    return 0;
}

/* Rotates n rows (row stride D) and rounds each result to bf16 (RNE). */
int ora_rope_rotate_rows_bf16(const uint16_t *x, uint64_t n, int D, double delta,
                              double theta, int style, uint16_t *out) {
    double *y = (double *)malloc(sizeof(double) * (size_t)D);
    if (!y) return -2;
    for (uint64_t r = 0; r < n; ++r) {
        if (ora_rope_rotate_row(x + r * (uint64_t)D, D, delta, theta, style, y)) {
            free(y);
            return -1;
        }
        for (int d = 0; d < D; ++d) out[r * (uint64_t)D + d] = ora_bf16_rne(y[d]);
    }
    free(y);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* fp8 E4M3 KV codes (quantized KV blocks: the block's size depends on the   */
/* cache's quantization, Sec. 4.4).  Format: sign, 4 exponent bits (bias 7), */
/* 3 mantissa bits; exponent field 0 holds subnormals m * 2^-9; the code     */
/* S.1111.111 is NaN; there are no infinities; the largest finite is 448.    */
/* ------------------------------------------------------------------------ */

double ora_e4m3_to_f64(uint8_t c) {
    int s = c >> 7, e = (c >> 3) & 15, m = c & 7;
    double v;
    if (e == 15 && m == 7) return NAN;
    if (e == 0)
        v = ldexp((double)m, -9);
    else
        v = ldexp(1.0 + m / 8.0, e - 7);
    return s ? -v : v;
}

/* Round-to-nearest-even onto the E4M3 grid, saturating: magnitudes above the
 * largest finite (448) give 448; NaN gives the NaN code 0x7F. */
uint8_t ora_e4m3_rne_sat(double x) {
    if (isnan(x)) return 0x7F;
    uint8_t s = signbit(x) ? 0x80 : 0x00;
    double a = fabs(x);
    if (a > 448.0) return s | 0x7E;
    if (a < ldexp(1.0, -6)) {
        /* subnormal grid m * 2^-9, m in 0..8 (8 is the smallest normal) */
        double q = nearbyint(a / ldexp(1.0, -9));
        return s | (uint8_t)q; /* q == 8 encodes exponent field 1, mantissa 0 */
    }
    int e;
    frexp(a, &e);       /* a = f * 2^e, f in [0.5, 1): a in [2^(e-1), 2^e) */
    int E = e - 1;      /* a in [2^E, 2^(E+1)), E in [-6, 8] */
    double q = nearbyint(a / ldexp(1.0, E - 3)); /* 8 .. 16 units of 2^(E-3) */
    if (q == 16.0) {
        q = 8.0;
        E += 1;
    }
    if (E > 8 || (E == 8 && q > 14.0)) return s | 0x7E; /* cannot happen after the clamp */
    return s | (uint8_t)(((E + 7) << 3) | ((int)q - 8));
}

/* Quantization of bf16 values with a per-tensor scale: r = 1 / scale as an
 * fp32 quotient; each bf16 value as fp32 times r, rounded once to fp32; then
 * E4M3 RNE with saturation. */
void ora_e4m3_quantize_bf16(const uint16_t *x, uint64_t n, float scale, uint8_t *out) {
    float r = 1.0f / scale;
    for (uint64_t i = 0; i < n; ++i) {
        float f = (float)ora_bf16_to_f64(x[i]);
        float y = f * r;
        out[i] = ora_e4m3_rne_sat((double)y);
    }
}

/* Dequantized values: code value times the scale, in fp64 (exact). */
void ora_e4m3_dequant(const uint8_t *c, uint64_t n, float scale, double *out) {
    for (uint64_t i = 0; i < n; ++i) out[i] = ora_e4m3_to_f64(c[i]) * (double)scale;
}

/* ------------------------------------------------------------------------ */
/* Decode attention in fp64 (Sec. 3.2 / Sec. 4.3: the query decoded on top   */
/* of the restored prefix attends to every cached token).                   */
/* ------------------------------------------------------------------------ */

/* One query head over one KV head's context.
 *   q[D]                         bf16 bits
 *   k, v: n rows, row r at k + r*row_stride (bf16 bits, D contiguous values)
 *   o[D]                         fp64 output
 * s_t = scale * sum_d q_d k_{t,d};  m = max_t s_t;  w_t = exp(s_t - m);
 * o = sum_t w_t v_t / sum_t w_t.  n == 0 leaves o = 0. */
void ora_attention_head(const uint16_t *q, const uint16_t *k, const uint16_t *v, uint64_t n,
                        uint64_t row_stride, int D, double scale, double *o) {
    for (int d = 0; d < D; ++d) o[d] = 0.0;
    if (n == 0) return;
    double *s = (double *)malloc(sizeof(double) * n);
    if (!s) return;
    double m = -INFINITY;
    for (uint64_t t = 0; t < n; ++t) {
        double acc = 0.0;
        for (int d = 0; d < D; ++d)
            acc += ora_bf16_to_f64(q[d]) * ora_bf16_to_f64(k[t * row_stride + d]);
        s[t] = acc * scale;
        if (s[t] > m) m = s[t];
    }
    double l = 0.0;
    for (uint64_t t = 0; t < n; ++t) {
        double w = exp(s[t] - m);
        l += w;
        for (int d = 0; d < D; ++d) o[d] += w * ora_bf16_to_f64(v[t * row_stride + d]);
    }
    for (int d = 0; d < D; ++d) o[d] /= l;
    free(s);
}

/* Grouped-query decode attention over a logical (unpaged) context.
 *   q   [Hq][D]        bf16 bits
 *   k,v [n][Hkv][D]    bf16 bits (token-major, as written by a prefill)
 *   o   [Hq][D]        fp64
 * Query head h reads KV head h / (Hq / Hkv).  Heads are independent, so the
 * loop over heads may run in parallel; each head is the serial definition. */
int ora_gqa_decode(const uint16_t *q, const uint16_t *k, const uint16_t *v, uint64_t n,
                   int Hq, int Hkv, int D, double scale, double *o) {
    if (Hkv <= 0 || Hq % Hkv) return -1;
    int G = Hq / Hkv;
#pragma omp parallel for schedule(dynamic, 1)
    for (int h = 0; h < Hq; ++h) {
        int g = h / G;
        ora_attention_head(q + (uint64_t)h * D, k + (uint64_t)g * D, v + (uint64_t)g * D, n,
                           (uint64_t)Hkv * D, D, scale, o + (uint64_t)h * D);
    }
    return 0;
}

/* The same attention with K and V given as fp64 values (dequantized rows):
 * identical steps, only the loads differ. */
static void attention_head_f64kv(const uint16_t *q, const double *k, const double *v, uint64_t n,
                                 uint64_t row_stride, int D, double scale, double *o) {
    for (int d = 0; d < D; ++d) o[d] = 0.0;
    if (n == 0) return;
    double *s = (double *)malloc(sizeof(double) * n);
    if (!s) return;
    double m = -INFINITY;
    for (uint64_t t = 0; t < n; ++t) {
        double acc = 0.0;
        for (int d = 0; d < D; ++d) acc += ora_bf16_to_f64(q[d]) * k[t * row_stride + d];
        s[t] = acc * scale;
        if (s[t] > m) m = s[t];
    }
    double l = 0.0;
    for (uint64_t t = 0; t < n; ++t) {
        double w = exp(s[t] - m);
        l += w;
        for (int d = 0; d < D; ++d) o[d] += w * v[t * row_stride + d];
    }
    for (int d = 0; d < D; ++d) o[d] /= l;
    free(s);
}

int ora_gqa_decode_f64kv(const uint16_t *q, const double *k, const double *v, uint64_t n, int Hq, int Hkv,
                         int D, double scale, double *o) {
    if (Hkv <= 0 || Hq % Hkv) return -1;
    int G = Hq / Hkv;
#pragma omp parallel for schedule(dynamic, 1)
    for (int h = 0; h < Hq; ++h) {
        int g = h / G;
        attention_head_f64kv(q + (uint64_t)h * D, k + (uint64_t)g * D, v + (uint64_t)g * D, n,
                             (uint64_t)Hkv * D, D, scale, o + (uint64_t)h * D);
    }
    return 0;
}

int ora_omp_threads(void) {
#ifdef _OPENMP
    extern int omp_get_max_threads(void);
    return omp_get_max_threads();
#else
    return 1;
#endif
}

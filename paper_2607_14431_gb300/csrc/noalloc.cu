// noalloc.cu — decode attention for callers that cannot allocate GPU memory.
//
// kvg_decode_attention() keeps its split-K partial results in per-cache
// scratch that it grows with cudaMalloc on first use (and whenever a larger
// batch or context needs more).  Some callers cannot allow that:
//   - serving loops with a latency budget: cudaMalloc and cudaFree
//     synchronise the whole device, stalling every stream in the process;
//   - processes whose HBM is reserved up front by another allocator (a
//     framework's caching allocator holding nearly all memory), where a new
//     cudaMalloc can fail with out-of-memory at an arbitrary request;
//   - deployments that fix their memory footprint at start-up and must not
//     fail for lack of memory once serving.
// kvg_decode_attention_noalloc() runs the same kernels with the partials in
// the file-scope device array below instead, and calls no allocating routine.
#include <cstdio>
#include <cstdlib>
#include <mutex>
#include <string>

#include "common.cuh"

namespace {

// Scratch for the split-K partials: float o[units][splits][G][D] followed by
// float2 (m, l)[units][splits][G].  Every GPU that loads the library holds it
// until the process exits.
constexpr size_t kScratchBytes = 16u << 20;
static __device__ __align__(256) unsigned char g_decode_scratch[kScratchBytes];

// Device address of g_decode_scratch per device ordinal.  In host code the
// symbol names a host-side stand-in, so the address must come from
// cudaGetSymbolAddress with that device current.
constexpr int kMaxDevices = 64;
std::mutex g_mu;
void *g_scratch_dev[kMaxDevices] = {};

// The split plan of kvg_decode_attention: about KVG_SPLIT_WAVES (default 16)
// CTAs per SM over the whole call.
int split_waves() {
    static int w = [] {
        const char *e = getenv("KVG_SPLIT_WAVES");
        int v = e ? atoi(e) : 0;
        return v > 0 ? v : 16;
    }();
    return w;
}

}  // namespace

namespace kvg {
// Read-only views of a cache's geometry and host bookkeeping (runtime.cu).
struct CacheShape {
    int32_t n_layers, n_kv_heads, head_dim, page_size, n_pages, max_seqs, max_pages, device, n_sm;
    uint8_t *pool;
    int32_t *page_table, *page_fill;
    DevStatus *status;
};
bool cache_shape(const kvg_cache *c, CacheShape *out);
int32_t cache_seq_pages(const kvg_cache *c, int32_t seq);
void set_last_error(const char *msg);
}  // namespace kvg

using namespace kvg;

extern "C" kvg_status kvg_decode_attention_noalloc(kvg_cache *c, int32_t layer, const int32_t *seq_ids,
                                                   int32_t B, const void *q, int32_t n_q_heads, void *out,
                                                   float scale, void *stream) {
    CacheShape cs;
    if (!c || !seq_ids || !q || !out || !cache_shape(c, &cs)) {
        set_last_error("null argument");
        return KVG_ERR_ARG;
    }
    auto reject = [](kvg_status st, const std::string &m) {
        set_last_error(m.c_str());
        return st;
    };
    if (layer < -1 || layer >= cs.n_layers) return reject(KVG_ERR_ARG, "bad layer");
    if (B <= 0 || B > 4096) return reject(KVG_ERR_ARG, "B must be in [1, 4096]");
    if (n_q_heads <= 0 || n_q_heads % cs.n_kv_heads)
        return reject(KVG_ERR_ARG, "n_q_heads must be a multiple of n_kv_heads");
    const int G = n_q_heads / cs.n_kv_heads;
    if (!decode_supported(cs.head_dim, G)) return reject(KVG_ERR_ARG, "unsupported head_dim / group");
    if ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(out)) & 15)
        return reject(KVG_ERR_ARG, "q/out must be 16-byte aligned");
    if (cs.device < 0 || cs.device >= kMaxDevices) return reject(KVG_ERR_ARG, "device ordinal out of range");
    int64_t max_np = 0, total_np = 0;
    for (int32_t b = 0; b < B; ++b) {
        if (seq_ids[b] < 0 || seq_ids[b] >= cs.max_seqs) return reject(KVG_ERR_ARG, "bad seq id");
        const int64_t np = cache_seq_pages(c, seq_ids[b]);
        max_np = np > max_np ? np : max_np;
        total_np += np;
    }
    const int Lrun = layer < 0 ? cs.n_layers : 1;
    const int64_t bchunk = B < kMaxBatchPerLaunch ? B : kMaxBatchPerLaunch;
    // bytes of one split's partials for the whole launch
    const uint64_t per_split = (uint64_t)Lrun * bchunk * cs.n_kv_heads * G * ((uint64_t)cs.head_dim * 4 + 8);
    // (m, l) start 256-byte aligned after o: keep 256 bytes of slack
    const int64_t s_cap = (int64_t)((kScratchBytes - 256) / per_split);
    if (s_cap < 1) {
        char m[256];
        snprintf(m, sizeof m,
                 "noalloc decode: %d layer(s) x %lld batch rows need %llu bytes of partials per split, "
                 "above the %zu-byte static scratch; use kvg_decode_attention or fewer rows per call",
                 Lrun, (long long)bchunk, (unsigned long long)per_split, kScratchBytes);
        return reject(KVG_ERR_CAPACITY, m);
    }
    // same split plan as kvg_decode_attention, capped so the partials fit
    const int64_t work = (int64_t)Lrun * cs.n_kv_heads * total_np;
    const int64_t target = (int64_t)cs.n_sm * split_waves();
    int64_t pps = work > 0 ? (work + target - 1) / target : 1;
    if (pps < 1 || max_np == 0) pps = 1;
    int64_t S = max_np > 0 ? (max_np + pps - 1) / pps : 1;
    if (S > s_cap) {
        S = s_cap;
        pps = (max_np + S - 1) / S;
        S = (max_np + pps - 1) / pps;
    }

    int prev = -1;
    cudaGetDevice(&prev);
    if (prev != cs.device && cudaSetDevice(cs.device) != cudaSuccess)
        return reject(KVG_ERR_CUDA, "cudaSetDevice failed");
    struct Restore {
        int prev, dev;
        ~Restore() {
            if (prev >= 0 && prev != dev) cudaSetDevice(prev);
        }
    } restore{prev, cs.device};
    void *scratch = nullptr;
    {
        // first call on a device: look up the array's device address with
        // that device current (no allocation happens here)
        std::lock_guard<std::mutex> lk(g_mu);
        if (!g_scratch_dev[cs.device]) {
            cudaError_t e = cudaGetSymbolAddress(&g_scratch_dev[cs.device], g_decode_scratch);
            if (e != cudaSuccess) {
                g_scratch_dev[cs.device] = nullptr;
                return reject(KVG_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
            }
        }
        scratch = g_scratch_dev[cs.device];
    }
    const size_t units = (size_t)Lrun * bchunk * cs.n_kv_heads * S * G;
    float *part_o = static_cast<float *>(scratch);
    float2 *part_ml = reinterpret_cast<float2 *>(static_cast<unsigned char *>(scratch) +
                                                 ((units * cs.head_dim * 4 + 255) / 256) * 256);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    for (int64_t b0 = 0; b0 < B; b0 += kMaxBatchPerLaunch) {
        const int32_t nb = (int32_t)((B - b0) < kMaxBatchPerLaunch ? (B - b0) : kMaxBatchPerLaunch);
        DecodeParams p{};
        p.pool = cs.pool;
        p.pool_pages = cs.n_pages;
        p.n_kv_heads = cs.n_kv_heads;
        p.page_size = cs.page_size;
        p.n_q_heads = n_q_heads;
        p.layer0 = layer < 0 ? 0 : layer;
        p.n_layers_run = Lrun;
        p.B = nb;
        p.n_splits = (int32_t)S;
        p.pages_per_split = (int32_t)pps;
        p.page_table = cs.page_table;
        p.page_fill = cs.page_fill;
        p.max_pages = cs.max_pages;
        p.q = static_cast<const __nv_bfloat16 *>(q);
        p.q_row_stride_b = B;
        p.b0 = (int32_t)b0;
        p.qscale = scale * 1.4426950408889634f;
        p.part_o = part_o;
        p.part_ml = part_ml;
        p.status = cs.status;
        for (int32_t i = 0; i < nb; ++i) {
            p.rows.seq[i] = seq_ids[b0 + i];
            p.rows.npages[i] = cache_seq_pages(c, seq_ids[b0 + i]);
        }
        cudaError_t e = launch_decode(cs.head_dim, G, p, st);
        if (e != cudaSuccess) return reject(KVG_ERR_CUDA, std::string("decode launch: ") + cudaGetErrorString(e));
        CombineParams cp{};
        cp.part_o = part_o;
        cp.part_ml = part_ml;
        cp.out = static_cast<__nv_bfloat16 *>(out);
        cp.n_kv_heads = cs.n_kv_heads;
        cp.n_q_heads = n_q_heads;
        cp.n_splits = (int32_t)S;
        cp.B = nb;
        cp.q_row_stride_b = B;
        cp.b0 = (int32_t)b0;
        e = launch_combine(cs.head_dim, G, cp, Lrun, nb, st);
        if (e != cudaSuccess) return reject(KVG_ERR_CUDA, std::string("combine launch: ") + cudaGetErrorString(e));
    }
    return KVG_OK;
}

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
#include <vector>

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
std::mutex g_mu;
void *g_scratch_dev[kvg::kMaxDevices] = {};

}  // namespace

namespace kvg {
cudaError_t noalloc_prepare_device(int device) {
    if (device < 0 || device >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_mu);
    if (g_scratch_dev[device]) return cudaSuccess;
    void *p = nullptr;
    // with the device current: resolves (and, under lazy module loading,
    // loads) this file's module on it, which places the array in its memory
    const cudaError_t e = cudaGetSymbolAddress(&p, g_decode_scratch);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return e;
    }
    g_scratch_dev[device] = p;
    return cudaSuccess;
}
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
    const bool fp8 = cs.kv_dtype == KVG_KV_E4M3;
    if (!decode_supported(cs.head_dim, G, fp8)) return reject(KVG_ERR_ARG, "unsupported head_dim / group");
    if ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(out)) & 15)
        return reject(KVG_ERR_ARG, "q/out must be 16-byte aligned");
    if (cs.device < 0 || cs.device >= kMaxDevices) return reject(KVG_ERR_ARG, "device ordinal out of range");
    for (int32_t b = 0; b < B; ++b)
        if (seq_ids[b] < 0 || seq_ids[b] >= cs.max_seqs) return reject(KVG_ERR_ARG, "bad seq id");
    // the launches (as kvg_decode_attention makes them); host memory only
    std::vector<DecodeParams> plan;
    int64_t units = 0;
    const kvg_status pst = cache_plan_decode(c, layer, seq_ids, B, &plan, &units);
    if (pst != KVG_OK) return pst;
    // partials: (units + workers) slots of G * (4 * head_dim + 8) bytes; the
    // (m, l) part starts 256-byte aligned after o, so keep 256 bytes of slack
    const uint64_t per_slot = (uint64_t)G * ((uint64_t)cs.head_dim * 4 + 8);
    const int64_t cap_slots = (int64_t)((kScratchBytes - 256) / per_slot);
    if (cap_slots - units < 1) {
        char m[320];
        snprintf(m, sizeof m,
                 "noalloc decode: %lld units (layers x batch rows x kv heads of one launch) need at least %llu "
                 "bytes of partials, above the %zu-byte static scratch; use kvg_decode_attention or fewer rows "
                 "per call",
                 (long long)units, (unsigned long long)((units + 1) * per_slot), kScratchBytes);
        return reject(KVG_ERR_CAPACITY, m);
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
        // the address was looked up when the cache was created on this
        // device (kvg_cache_create); this call only reads it
        std::lock_guard<std::mutex> lk(g_mu);
        scratch = g_scratch_dev[cs.device];
    }
    if (!scratch) return reject(KVG_ERR_CUDA, "static decode scratch was not set up on the cache's device");
    const int w_max = decode_max_warps(cs.head_dim, G, fp8, cs.n_sm);
    if (w_max <= 0) return reject(KVG_ERR_CUDA, "decode kernel cannot be made resident");
    const int64_t w_cap = cap_slots - units < w_max ? cap_slots - units : w_max;
    const size_t slots = (size_t)units + (size_t)w_cap;
    float *part_o = static_cast<float *>(scratch);
    float2 *part_ml = reinterpret_cast<float2 *>(static_cast<unsigned char *>(scratch) +
                                                 ((slots * G * cs.head_dim * 4 + 255) / 256) * 256);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    for (DecodeParams &p : plan) {
        p.n_warps = (int32_t)(p.n_tiles < w_cap ? (p.n_tiles > 1 ? p.n_tiles : 1) : w_cap);
        p.n_q_heads = n_q_heads;
        p.q = static_cast<const __nv_bfloat16 *>(q);
        p.q_row_stride_b = B;
        p.qscale = scale * 1.4426950408889634f * (fp8 ? cs.k_scale : 1.f);
        p.vscale = fp8 ? cs.v_scale : 1.f;
        p.part_o = part_o;
        p.part_ml = part_ml;
        p.out = static_cast<__nv_bfloat16 *>(out);
        cudaError_t e = launch_decode(cs.head_dim, G, fp8, p, *cs.pool_map, st);
        if (e != cudaSuccess) return reject(KVG_ERR_CUDA, std::string("decode launch: ") + cudaGetErrorString(e));
        e = launch_combine(cs.head_dim, G, p, st);
        if (e != cudaSuccess) return reject(KVG_ERR_CUDA, std::string("combine launch: ") + cudaGetErrorString(e));
    }
    return KVG_OK;
}

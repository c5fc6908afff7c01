// decode_noalloc.cu -- attn_decode_noalloc: the decode stage for callers that cannot
// allocate device memory.
//
// Who needs it: code that runs where cudaMalloc is not available or not allowed --
// for example inside an allocator-owning framework that hands out only its own
// pre-reserved buffers, in a process whose device memory is fully provisioned up
// front, or in a callback that must not touch the allocator.  Such a caller cannot
// create an attn_ctx (attn_create allocates the tables and the split-KV partials).
//
// This entry point runs the same kernels as attn_decode (K3 with the new token's
// append; for head_dim 64 also K4, which merges the splits) but needs no context: the
// caller passes every input and output, including the RoPE tables and the error word,
// and the split-KV partials and merge counters live in the file-scope arrays below,
// which the library holds on every device that loads it until the process exits.
// Nothing is allocated or freed.
//
// Host code must not pass `g_noalloc_scratch` itself to a kernel: in host code that
// name denotes a host-side shadow, not device memory.  The device address is looked
// up with cudaGetSymbolAddress once per device (with that device current) on the
// first call made on that device, and cached.  A cudaDeviceReset unloads the module and
// with it that set-up (the cached addresses and the kernels' shared-memory limits):
// after one, the process must not call this entry point on that device again.
#include <cuda_runtime.h>

#include <mutex>

#include "attn.h"
#include "internal.h"

namespace {

// Split-KV partials of attn_decode_noalloc: [B*Hq*nsplit*D] accumulators followed by
// [B*Hq*nsplit*2] (max, sum) pairs.  Shared by every call on the device.
static __device__ __align__(256) float g_noalloc_scratch[ATTN_NOALLOC_SCRATCH_FLOATS];
// Counters of the tensor-core decode for up to kNoallocCounters (sequence, kv head) items
// (decode_tc_counter_ints of them); zero at load and left zero by every launch.
// B*Hkv <= B*Hq <= scratch / (D + 2) < 8192.
constexpr int kNoallocCounters = 8192;
static __device__ __align__(16) int g_noalloc_counters[5 * kNoallocCounters + 1] = {0};

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
float* g_scratch_ptr[kMaxDevices] = {};
int* g_counter_ptr[kMaxDevices] = {};
int g_num_sms[kMaxDevices] = {};
attn::PFN_encodeTiled g_encode = nullptr;

// Per-device set-up, on the current device: the device address of the scratch
// array, the SM count, the kernels' shared-memory limits and (once per process)
// the driver's tensor-map encoder.  Returns ATTN_OK, ATTN_EARCH or ATTN_ECUDA.
int setup_device(int dev, float** scratch, int** counters, int* num_sms) {
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (g_encode == nullptr) {
        cudaDriverEntryPointQueryResult qres;
        void* fn = nullptr;
        const cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                                               &qres);
        if (e != cudaSuccess) return attn::record_cuda_error(e, "attn_decode_noalloc: cuTensorMapEncodeTiled entry point");
        if (qres != cudaDriverEntryPointSuccess || fn == nullptr) {
            attn::record_error_text("attn_decode_noalloc: the driver has no cuTensorMapEncodeTiled");
            return ATTN_ECUDA;
        }
        g_encode = reinterpret_cast<attn::PFN_encodeTiled>(fn);
    }
    if (g_scratch_ptr[dev] == nullptr) {
        int major = 0, minor = 0, sms = 0;
        cudaError_t e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return attn::record_cuda_error(e, "attn_decode_noalloc: device attributes");
        if (major != 10 || minor != 3) return ATTN_EARCH;
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return attn::record_cuda_error(e, "attn_decode_noalloc: scratch array address");
        void* pc = nullptr;
        e = cudaGetSymbolAddress(&pc, g_noalloc_counters);
        if (e != cudaSuccess) return attn::record_cuda_error(e, "attn_decode_noalloc: counter array address");
        e = attn::configure_decode();
        if (e == cudaSuccess) e = attn::configure_decode_tc();
        if (e != cudaSuccess) return attn::record_cuda_error(e, "attn_decode_noalloc: kernel attributes");
        g_counter_ptr[dev] = static_cast<int*>(pc);
        g_num_sms[dev] = sms;
        g_scratch_ptr[dev] = static_cast<float*>(p);
    }
    *scratch = g_scratch_ptr[dev];
    *counters = g_counter_ptr[dev];
    *num_sms = g_num_sms[dev];
    return ATTN_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" int attn_decode_noalloc(const attn_cfg* cfg, const float* d_cos, const float* d_sin, const uint16_t* q,
                                   const uint16_t* k, const uint16_t* v, const int32_t* d_hist_len,
                                   uint16_t* k_cache, uint16_t* v_cache, uint16_t* out, int32_t* d_err,
                                   attn_stream_t stream) {
    if (cfg == nullptr || d_cos == nullptr || d_sin == nullptr || q == nullptr || k == nullptr || v == nullptr ||
        d_hist_len == nullptr || k_cache == nullptr || v_cache == nullptr || out == nullptr || d_err == nullptr)
        return ATTN_EINVAL;
    if (cfg->batch < 1 || cfg->batch > 65535 || cfg->n_q_heads < 1 || cfg->n_kv_heads < 1 ||
        cfg->n_q_heads % cfg->n_kv_heads != 0 || cfg->n_q_heads / cfg->n_kv_heads > 16 ||
        (cfg->head_dim != 64 && cfg->head_dim != 128) || cfg->max_len < 1 || cfg->max_len > (1 << 20))
        return ATTN_EINVAL;
    if (!aligned16(d_cos) || !aligned16(d_sin) || !aligned16(q) || !aligned16(k) || !aligned16(v) ||
        !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(out) ||
        (reinterpret_cast<uintptr_t>(d_hist_len) & 3u) || (reinterpret_cast<uintptr_t>(d_err) & 3u))
        return ATTN_EINVAL;
    // Partials need B*Hq*(D+2) floats per split; at least one split must fit.
    const long long per_split = static_cast<long long>(cfg->batch) * cfg->n_q_heads * (cfg->head_dim + 2);
    if (per_split > ATTN_NOALLOC_SCRATCH_FLOATS) return ATTN_EINVAL;

    int dev = 0;
    const cudaError_t de = cudaGetDevice(&dev);
    if (de != cudaSuccess) return attn::record_cuda_error(de, "attn_decode_noalloc: cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) {
        attn::record_error_text("attn_decode_noalloc: device ordinal beyond the library's table of 64 devices");
        return ATTN_ECUDA;
    }
    float* scratch = nullptr;
    int* counters = nullptr;
    int num_sms = 0;
    const int rc = setup_device(dev, &scratch, &counters, &num_sms);
    if (rc != ATTN_OK) return rc;

    // Same split rule as attn_decode, capped by what the scratch array holds.
    const attn::Shape s{cfg->batch, cfg->n_q_heads, cfg->n_kv_heads, cfg->head_dim, cfg->max_len};
    const long long fit = ATTN_NOALLOC_SCRATCH_FLOATS / per_split;
    const int cap = static_cast<int>(fit < 256 ? fit : 256);
    const bool tc = cfg->head_dim == 128;
    int nsplit = tc ? attn::decode_tc_num_splits(s, num_sms) : attn::decode_num_splits(s, num_sms, cap);
    nsplit = nsplit < cap ? nsplit : cap;
    float* part_o = scratch;
    float* part_ml = scratch + static_cast<size_t>(cfg->batch) * cfg->n_q_heads * nsplit * cfg->head_dim;

    attn::DecodeMaps maps;
    const cudaError_t me = tc ? attn::make_decode_tc_maps(g_encode, s, k_cache, v_cache, &maps)
                              : attn::make_decode_maps(g_encode, s, k_cache, v_cache, &maps);
    if (me != cudaSuccess) {
        attn::record_error_text("attn_decode_noalloc: cuTensorMapEncodeTiled failed for the caches");
        return ATTN_ECUDA;
    }
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (tc && static_cast<long long>(cfg->batch) * cfg->n_kv_heads > kNoallocCounters) return ATTN_EINVAL;
    cudaError_t e = tc ? attn::launch_decode_tc(s, maps, q, k, v, d_hist_len, 0, k_cache, v_cache, d_cos, d_sin, part_o,
                                                part_ml, counters, nsplit, out, d_err, false, 1, st, false,
                                                attn::kWaitLimitNs, num_sms)
                       : attn::launch_decode_split(s, maps, q, k, v, d_hist_len, 0, k_cache, v_cache, d_cos, d_sin,
                                                   part_o, part_ml, nsplit, d_err, st);
    if (e == cudaSuccess && !tc) e = attn::launch_decode_combine(s, d_hist_len, 0, part_o, part_ml, nsplit, out, st);
    return e == cudaSuccess ? ATTN_OK : attn::record_cuda_error(e, "attn_decode_noalloc: launch");
}

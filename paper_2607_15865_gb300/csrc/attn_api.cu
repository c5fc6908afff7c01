// attn_api.cu -- host side of the C ABI declared in include/attn.h.
//
// Validates arguments, owns the per-shape context (RoPE tables, decode split-KV
// partials, device error word), builds the TMA tensor maps for K2, and enqueues
// the kernels of each stage on the caller's stream:
//   prefill / prefill_kv : K1 rope_append (new k rotated + k, v appended in place)
//                          -> K2 flash_fwd (q rotated in-kernel, causal attention)
//   decode               : K3 decode_split (new k rotated + k, v appended at slot
//                          hist_len[b], read on the device) -> K4 decode_combine
// No call allocates, frees or synchronises except attn_create/attn_destroy and
// attn_device_error.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <new>
#include <vector>

#include "attn.h"
#include "internal.h"

struct attn_ctx {
    attn_cfg cfg;
    attn::Shape shape;
    int device;
    int num_sms;
    int nsplit_max;
    float* d_cos;       // RoPE tables [max_len][D/2]
    float* d_sin;
    float* d_cos_t;     // the same in groups of four pairs, [D/8][max_len][4] (flash_fwd's q rows)
    float* d_sin_t;
    float* d_part_o;
    float* d_part_ml;
    int* d_counters;    // decode counters, [2][B * Hkv] (merge count, tile claims), zero between launches
    uint16_t* d_lq;     // decode layer: q, k, v of the fused QKV projection and the attention
    uint16_t* d_lk;     // output, bf16 [B][Hq*D], [B][Hkv*D], [B][Hkv*D], [B][Hq*D]
    uint16_t* d_lv;
    uint16_t* d_lo;
    float* d_flash_o;   // flash tail pieces: [num_sms * 256, D] partial O
    float* d_flash_ml;  // and [num_sms * 256, 2] (m, l)
    int* d_err;
    PFN_cuTensorMapEncodeTiled_v12000 encode;
    // decode tensor maps of the last cache pair seen
    const uint16_t* dec_k;
    const uint16_t* dec_v;
    attn::DecodeMaps dec_maps;
    // kernel timing: event pairs recorded around each launch while enabled
    std::vector<cudaEvent_t> ev;
    std::vector<int> ev_kind;
    int ev_used;
    long long launches[ATTN_NUM_KERNELS];
    uint64_t wait_ns;  // limit of the kernels' bounded waits (attn_set_wait_limit)
};

namespace {

thread_local char g_cuda_msg[256] = "no error";

// New tokens per sequence of one multi-token decode call, and the column groups of 16
// (query head, token) columns that many take at the largest group size (16 heads).
constexpr int kMaxDraftTokens = 16;
constexpr int kMaxColumnGroups = 16;

// Per device: whether it is an sm_103 part (attn_w4bf16_gemv checks once per device).
constexpr int kArchCacheDevices = 64;
std::atomic<int> g_arch_ok[kArchCacheDevices];

int cuda_fail(cudaError_t e, const char* where) {
    std::snprintf(g_cuda_msg, sizeof g_cuda_msg, "%s: %s (%s)", where, cudaGetErrorName(e), cudaGetErrorString(e));
    return ATTN_ECUDA;
}
}  // namespace

namespace attn {
int record_cuda_error(cudaError_t e, const char* where) { return cuda_fail(e, where); }
void record_error_text(const char* text) { std::snprintf(g_cuda_msg, sizeof g_cuda_msg, "%s", text); }
}  // namespace attn

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool cfg_valid(const attn_cfg* c) {
    if (c == nullptr) return false;
    if (c->batch < 1 || c->batch > 65535) return false;
    if (c->n_q_heads < 1 || c->n_kv_heads < 1 || c->n_q_heads % c->n_kv_heads != 0) return false;
    if (c->n_q_heads / c->n_kv_heads > 16 || c->n_q_heads > 65535) return false;
    if (c->head_dim != 64 && c->head_dim != 128) return false;
    if (c->max_len < 1 || c->max_len > (1 << 20)) return false;
    if (!(c->rope_theta > 0.0) || !std::isfinite(c->rope_theta)) return false;
    return true;
}

// Enqueue one kernel through `launch`, bracketed by a timing event pair when enabled.
// `launch` returns the CUDA status and may report how many kernels it enqueued.
template <typename F>
cudaError_t timed(attn_ctx* c, int kind, cudaStream_t st, F&& launch) {
    const bool rec = !c->ev_kind.empty() && c->ev_used < static_cast<int>(c->ev_kind.size());
    if (rec) {
        const cudaError_t e = cudaEventRecord(c->ev[2 * c->ev_used], st);
        if (e != cudaSuccess) return e;
    }
    int n = 1;
    const cudaError_t e = launch(&n);
    if (e != cudaSuccess) return e;
    c->launches[kind] += n;
    if (rec) {
        const cudaError_t e2 = cudaEventRecord(c->ev[2 * c->ev_used + 1], st);
        if (e2 != cudaSuccess) return e2;
        c->ev_kind[c->ev_used++] = kind;
    }
    return cudaSuccess;
}

void free_events(attn_ctx* c) {
    for (cudaEvent_t e : c->ev) cudaEventDestroy(e);
    c->ev.clear();
    c->ev_kind.clear();
    c->ev_used = 0;
}

int encode_map(const attn_ctx* c, CUtensorMap* map, const void* gaddr, cuuint32_t rank, const cuuint64_t* dims,
               const cuuint64_t* strides, const cuuint32_t* box) {
    const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    const CUresult r = c->encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(gaddr), dims, strides,
                                 box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                 CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        std::snprintf(g_cuda_msg, sizeof g_cuda_msg, "cuTensorMapEncodeTiled failed (CUresult %d)", static_cast<int>(r));
        return ATTN_ECUDA;
    }
    return ATTN_OK;
}

// The prefill stages: validate, K1, build the maps over [0, hist+chunk), K2.  q/k/v/out
// hold `chunk` tokens of each sequence, sequence b starting at token b * seq_stride
// (seq_stride = chunk for a dense chunk; the prompt length for a segment of a prompt).
int run_prefill(attn_ctx* c, const uint16_t* q, const uint16_t* k, const uint16_t* v, int hist, int chunk,
                int seq_stride, uint16_t* kc, uint16_t* vc, uint16_t* out, cudaStream_t st) {
    if (c == nullptr || q == nullptr || k == nullptr || v == nullptr || kc == nullptr || vc == nullptr ||
        out == nullptr)
        return ATTN_EINVAL;
    if (chunk < 1 || seq_stride < chunk || hist < 0 || static_cast<long>(hist) + chunk > c->cfg.max_len)
        return ATTN_EINVAL;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(kc) || !aligned16(vc) || !aligned16(out))
        return ATTN_EINVAL;
    const attn::Shape& s = c->shape;
    // flash_fwd's work items (pairs of 128-row query tiles x query heads x sequences) are
    // counted in int: keep them well inside it
    if ((static_cast<long long>(chunk) + 255) / 256 * s.n_q_heads * s.batch > (1LL << 30)) return ATTN_EINVAL;
    const cuuint64_t D = static_cast<cuuint64_t>(s.head_dim);
    attn::FlashMaps maps;
    {
        const cuuint64_t dims[4] = {D, static_cast<cuuint64_t>(s.n_q_heads), static_cast<cuuint64_t>(chunk),
                                    static_cast<cuuint64_t>(s.batch)};
        const cuuint64_t strides[3] = {D * 2, D * 2 * s.n_q_heads,
                                       D * 2 * s.n_q_heads * static_cast<cuuint64_t>(seq_stride)};
        const cuuint32_t box[4] = {64, 1, 128, 1};
        const int rc = encode_map(c, &maps.q, q, 4, dims, strides, box);
        if (rc != ATTN_OK) return rc;
    }
    {
        const cuuint64_t dims[3] = {D, static_cast<cuuint64_t>(hist + chunk),
                                    static_cast<cuuint64_t>(s.batch) * s.n_kv_heads};
        const cuuint64_t strides[2] = {D * 2, D * 2 * static_cast<cuuint64_t>(s.max_len)};
        const cuuint32_t box[3] = {64, 128, 1};
        int rc = encode_map(c, &maps.k, kc, 3, dims, strides, box);
        if (rc == ATTN_OK) rc = encode_map(c, &maps.v, vc, 3, dims, strides, box);
        if (rc != ATTN_OK) return rc;
    }
    cudaError_t e = timed(c, ATTN_KERNEL_ROPE_APPEND, st, [&](int*) {
        return attn::launch_rope_append(s, k, v, hist, nullptr, chunk, seq_stride, c->d_cos, c->d_sin, c->d_cos_t,
                                        c->d_sin_t, kc, vc, c->d_err,
                                        st);
    });
    if (e != cudaSuccess) return cuda_fail(e, "rope_append launch");
    e = timed(c, ATTN_KERNEL_FLASH_FWD, st, [&](int* n) {
        return attn::launch_flash_fwd(s, maps, hist, chunk, seq_stride, c->d_cos_t, c->d_sin_t, out, c->d_flash_o,
                                      c->d_flash_ml, c->d_err, c->num_sms, st, n, c->wait_ns);
    });
    if (e != cudaSuccess) return cuda_fail(e, "flash_fwd launch");
    return ATTN_OK;
}

}  // namespace

extern "C" {

int attn_create(const attn_cfg* cfg, attn_ctx** out) {
    if (out == nullptr) return ATTN_EINVAL;
    *out = nullptr;
    if (!cfg_valid(cfg)) return ATTN_EINVAL;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    cudaDeviceProp prop;
    e = cudaGetDeviceProperties(&prop, dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDeviceProperties");
    if (prop.major != 10 || prop.minor != 3) return ATTN_EARCH;

    attn_ctx* c = new (std::nothrow) attn_ctx();
    if (c == nullptr) return ATTN_ENOMEM;
    c->cfg = *cfg;
    c->shape = attn::Shape{cfg->batch, cfg->n_q_heads, cfg->n_kv_heads, cfg->head_dim, cfg->max_len};
    c->device = dev;
    c->num_sms = prop.multiProcessorCount;
    c->nsplit_max = 256;
    c->wait_ns = attn::kWaitLimitNs;

    cudaDriverEntryPointQueryResult qres;
    void* fn = nullptr;
    e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &qres);
    if (e != cudaSuccess || qres != cudaDriverEntryPointSuccess || fn == nullptr) {
        delete c;
        return cuda_fail(e == cudaSuccess ? cudaErrorNotSupported : e, "cuTensorMapEncodeTiled entry point");
    }
    c->encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    e = attn::configure_flash_fwd();
    if (e == cudaSuccess) e = attn::configure_decode();
    if (e == cudaSuccess) e = attn::configure_decode_tc();
    if (e != cudaSuccess) {
        delete c;
        return cuda_fail(e, "configure kernels");
    }

    // RoPE tables (Section 4.6.2): cos/sin of p * theta^(-2j/D), evaluated in double, stored as float.
    const int half = cfg->head_dim / 2;
    const size_t ntab = static_cast<size_t>(cfg->max_len) * half;
    std::vector<float> hc(ntab), hs(ntab), hct(ntab), hst(ntab);
    for (int p = 0; p < cfg->max_len; ++p) {
        for (int j = 0; j < half; ++j) {
            const double inv_freq = std::pow(cfg->rope_theta, -(2.0 * j) / static_cast<double>(cfg->head_dim));
            const double ang = static_cast<double>(p) * inv_freq;
            hc[static_cast<size_t>(p) * half + j] = static_cast<float>(std::cos(ang));
            hs[static_cast<size_t>(p) * half + j] = static_cast<float>(std::sin(ang));
            const size_t q4 = (static_cast<size_t>(j / 4) * cfg->max_len + p) * 4 + j % 4;
            hct[q4] = hc[static_cast<size_t>(p) * half + j];
            hst[q4] = hs[static_cast<size_t>(p) * half + j];
        }
    }
    const size_t part_rows = static_cast<size_t>(cfg->batch) * cfg->n_q_heads * c->nsplit_max;
    bool oom = false;
    oom |= cudaMalloc(&c->d_cos, ntab * sizeof(float)) != cudaSuccess;
    oom |= cudaMalloc(&c->d_sin, ntab * sizeof(float)) != cudaSuccess;
    oom |= cudaMalloc(&c->d_cos_t, ntab * sizeof(float)) != cudaSuccess;
    oom |= cudaMalloc(&c->d_sin_t, ntab * sizeof(float)) != cudaSuccess;
    oom |= cudaMalloc(&c->d_part_o, part_rows * cfg->head_dim * sizeof(float)) != cudaSuccess;
    oom |= cudaMalloc(&c->d_part_ml, part_rows * 2 * sizeof(float)) != cudaSuccess;
    const size_t piece_rows = static_cast<size_t>(c->num_sms) * 256;
    oom |= cudaMalloc(&c->d_flash_o, piece_rows * cfg->head_dim * sizeof(float)) != cudaSuccess;
    oom |= cudaMalloc(&c->d_flash_ml, piece_rows * 2 * sizeof(float)) != cudaSuccess;
    oom |= cudaMalloc(&c->d_err, sizeof(int)) != cudaSuccess;
    const size_t qd = static_cast<size_t>(cfg->batch) * cfg->n_q_heads * cfg->head_dim;
    const size_t kd = static_cast<size_t>(cfg->batch) * cfg->n_kv_heads * cfg->head_dim;
    oom |= cudaMalloc(&c->d_lq, qd * sizeof(uint16_t)) != cudaSuccess;
    oom |= cudaMalloc(&c->d_lk, kd * sizeof(uint16_t)) != cudaSuccess;
    oom |= cudaMalloc(&c->d_lv, kd * sizeof(uint16_t)) != cudaSuccess;
    oom |= cudaMalloc(&c->d_lo, qd * sizeof(uint16_t)) != cudaSuccess;
    // merge counts and tile claims per (sequence, kv head, column group of the multi-token decode)
    const size_t n_counters = static_cast<size_t>(
        attn::decode_tc_counter_ints(static_cast<long long>(cfg->batch) * cfg->n_kv_heads * kMaxColumnGroups));
    oom |= cudaMalloc(&c->d_counters, n_counters * sizeof(int)) != cudaSuccess;
    if (oom) {
        cudaGetLastError();
        attn_destroy(c);
        return ATTN_ENOMEM;
    }
    e = cudaMemcpy(c->d_cos, hc.data(), ntab * sizeof(float), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(c->d_sin, hs.data(), ntab * sizeof(float), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(c->d_cos_t, hct.data(), ntab * sizeof(float), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(c->d_sin_t, hst.data(), ntab * sizeof(float), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemset(c->d_err, 0, sizeof(int));
    if (e == cudaSuccess) e = cudaMemset(c->d_counters, 0, n_counters * sizeof(int));
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        attn_destroy(c);
        return cuda_fail(e, "attn_create upload");
    }
    *out = c;
    return ATTN_OK;
}

void attn_destroy(attn_ctx* c) {
    if (c == nullptr) return;
    cudaDeviceSynchronize();
    free_events(c);
    cudaFree(c->d_cos);
    cudaFree(c->d_sin);
    cudaFree(c->d_cos_t);
    cudaFree(c->d_sin_t);
    cudaFree(c->d_part_o);
    cudaFree(c->d_part_ml);
    cudaFree(c->d_flash_o);
    cudaFree(c->d_flash_ml);
    cudaFree(c->d_err);
    cudaFree(c->d_counters);
    cudaFree(c->d_lq);
    cudaFree(c->d_lk);
    cudaFree(c->d_lv);
    cudaFree(c->d_lo);
    delete c;
}

int attn_prefill(attn_ctx* c, const uint16_t* q, const uint16_t* k, const uint16_t* v, int chunk_len,
                 uint16_t* k_cache, uint16_t* v_cache, uint16_t* out, attn_stream_t stream) {
    return run_prefill(c, q, k, v, 0, chunk_len, chunk_len, k_cache, v_cache, out,
                       reinterpret_cast<cudaStream_t>(stream));
}

int attn_prefill_kv(attn_ctx* c, const uint16_t* q, const uint16_t* k, const uint16_t* v, int hist_len,
                    int chunk_len, uint16_t* k_cache, uint16_t* v_cache, uint16_t* out, attn_stream_t stream) {
    return run_prefill(c, q, k, v, hist_len, chunk_len, chunk_len, k_cache, v_cache, out,
                       reinterpret_cast<cudaStream_t>(stream));
}

}  // extern "C"

namespace {

// One decode step of ntok new tokens per sequence at positions d_hist_len[b] + hist_add + i.
// after_decode: the previous launch on `st` was this context's decode of the same caches
// (a decode loop).
// producer_early: the previous launch wrote q, k and v and nothing the decode streams (the
// fused QKV GEMV of attn_decode_layer); the head_dim 128 decode then starts its K/V stream as
// a dependent launch before that kernel has finished.
int run_decode(attn_ctx* c, const uint16_t* q, const uint16_t* k, const uint16_t* v, const int32_t* d_hist_len,
               int hist_add, bool after_decode, uint16_t* k_cache, uint16_t* v_cache, uint16_t* out, cudaStream_t st,
               int ntok = 1, bool producer_early = false) {
    if (c == nullptr || q == nullptr || k == nullptr || v == nullptr || d_hist_len == nullptr ||
        k_cache == nullptr || v_cache == nullptr || out == nullptr)
        return ATTN_EINVAL;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(k_cache) || !aligned16(v_cache) ||
        !aligned16(out) || (reinterpret_cast<uintptr_t>(d_hist_len) & 3u))
        return ATTN_EINVAL;
    const bool tc = c->cfg.head_dim == 128;  // tensor-core decode; head_dim 64 on the CUDA cores
    if (k_cache != c->dec_k || v_cache != c->dec_v) {
        const cudaError_t me = tc ? attn::make_decode_tc_maps(c->encode, c->shape, k_cache, v_cache, &c->dec_maps)
                                  : attn::make_decode_maps(c->encode, c->shape, k_cache, v_cache, &c->dec_maps);
        if (me != cudaSuccess) {
            c->dec_k = c->dec_v = nullptr;
            std::snprintf(g_cuda_msg, sizeof g_cuda_msg, "cuTensorMapEncodeTiled failed for the decode caches");
            return ATTN_ECUDA;
        }
        c->dec_k = k_cache;
        c->dec_v = v_cache;
    }
    if (ntok < 1 || ntok > kMaxDraftTokens || (ntok > 1 && !tc)) return ATTN_EINVAL;
    // the partials hold batch * Hq * nsplit_max rows: ntok tokens share them
    const int ncg = attn::decode_tc_column_groups(c->cfg.n_q_heads / c->cfg.n_kv_heads, ntok);
    // grid y and z (kv heads; sequences x column groups, or kv heads x head passes) stay
    // within the 65535 limit of those grid dimensions
    const int G = c->cfg.n_q_heads / c->cfg.n_kv_heads;
    if (tc ? static_cast<long>(c->cfg.batch) * ncg > 65535 : static_cast<long>(c->cfg.n_kv_heads) * ((G + 7) / 8) > 65535)
        return ATTN_EINVAL;
    const int nsplit = tc ? std::min(attn::decode_tc_num_splits(c->shape, c->num_sms, ncg, ntok), c->nsplit_max / ntok)
                          : attn::decode_num_splits(c->shape, c->num_sms, c->nsplit_max);
    cudaError_t e = timed(c, ATTN_KERNEL_DECODE_SPLIT, st, [&](int*) {
        if (tc)
            return attn::launch_decode_tc(c->shape, c->dec_maps, q, k, v, d_hist_len, hist_add, k_cache, v_cache, c->d_cos,
                                          c->d_sin, c->d_part_o, c->d_part_ml, c->d_counters, nsplit, out,
                                          c->d_err, after_decode, ntok, st, producer_early, c->wait_ns, c->num_sms);
        return attn::launch_decode_split(c->shape, c->dec_maps, q, k, v, d_hist_len, hist_add, k_cache, v_cache, c->d_cos,
                                         c->d_sin, c->d_part_o, c->d_part_ml, nsplit, c->d_err, st, c->wait_ns);
    });
    if (e != cudaSuccess) return cuda_fail(e, "decode_split launch");
    if (tc) return ATTN_OK;  // the tensor-core decode merges its splits itself
    e = timed(c, ATTN_KERNEL_DECODE_COMBINE, st, [&](int*) {
        return attn::launch_decode_combine(c->shape, d_hist_len, hist_add, c->d_part_o, c->d_part_ml, nsplit, out, st);
    });
    if (e != cudaSuccess) return cuda_fail(e, "decode_combine launch");
    return ATTN_OK;
}

}  // namespace

extern "C" {

int attn_decode(attn_ctx* c, const uint16_t* q, const uint16_t* k, const uint16_t* v, const int32_t* d_hist_len,
                uint16_t* k_cache, uint16_t* v_cache, uint16_t* out, attn_stream_t stream) {
    return run_decode(c, q, k, v, d_hist_len, 0, false, k_cache, v_cache, out, reinterpret_cast<cudaStream_t>(stream));
}

int attn_decode_multi(attn_ctx* c, const uint16_t* q, const uint16_t* k, const uint16_t* v,
                      const int32_t* d_hist_len, int n_new, uint16_t* k_cache, uint16_t* v_cache, uint16_t* out,
                      attn_stream_t stream) {
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (c == nullptr || c->cfg.head_dim == 128 || n_new == 1)
        return run_decode(c, q, k, v, d_hist_len, 0, false, k_cache, v_cache, out, st, n_new);
    // head_dim 64: the n_new tokens as n_new decode steps in order (token t at hist_len[b] + t
    // sees the tokens before it in the cache, which is the same computation); each step's
    // rows are gathered into the context's decode-block buffers and its output scattered back.
    if (q == nullptr || k == nullptr || v == nullptr || out == nullptr || n_new < 1 || n_new > c->cfg.max_len)
        return ATTN_EINVAL;
    const size_t D = static_cast<size_t>(c->cfg.head_dim), B = static_cast<size_t>(c->cfg.batch);
    const size_t qrow = c->cfg.n_q_heads * D * 2, krow = c->cfg.n_kv_heads * D * 2;  // bytes of one token's rows
    for (int t = 0; t < n_new; ++t) {
        cudaError_t e = cudaMemcpy2DAsync(c->d_lq, qrow, reinterpret_cast<const uint8_t*>(q) + t * qrow, n_new * qrow,
                                          qrow, B, cudaMemcpyDeviceToDevice, st);
        if (e == cudaSuccess)
            e = cudaMemcpy2DAsync(c->d_lk, krow, reinterpret_cast<const uint8_t*>(k) + t * krow, n_new * krow, krow, B,
                                  cudaMemcpyDeviceToDevice, st);
        if (e == cudaSuccess)
            e = cudaMemcpy2DAsync(c->d_lv, krow, reinterpret_cast<const uint8_t*>(v) + t * krow, n_new * krow, krow, B,
                                  cudaMemcpyDeviceToDevice, st);
        if (e != cudaSuccess) return cuda_fail(e, "decode_multi gather");
        const int rc = run_decode(c, c->d_lq, c->d_lk, c->d_lv, d_hist_len, t, false, k_cache, v_cache, c->d_lo, st);
        if (rc != ATTN_OK) return rc;
        e = cudaMemcpy2DAsync(reinterpret_cast<uint8_t*>(out) + t * qrow, n_new * qrow, c->d_lo, qrow, qrow, B,
                              cudaMemcpyDeviceToDevice, st);
        if (e != cudaSuccess) return cuda_fail(e, "decode_multi scatter");
    }
    return ATTN_OK;
}

int attn_prompt(attn_ctx* c, const uint16_t* q, const uint16_t* k, const uint16_t* v, int hist_len, int prompt_len,
                int seg_len, uint16_t* k_cache, uint16_t* v_cache, uint16_t* out, attn_stream_t stream) {
    // Section 4.1, third scenario: a prompt longer than the stages' static chunk runs as
    // one prefill (no history) or prefill_kv, then prefill_kv for every further segment,
    // each over everything before it.  Checked whole before the first launch.
    if (c == nullptr || q == nullptr || k == nullptr || v == nullptr || k_cache == nullptr || v_cache == nullptr ||
        out == nullptr)
        return ATTN_EINVAL;
    if (prompt_len < 1 || seg_len < 1 || hist_len < 0 || static_cast<long>(hist_len) + prompt_len > c->cfg.max_len)
        return ATTN_EINVAL;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(k_cache) || !aligned16(v_cache) ||
        !aligned16(out))
        return ATTN_EINVAL;
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const size_t q_tok = static_cast<size_t>(c->cfg.n_q_heads) * c->cfg.head_dim;   // elements per token
    const size_t kv_tok = static_cast<size_t>(c->cfg.n_kv_heads) * c->cfg.head_dim;
    for (int s0 = 0; s0 < prompt_len; s0 += seg_len) {
        const int n = std::min(seg_len, prompt_len - s0);
        const int rc = run_prefill(c, q + s0 * q_tok, k + s0 * kv_tok, v + s0 * kv_tok, hist_len + s0, n, prompt_len,
                                   k_cache, v_cache, out + s0 * q_tok, st);
        if (rc != ATTN_OK) return rc;
    }
    return ATTN_OK;
}

int attn_decode_steps(attn_ctx* c, const uint16_t* q, const uint16_t* k, const uint16_t* v, const int32_t* d_hist_len,
                      int n_steps, uint16_t* k_cache, uint16_t* v_cache, uint16_t* out, attn_stream_t stream) {
    // Section 4.5, steps 3-5 restricted to attention: n_steps decode steps back to back,
    // step t at positions d_hist_len[b] + t (the lengths array is read, never written).
    if (c == nullptr || q == nullptr || k == nullptr || v == nullptr || d_hist_len == nullptr ||
        k_cache == nullptr || v_cache == nullptr || out == nullptr || n_steps < 1 || n_steps > c->cfg.max_len)
        return ATTN_EINVAL;
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const size_t q_step = static_cast<size_t>(c->cfg.batch) * c->cfg.n_q_heads * c->cfg.head_dim;
    const size_t kv_step = static_cast<size_t>(c->cfg.batch) * c->cfg.n_kv_heads * c->cfg.head_dim;
    for (int t = 0; t < n_steps; ++t) {
        const int rc = run_decode(c, q + t * q_step, k + t * kv_step, v + t * kv_step, d_hist_len, t, t > 0, k_cache,
                                  v_cache, out + t * q_step, st);
        if (rc != ATTN_OK) return rc;
    }
    return ATTN_OK;
}

int attn_set_wait_limit(attn_ctx* c, long long limit_ns) {
    if (c == nullptr) return ATTN_EINVAL;
    c->wait_ns = limit_ns > 0 ? static_cast<uint64_t>(limit_ns) : attn::kWaitLimitNs;
    return ATTN_OK;
}

int attn_device_error(attn_ctx* c, attn_stream_t stream, int* flags) {
    if (c == nullptr) return ATTN_EINVAL;
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int h = 0;
    cudaError_t e = cudaMemcpyAsync(&h, c->d_err, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e == cudaSuccess && h != 0) e = cudaMemsetAsync(c->d_err, 0, sizeof(int), st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "attn_device_error");
    if (flags != nullptr) *flags = h;
    return h ? ATTN_EDEVICE : ATTN_OK;
}

int attn_timing_enable(attn_ctx* c, int max_launches) {
    if (c == nullptr || max_launches < 0 || max_launches > (1 << 20)) return ATTN_EINVAL;
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(e, "attn_timing_enable");
    free_events(c);
    if (max_launches == 0) return ATTN_OK;
    c->ev.resize(2 * static_cast<size_t>(max_launches), nullptr);
    c->ev_kind.assign(static_cast<size_t>(max_launches), -1);
    for (cudaEvent_t& ev : c->ev) {
        e = cudaEventCreate(&ev);
        if (e != cudaSuccess) {
            ev = nullptr;
            free_events(c);
            return cuda_fail(e, "cudaEventCreate");
        }
    }
    return ATTN_OK;
}

int attn_timing_read(attn_ctx* c, double* ms, long long* launches) {
    if (c == nullptr) return ATTN_EINVAL;
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(e, "attn_timing_read");
    double acc[ATTN_NUM_KERNELS] = {0.0, 0.0, 0.0, 0.0};
    for (int i = 0; i < c->ev_used; ++i) {
        float t = 0.f;
        e = cudaEventElapsedTime(&t, c->ev[2 * i], c->ev[2 * i + 1]);
        if (e != cudaSuccess) return cuda_fail(e, "cudaEventElapsedTime");
        acc[c->ev_kind[i]] += t;
    }
    for (int k = 0; k < ATTN_NUM_KERNELS; ++k) {
        if (ms != nullptr) ms[k] = acc[k];
        if (launches != nullptr) launches[k] = c->launches[k];
        c->launches[k] = 0;
    }
    c->ev_used = 0;
    return ATTN_OK;
}

int attn_w4bf16_rows_per_launch(int K) { return K >= 128 && K % 128 == 0 ? attn::w4_gemv_max_rows(K) : 0; }

int attn_w4bf16_gemv_fused(const void* w_tiles, const uint16_t* x, int M, int N, int K, const uint16_t* rms_gamma,
                           float rms_eps, const uint16_t* residual, uint16_t* y, int n_split0, uint16_t* y1,
                           int n_split1, uint16_t* y2, int32_t* d_err, int flags, attn_stream_t stream) {
    if (w_tiles == nullptr || x == nullptr || y == nullptr) return ATTN_EINVAL;
    if (flags & ~ATTN_W4_WEIGHTS_STATIC) return ATTN_EINVAL;
    if (M < 1 || N < 1 || K < 128 || K % 128 != 0) return ATTN_EINVAL;
    const int rows = attn::w4_gemv_max_rows(K);
    if (rows < 1) return ATTN_EINVAL;
    if ((reinterpret_cast<uintptr_t>(w_tiles) & 15u) || (reinterpret_cast<uintptr_t>(x) & 15u) ||
        (reinterpret_cast<uintptr_t>(y) & 1u) || (reinterpret_cast<uintptr_t>(d_err) & 3u) ||
        (reinterpret_cast<uintptr_t>(rms_gamma) & 7u) || (reinterpret_cast<uintptr_t>(residual) & 1u) ||
        (reinterpret_cast<uintptr_t>(y1) & 1u) || (reinterpret_cast<uintptr_t>(y2) & 1u))
        return ATTN_EINVAL;
    if (rms_gamma != nullptr && !(rms_eps >= 0.f && rms_eps < 1.f)) return ATTN_EINVAL;
    attn::W4Fused fz{rms_gamma, rms_eps, residual, N, N, nullptr, nullptr};
    if (y1 != nullptr || y2 != nullptr) {
        if (y1 == nullptr || y2 == nullptr || !(0 < n_split0 && n_split0 < n_split1 && n_split1 < N))
            return ATTN_EINVAL;
        fz.n0 = n_split0;
        fz.n1 = n_split1;
        fz.y1 = y1;
        fz.y2 = y2;
    }
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "attn_w4bf16_gemv device query");
    if (dev < 0 || dev >= kArchCacheDevices) return ATTN_EINVAL;
    int arch = g_arch_ok[dev].load(std::memory_order_relaxed);  // 0 unknown, 1 sm_103, 2 other
    if (arch == 0) {
        int major = 0, minor = 0;
        e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
        if (e != cudaSuccess) return cuda_fail(e, "attn_w4bf16_gemv device query");
        arch = major == 10 && minor == 3 ? 1 : 2;
        g_arch_ok[dev].store(arch, std::memory_order_relaxed);
    }
    if (arch != 1) return ATTN_EARCH;
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    // Rows of x past what one launch stages take further passes over the weights.
    for (int m0 = 0; m0 < M; m0 += rows) {
        const int mc = std::min(rows, M - m0);
        attn::W4Fused f = fz;
        const size_t r0 = static_cast<size_t>(m0);
        if (f.residual != nullptr) f.residual += r0 * N;
        if (f.y1 != nullptr) {
            f.y1 += r0 * (f.n1 - f.n0);
            f.y2 += r0 * (N - f.n1);
        }
        e = attn::launch_w4_gemv(static_cast<const uint8_t*>(w_tiles), x + r0 * K, mc, N, K, y + r0 * fz.n0, d_err,
                                 (flags & ATTN_W4_WEIGHTS_STATIC) != 0, f, st);
        if (e != cudaSuccess) return cuda_fail(e, "w4_gemv");
    }
    return ATTN_OK;
}

namespace {
// Workspace of attn_prefill_layer: xn [T][hidden], q [T][qd], k and v [T][kd], the attention
// output [T][qd] (T = batch * chunk_len), each region starting at a 256-byte boundary.
struct PrefillWs {
    size_t xn, q, k, v, o, bytes;
};
PrefillWs prefill_ws(const attn_cfg& cfg, int hidden, int chunk_len) {
    const size_t T = static_cast<size_t>(cfg.batch) * chunk_len;
    const size_t qd = static_cast<size_t>(cfg.n_q_heads) * cfg.head_dim, kd = static_cast<size_t>(cfg.n_kv_heads) * cfg.head_dim;
    auto up = [](size_t b) { return (b + 255) & ~static_cast<size_t>(255); };
    PrefillWs w;
    w.xn = 0;
    w.q = w.xn + up(T * hidden * 2);
    w.k = w.q + up(T * qd * 2);
    w.v = w.k + up(T * kd * 2);
    w.o = w.v + up(T * kd * 2);
    w.bytes = w.o + up(T * qd * 2);
    return w;
}
}  // namespace

size_t attn_prefill_layer_workspace(const attn_ctx* c, int hidden, int chunk_len) {
    if (c == nullptr || hidden < 1 || chunk_len < 1) return 0;
    return prefill_ws(c->cfg, hidden, chunk_len).bytes;
}

int attn_prefill_layer(attn_ctx* c, const uint16_t* x, const uint16_t* rms_gamma, float rms_eps,
                       const void* wqkv_tiles, const void* wo_tiles, int hidden, int hist_len, int chunk_len,
                       uint16_t* k_cache, uint16_t* v_cache, uint16_t* h_out, void* workspace, size_t workspace_bytes,
                       attn_stream_t stream) {
    if (c == nullptr || x == nullptr || rms_gamma == nullptr || wqkv_tiles == nullptr || wo_tiles == nullptr ||
        k_cache == nullptr || v_cache == nullptr || h_out == nullptr || workspace == nullptr)
        return ATTN_EINVAL;
    const int qd = c->cfg.n_q_heads * c->cfg.head_dim, kd = c->cfg.n_kv_heads * c->cfg.head_dim;
    if (hidden < 128 || hidden % 128 != 0 || qd % 128 != 0 || (qd + 2 * kd) % 128 != 0) return ATTN_EINVAL;
    if (chunk_len < 1 || hist_len < 0 || static_cast<long>(hist_len) + chunk_len > c->cfg.max_len) return ATTN_EINVAL;
    const long long T = static_cast<long long>(c->cfg.batch) * chunk_len;
    if (T > 65535LL * 128 || !std::isfinite(rms_eps) || rms_eps < 0.f) return ATTN_EINVAL;
    if (!aligned16(x) || !aligned16(rms_gamma) || !aligned16(wqkv_tiles) || !aligned16(wo_tiles) ||
        !aligned16(h_out) || (reinterpret_cast<uintptr_t>(workspace) & 255u))
        return ATTN_EINVAL;
    const PrefillWs ws = prefill_ws(c->cfg, hidden, chunk_len);
    if (workspace_bytes < ws.bytes) return ATTN_EINVAL;
    uint8_t* wb = static_cast<uint8_t*>(workspace);
    uint16_t* xn = reinterpret_cast<uint16_t*>(wb + ws.xn);
    uint16_t* q = reinterpret_cast<uint16_t*>(wb + ws.q);
    uint16_t* k = reinterpret_cast<uint16_t*>(wb + ws.k);
    uint16_t* v = reinterpret_cast<uint16_t*>(wb + ws.v);
    uint16_t* o = reinterpret_cast<uint16_t*>(wb + ws.o);
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    // input_layernorm: one factor per token, a pre-pass over the chunk
    cudaError_t e = attn::launch_rmsnorm_rows(x, rms_gamma, rms_eps, static_cast<int>(T), hidden, xn, st);
    if (e != cudaSuccess) return cuda_fail(e, "prefill layer RMSNorm");
    // q/k/v projections: one GEMM over the stacked rows, the output split three ways
    attn::W4GemmEpi split = {qd, qd + kd, k, v, nullptr};
    e = attn::launch_w4_gemm(static_cast<const uint8_t*>(wqkv_tiles), xn, static_cast<int>(T), qd + 2 * kd, hidden, q,
                             c->d_err, st, &split);
    if (e != cudaSuccess) return cuda_fail(e, "prefill layer QKV GEMM");
    // RoPE of q and k, cache append, causal attention over the history (the prefill stages)
    const int rc = run_prefill(c, q, k, v, hist_len, chunk_len, chunk_len, k_cache, v_cache, o, st);
    if (rc != ATTN_OK) return rc;
    // o_proj with the residual in the epilogue (h may be x)
    attn::W4GemmEpi res = {hidden, hidden, nullptr, nullptr, x};
    e = attn::launch_w4_gemm(static_cast<const uint8_t*>(wo_tiles), o, static_cast<int>(T), hidden, qd, h_out, c->d_err,
                             st, &res);
    return e == cudaSuccess ? ATTN_OK : cuda_fail(e, "prefill layer o_proj GEMM");
}

int attn_decode_layer(attn_ctx* c, const uint16_t* x, const uint16_t* rms_gamma, float rms_eps,
                      const void* wqkv_tiles, const void* wo_tiles, int hidden, const int32_t* d_hist_len,
                      uint16_t* k_cache, uint16_t* v_cache, uint16_t* h_out, int flags, attn_stream_t stream) {
    if (c == nullptr || x == nullptr || rms_gamma == nullptr || wqkv_tiles == nullptr || wo_tiles == nullptr ||
        h_out == nullptr)
        return ATTN_EINVAL;
    const int B = c->cfg.batch;
    const int qd = c->cfg.n_q_heads * c->cfg.head_dim, kd = c->cfg.n_kv_heads * c->cfg.head_dim;
    if (hidden < 128 || hidden % 128 != 0 || qd % 128 != 0) return ATTN_EINVAL;
    // input_layernorm + q/k/v projections (one GEMV over the stacked rows, split three ways)
    int rc = attn_w4bf16_gemv_fused(wqkv_tiles, x, B, qd + 2 * kd, hidden, rms_gamma, rms_eps, nullptr, c->d_lq, qd,
                                    c->d_lk, qd + kd, c->d_lv, c->d_err, flags, stream);
    if (rc != ATTN_OK) return rc;
    // RoPE of q and k, cache append, attention over the history (the decode stage)
    rc = run_decode(c, c->d_lq, c->d_lk, c->d_lv, d_hist_len, 0, false, k_cache, v_cache, c->d_lo,
                    reinterpret_cast<cudaStream_t>(stream), 1, true);
    if (rc != ATTN_OK) return rc;
    // o_proj + residual; the decode kernels never write the weights, so they may stream early
    return attn_w4bf16_gemv_fused(wo_tiles, c->d_lo, B, hidden, qd, nullptr, 0.f, x, h_out, 0, nullptr, 0, nullptr,
                                  c->d_err, ATTN_W4_WEIGHTS_STATIC, stream);
}

int attn_w4bf16_gemm(const void* w_tiles, const uint16_t* x, int T, int N, int K, uint16_t* y, int32_t* d_err,
                     attn_stream_t stream) {
    if (w_tiles == nullptr || x == nullptr || y == nullptr) return ATTN_EINVAL;
    if (T < 1 || T > 65535 * 128 || N < 128 || N % 128 != 0 || K < 128 || K % 128 != 0) return ATTN_EINVAL;
    if ((reinterpret_cast<uintptr_t>(w_tiles) & 15u) || (reinterpret_cast<uintptr_t>(x) & 15u) ||
        (reinterpret_cast<uintptr_t>(y) & 15u) || (reinterpret_cast<uintptr_t>(d_err) & 3u))
        return ATTN_EINVAL;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "attn_w4bf16_gemm device query");
    if (dev < 0 || dev >= kArchCacheDevices) return ATTN_EINVAL;
    int arch = g_arch_ok[dev].load(std::memory_order_relaxed);  // 0 unknown, 1 sm_103, 2 other
    if (arch == 0) {
        int major = 0, minor = 0;
        e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
        if (e != cudaSuccess) return cuda_fail(e, "attn_w4bf16_gemm device query");
        arch = major == 10 && minor == 3 ? 1 : 2;
        g_arch_ok[dev].store(arch, std::memory_order_relaxed);
    }
    if (arch != 1) return ATTN_EARCH;
    e = attn::launch_w4_gemm(static_cast<const uint8_t*>(w_tiles), x, T, N, K, y, d_err,
                             reinterpret_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ATTN_OK : cuda_fail(e, "w4_gemm");
}

int attn_w4bf16_gemv(const void* w_tiles, const uint16_t* x, int M, int N, int K, uint16_t* y, int32_t* d_err,
                     int flags, attn_stream_t stream) {
    return attn_w4bf16_gemv_fused(w_tiles, x, M, N, K, nullptr, 0.f, nullptr, y, 0, nullptr, 0, nullptr, d_err, flags,
                                  stream);
}

const char* attn_strerror(int code) {
    switch (code) {
        case ATTN_OK: return "success";
        case ATTN_EINVAL: return "invalid argument or unsupported shape";
        case ATTN_EARCH: return "the current CUDA device is not sm_103 (GB300)";
        case ATTN_ECUDA: return "CUDA runtime or launch error";
        case ATTN_ENOMEM: return "device memory allocation failed";
        case ATTN_EDEVICE: return "a kernel reported an error in the device error word";
        default: return "unknown error code";
    }
}

const char* attn_last_cuda_error_string(void) { return g_cuda_msg; }

}  // extern "C"

// internal.h -- launchers shared between the translation units of the library.
// Not part of the public ABI (include/attn.h).
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

namespace attn {

// Error-word bits (mirrors ATTN_DEVERR_* of attn.h).
constexpr int kDevErrHistRange = 1;
constexpr int kDevErrTimeout = 2;
// The thread's last failure text, read by attn_last_cuda_error_string (attn_api.cu).
// record_cuda_error formats a CUDA error with the failing step and returns ATTN_ECUDA
// (-3); record_error_text stores a plain text.
int record_cuda_error(cudaError_t e, const char* where);
void record_error_text(const char* text);

// Default limit of every bounded wait of the kernels (1 s).  The launchers of flash_fwd,
// decode_split and decode_tc take a limit for the waits of their main loops; the waits
// that let copies and MMAs already issued finish (before a CTA that gave up exits) always
// keep this default.
constexpr uint64_t kWaitLimitNs = 1000000000ull;

struct Shape {
    int batch, n_q_heads, n_kv_heads, head_dim, max_len;
};

// Division by a divisor fixed at launch time (Granlund and Montgomery, "Division by
// invariant integers using multiplication", 1994): with s = ceil(log2 d) and
// m = floor(2^32 (2^s - d) / d) + 1, n / d = (umulhi(n, m) + n) >> s for 0 <= n < 2^31
// and 1 <= d < 2^31.  The host builds it; kernels divide with fdiv() in a few
// instructions instead of the dozens of a generic integer division.
struct FastDiv {
    uint32_t d, m, s;
};
inline FastDiv make_fastdiv(int div) {
    FastDiv f;
    f.d = static_cast<uint32_t>(div);
    f.s = 0;
    while ((1ull << f.s) < f.d) ++f.s;
    f.m = static_cast<uint32_t>(((1ull << 32) * ((1ull << f.s) - f.d)) / f.d + 1);
    return f;
}
#ifdef __CUDACC__
__device__ __forceinline__ int fdiv(int n, const FastDiv& f) {
    return static_cast<int>((__umulhi(static_cast<uint32_t>(n), f.m) + static_cast<uint32_t>(n)) >> f.s);
}
#endif

// K1: RoPE of the new k (table gather, Section 4.6.2) and the in-place append of
// k and v into cache slots hist+i (Listing 2 "Concat"; Section 4.6.3).
// hist comes from `d_hist[b]` when non-null (decode), else `hist` for every b.  k and v
// hold `chunk` tokens of each sequence, sequence b starting at token b * seq_stride.
// cos_t / sin_t (the table copies in groups of four pairs, [D/8][max_len][4], or null):
// their lines for the chunk's positions are prefetched into L2 for K2's rotation of q.
cudaError_t launch_rope_append(const Shape& s, const uint16_t* k, const uint16_t* v, int hist,
                               const int32_t* d_hist, int chunk, int seq_stride, const float* cos_tab,
                               const float* sin_tab, const float* cos_t, const float* sin_t, uint16_t* k_cache,
                               uint16_t* v_cache, int* err, cudaStream_t st);

// K2: causal flash attention of `chunk` new queries at positions hist.. over cache
// slots [0, hist+chunk) (prefill: hist=0).  RoPE of q is applied in the kernel.
struct FlashMaps {
    CUtensorMap q;  // q [B, S, Hq, D] as 4-D {D, Hq, S, B}; box {64, 1, 128, 1}
    CUtensorMap k;  // k_cache as 3-D {D, hist+chunk, B*Hkv}; box {64, 128, 1}
    CUtensorMap v;  // v_cache, same as k
};
// Raise the dynamic shared-memory limit of K2 on the current device (once per device).
cudaError_t configure_flash_fwd();
// Work is split across num_sms persistent CTAs; items of the last, partial round are
// cut into KV pieces whose partials go to ws_o [num_sms*256, D] / ws_ml [num_sms*256, 2]
// and are merged by a second kernel (then *n_launched = 2).
// cos_t / sin_t: the RoPE tables in groups of four pairs, [D/8][max_len][4] (entry (j, p) at
// ((j / 4) * max_len + p) * 4 + j % 4).
// out holds `chunk` tokens of each sequence, sequence b starting at token b * s_stride (the
// q map carries the same stride).
cudaError_t launch_flash_fwd(const Shape& s, const FlashMaps& maps, int hist, int chunk, int s_stride,
                             const float* cos_t, const float* sin_t, uint16_t* out, float* ws_o, float* ws_ml, int* err,
                             int num_sms, cudaStream_t st, int* n_launched, uint64_t wait_ns = kWaitLimitNs);

// K3 + K4: decode.  The maps cover the whole caches as 3-D {D, max_len, B*Hkv}
// with 64-key boxes (built once per cache pair).  K3 also rotates the new key and
// appends k and v at slot hist[b]; K4 merges the splits (programmatic dependent launch).
using PFN_encodeTiled = PFN_cuTensorMapEncodeTiled_v12000;
struct DecodeMaps {
    CUtensorMap k;
    CUtensorMap v;
};
cudaError_t configure_decode();  // dynamic shared-memory limits of K3 (once per device)
int decode_num_splits(const Shape& s, int num_sms, int max_splits);
cudaError_t make_decode_maps(PFN_encodeTiled encode, const Shape& s, const uint16_t* k_cache,
                             const uint16_t* v_cache, DecodeMaps* maps);
// Decode lengths: sequence b's new token takes position d_hist[b] + hist_add (hist_add >= 0
// lets a run of decode steps share one length array); see decode_hist().
cudaError_t launch_decode_split(const Shape& s, const DecodeMaps& maps, const uint16_t* q, const uint16_t* k_new,
                                const uint16_t* v_new, const int32_t* d_hist, int hist_add, uint16_t* k_cache,
                                uint16_t* v_cache,
                                const float* cos_tab, const float* sin_tab, float* part_o, float* part_ml,
                                int nsplit, int* err, cudaStream_t st, uint64_t wait_ns = kWaitLimitNs);
// K3 for head_dim 128 on the tensor cores (decode_tc.cu): maps with 128-key boxes; same
// partial layout as launch_decode_split, but the merge is fused in (the split that
// completes an item's tiles merges and writes `out`), so no K4 follows.  Splits claim key
// tiles from a per-item counter (item: sequence, kv head, column group).  `counters`:
// decode_tc_counter_ints(items) ints, zero before the first launch; every launch leaves
// them zero.  num_sms: whether the grid fits one wave.  1 <= ntok <= 16 new tokens per
// sequence (q/k/v/out
// [B, ntok, H, D]) at positions d_hist[b] + hist_add + i, token i attending causally to
// slots [0, that position]; the partials need B * ntok * Hq * nsplit rows.
// after_decode: the stream's previous kernel is a decode_tc launch (the
// previous step of a decode loop); this one then starts as a dependent launch whose
// setup overlaps that step's tail.  Never set it after any other kernel: the inputs
// are read before the grid waits on its predecessor.
// producer_early: a dependent launch after a kernel that writes q / the new k, v (and
// neither the caches, the lengths nor the counters); the K/V stream starts before the wait.
cudaError_t configure_decode_tc();
// Column groups of 16 (query head, new token) columns one launch runs for ntok new tokens
// per sequence: ceil(G * ntok / 16); items = B * Hkv * that many.
int decode_tc_column_groups(int G, int ntok);
// Ints of the counter array for `items` items: claims, slots and visits, then 64-bit
// (contributors, tiles done) words from an even offset.
inline long long decode_tc_counter_ints(long long items) { return 3 * items + 1 + 2 * items; }
// Splits per item for a decode of ntok new tokens with ncg column groups (after the
// configuration, which measures the cluster sizes that fit).
int decode_tc_num_splits(const Shape& s, int num_sms, int ncg = 1, int ntok = 1);
cudaError_t make_decode_tc_maps(PFN_encodeTiled encode, const Shape& s, const uint16_t* k_cache,
                                const uint16_t* v_cache, DecodeMaps* maps);
cudaError_t launch_decode_tc(const Shape& s, const DecodeMaps& maps, const uint16_t* q, const uint16_t* k_new,
                             const uint16_t* v_new, const int32_t* d_hist, int hist_add, uint16_t* k_cache,
                             uint16_t* v_cache,
                             const float* cos_tab, const float* sin_tab, float* part_o, float* part_ml,
                             int* counters, int nsplit, uint16_t* out, int* err, bool after_decode, int ntok,
                             cudaStream_t st, bool producer_early, uint64_t wait_ns, int num_sms);
cudaError_t launch_decode_combine(const Shape& s, const int32_t* d_hist, int hist_add, const float* part_o,
                                  const float* part_ml, int nsplit, uint16_t* out, cudaStream_t st);

// W4BF16 GEMV (w4_gemv.cu): y[m, n] = sum_k x[m, k] (q[n, k] - z[n, k/128]) s[n, k/128] for
// the 1 <= M <= w4_gemv_max_rows(K) activation rows of one launch.  tiles: the tile
// stream of attn_w4bf16_gemv (16-byte aligned); x: bf16 [M][K] (16-byte aligned);
// y: bf16 [M][N].  K a multiple of 128.  A launch stages x and its group sums in the
// shared memory its rings leave free.  A bounded wait that runs out sets
// kDevErrTimeout in *err (when err is not null).
int w4_gemv_max_rows(int K);  // 8, 4, 2, 1 or 0 (K too large)
// Fused parts of a GEMV (all optional): RMSNorm of x before the product (gamma: bf16 [K],
// 8-byte aligned), a residual added before rounding (bf16 [M][N]), and the output columns
// split three ways: [0, n0) -> y (row stride n0), [n0, n1) -> y1, [n1, N) -> y2 (no split:
// n0 = n1 = N).
struct W4Fused {
    const uint16_t* gamma;
    float eps;
    const uint16_t* residual;
    int n0, n1;
    uint16_t* y1;
    uint16_t* y2;
};
// The launch is a programmatic dependent of the stream's previous kernel; early_weights lets
// it read the tiles before that kernel has finished (see attn_w4bf16_gemv).
cudaError_t launch_w4_gemv(const uint8_t* tiles, const uint16_t* x, int M, int N, int K, uint16_t* y, int* err,
                           bool early_weights, const W4Fused& fz, cudaStream_t st);

// W4BF16 GEMM (w4_gemm.cu): y[t, n] = sum_k x[t, k] bf16((q - z) s)[n, k] for T tokens;
// N and K multiples of 128; x bf16 [T][K] and y bf16 [T][N] 16-byte aligned; tiles: the
// tile stream of attn_w4bf16_gemv.
// Epilogue options (all optional): the output columns split three ways -- [0, n0) -> y
// (row stride n0), [n0, n1) -> y1, [n1, N) -> y2 (n0, n1 multiples of 32; no split: n0 =
// n1 = N) -- or a bf16 residual [T][N] added in float before rounding (unsplit only; it
// may be y itself: each element is read before it is written).
struct W4GemmEpi {
    int n0, n1;
    uint16_t* y1;
    uint16_t* y2;
    const uint16_t* residual;
};
cudaError_t launch_w4_gemm(const uint8_t* tiles, const uint16_t* x, int T, int N, int K, uint16_t* y, int* err,
                           cudaStream_t st, const W4GemmEpi* epi = nullptr);
// RMSNorm of T rows of x (bf16 [T][K], K a multiple of 8, 16-byte aligned) into xn (same
// shape): xn = bf16(x * r * gamma), r = 1 / sqrt(mean_k x^2 + eps) per row, float math (the
// sum of squares in a fixed order); gamma bf16 [K].
cudaError_t launch_rmsnorm_rows(const uint16_t* x, const uint16_t* gamma, float eps, int T, int K, uint16_t* xn,
                                cudaStream_t st);

#ifdef __CUDACC__
// Position of sequence b's decode token: d_hist[b] + hist_add, or -1 (out of range, so
// the caller flags and skips the sequence) when the sum leaves int.
__device__ __forceinline__ int decode_hist(const int32_t* d_hist, int b, int hist_add) {
    const long long h = static_cast<long long>(d_hist[b]) + hist_add;
    return h > 0x7FFFFFFFLL ? -1 : static_cast<int>(h);
}
#endif

}  // namespace attn

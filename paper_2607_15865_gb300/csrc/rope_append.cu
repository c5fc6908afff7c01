// rope_append.cu -- K1: RoPE of the new keys and in-place KV-cache append.
//
// For every sequence b and new token i at position p = hist + i (decode: hist =
// hist_len[b] read on the device), kv head g:
//   k_cache[b, g, p, :] = bf16(rope(k[b, i, g, :], p)),  v_cache[b, g, p, :] = v[b, i, g, :]
// (Listing 2 "Rope" + "Concat", implemented as an in-place update as Section
// 4.6.3 asks).  RoPE pairs element j with j + D/2; cos/sin are gathered from the
// context's float table row p (Section 4.6.2).  The products and the difference
// (or sum) are each rounded to float (no fused multiply-add), then the result is
// rounded to bf16, nearest even.  No other cache slot is touched.
//
// One CTA per (token, sequence); each thread handles 8 rotation pairs or 8 v
// elements with 16-byte loads and stores.  Pure bandwidth: 2*D*2 bytes read and
// written per (token, kv head), plus 2*(D/2)*4 table bytes per token (L2-resident).
#include <cuda_bf16.h>

#include "internal.h"

namespace attn {
namespace {

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    const __nv_bfloat162 t = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&t);
}

template <int D>
__global__ void __launch_bounds__(128) rope_append_kernel(const uint16_t* __restrict__ k,
                                                          const uint16_t* __restrict__ v, int hist,
                                                          const int32_t* __restrict__ d_hist, int chunk,
                                                          int seq_stride, int Hkv,
                                                          int max_len, const float* __restrict__ cos_tab,
                                                          const float* __restrict__ sin_tab,
                                                          const float* __restrict__ cos_t, const float* __restrict__ sin_t,
                                                          uint16_t* __restrict__ k_cache,
                                                          uint16_t* __restrict__ v_cache, int* __restrict__ err) {
    constexpr int HALF = D / 2;
    constexpr int ROPE_UNITS = D / 16;  // 8 pairs per unit
    constexpr int COPY_UNITS = D / 8;   // 8 elements per unit
    // K1 is launched in stream order (its inputs are complete when it starts); the K2
    // launch that follows it may begin its q-side prologue as soon as every K1 CTA runs.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int i = blockIdx.x;
    const int b = blockIdx.y;
    int h0 = hist;
    if (d_hist != nullptr) {
        h0 = d_hist[b];
        if (h0 < 0 || h0 + chunk > max_len) {
            if (threadIdx.x == 0) atomicOr(err, kDevErrHistRange);
            return;
        }
    }
    const int p = h0 + i;
    // Warm L2 with the lines of the table copies in groups of four pairs (cos_t, sin_t:
    // [D/8][max_len][4]) that the attention kernel's softmax threads read to rotate the q
    // rows of this chunk: the CTA of every 32nd position (and the first) touches the four
    // 128-byte lines of the 32 positions from p & ~31 in every group and table (a line
    // that starts past the table's end is skipped).
    const int p32 = p & ~31, line = static_cast<int>(threadIdx.x) & 3;
    if (cos_t != nullptr && b == 0 && threadIdx.x < D && (i == 0 || (p & 31) == 0) && p32 + 8 * line < max_len) {
        const float* tab = threadIdx.x < HALF ? cos_t : sin_t;
        const int g = (static_cast<int>(threadIdx.x) % HALF) / 4;
        asm volatile("prefetch.global.L2 [%0];" ::"l"(tab + (static_cast<size_t>(g) * max_len + p32) * 4 + 32 * line));
    }
    const int n_rope = Hkv * ROPE_UNITS;
    const int n_units = n_rope + Hkv * COPY_UNITS;
    for (int u = threadIdx.x; u < n_units; u += blockDim.x) {
        if (u < n_rope) {
            const int g = u / ROPE_UNITS;
            const int j0 = (u % ROPE_UNITS) * 8;
            const size_t src = ((static_cast<size_t>(b) * seq_stride + i) * Hkv + g) * D;
            const size_t dst = ((static_cast<size_t>(b) * Hkv + g) * max_len + p) * D;
            const uint4 xa = *reinterpret_cast<const uint4*>(k + src + j0);
            const uint4 xb = *reinterpret_cast<const uint4*>(k + src + j0 + HALF);
            const float4* cp = reinterpret_cast<const float4*>(cos_tab + static_cast<size_t>(p) * HALF + j0);
            const float4* sp = reinterpret_cast<const float4*>(sin_tab + static_cast<size_t>(p) * HALF + j0);
            const float4 c0 = cp[0], c1 = cp[1], s0 = sp[0], s1 = sp[1];
            const float c[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
            const float s[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
            const uint32_t wa[4] = {xa.x, xa.y, xa.z, xa.w};
            const uint32_t wb[4] = {xb.x, xb.y, xb.z, xb.w};
            uint32_t ya[4], yb[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                float lo[2], hi[2];
#pragma unroll
                for (int t = 0; t < 2; ++t) {
                    const float a = t ? bf_hi(wa[e]) : bf_lo(wa[e]);
                    const float bb = t ? bf_hi(wb[e]) : bf_lo(wb[e]);
                    const float cc = c[2 * e + t], ss = s[2 * e + t];
                    lo[t] = __fsub_rn(__fmul_rn(a, cc), __fmul_rn(bb, ss));
                    hi[t] = __fadd_rn(__fmul_rn(bb, cc), __fmul_rn(a, ss));
                }
                ya[e] = pack_bf16(lo[0], lo[1]);
                yb[e] = pack_bf16(hi[0], hi[1]);
            }
            *reinterpret_cast<uint4*>(k_cache + dst + j0) = make_uint4(ya[0], ya[1], ya[2], ya[3]);
            *reinterpret_cast<uint4*>(k_cache + dst + j0 + HALF) = make_uint4(yb[0], yb[1], yb[2], yb[3]);
        } else {
            const int w = u - n_rope;
            const int g = w / COPY_UNITS;
            const int off = (w % COPY_UNITS) * 8;
            const size_t src = ((static_cast<size_t>(b) * seq_stride + i) * Hkv + g) * D + off;
            const size_t dst = ((static_cast<size_t>(b) * Hkv + g) * max_len + p) * D + off;
            *reinterpret_cast<uint4*>(v_cache + dst) = *reinterpret_cast<const uint4*>(v + src);
        }
    }
}

}  // namespace

cudaError_t launch_rope_append(const Shape& s, const uint16_t* k, const uint16_t* v, int hist,
                               const int32_t* d_hist, int chunk, int seq_stride, const float* cos_tab,
                               const float* sin_tab, const float* cos_t, const float* sin_t, uint16_t* k_cache,
                               uint16_t* v_cache, int* err, cudaStream_t st) {
    const dim3 grid(static_cast<unsigned>(chunk), static_cast<unsigned>(s.batch));
    if (s.head_dim == 128)
        rope_append_kernel<128><<<grid, 128, 0, st>>>(k, v, hist, d_hist, chunk, seq_stride, s.n_kv_heads, s.max_len, cos_tab,
                                                      sin_tab, cos_t, sin_t, k_cache, v_cache, err);
    else
        rope_append_kernel<64><<<grid, 128, 0, st>>>(k, v, hist, d_hist, chunk, seq_stride, s.n_kv_heads, s.max_len, cos_tab,
                                                     sin_tab, cos_t, sin_t, k_cache, v_cache, err);
    return cudaGetLastError();
}

}  // namespace attn

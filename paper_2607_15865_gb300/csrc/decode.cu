// decode.cu -- K3 split-KV decode attention and K4 log-sum-exp combine.
//
// Decode (Section 4.4): one new query per sequence b at position p = hist_len[b]
// attends to cache slots [0, p] of its kv head (the new token's own k/v were
// written to slot p by K1 before this kernel runs).  The length mask of the paper
// is given as hist_len; slots past p are never read.
//
// K3: CTA (split s, kv head g [x head pass], sequence b) streams the keys
// [s*per, min((s+1)*per, p+1)) of kv head g once, for all G = Hq/Hkv query heads
// of the group together, so each cache byte is read from HBM exactly once.
// D/8 lanes share one key row (16-byte loads, a warp reads consecutive rows, so
// every load instruction covers contiguous 512 bytes); each thread keeps U rows
// of K and V in flight.  Scores are reduced across the row's lanes with xor
// shuffles, then an online softmax in the log2 domain (scale*log2(e) folded into
// the rotated query) updates a per-row-group (m, l, acc).  Row groups and warps
// are merged with the log-sum-exp rule and the split writes its unnormalised
// partial (m, l, acc[D]).
// K4: per (query head, sequence): m* = max m_s, l = sum l_s 2^(m_s-m*),
// out = sum acc_s 2^(m_s-m*) / l, rounded to bf16.
// The query's RoPE (table gather, Section 4.6.2) is applied in K3's prologue with
// the same float arithmetic and bf16 rounding as K1 applies to keys.
#include <cuda_bf16.h>

#include <cmath>

#include "internal.h"
#include "sm100_ptx.cuh"

namespace attn {
namespace {

constexpr int kDecodeWarps = 4;
constexpr int kDecodeUnroll = 4;

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ uint4 ld_stream(const uint16_t* p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

__device__ __forceinline__ void unpack8(const uint4& w, float (&f)[8]) {
    f[0] = bf_lo(w.x); f[1] = bf_hi(w.x); f[2] = bf_lo(w.y); f[3] = bf_hi(w.y);
    f[4] = bf_lo(w.z); f[5] = bf_hi(w.z); f[6] = bf_lo(w.w); f[7] = bf_hi(w.w);
}

__device__ __forceinline__ float round_bf16(float x) {
    return __bfloat162float(__float2bfloat16_rn(x));
}

// Merge (m2, l2, a2) into (m1, l1, a1); m in the log2 domain, -inf = empty.
template <int N>
__device__ __forceinline__ void lse_merge(float& m1, float& l1, float (&a1)[N], float m2, float l2,
                                          const float (&a2)[N]) {
    const float mm = fmaxf(m1, m2);
    if (mm == -INFINITY) return;
    const float w1 = (m1 == -INFINITY) ? 0.f : fast_exp2(m1 - mm);
    const float w2 = (m2 == -INFINITY) ? 0.f : fast_exp2(m2 - mm);
    l1 = l1 * w1 + l2 * w2;
#pragma unroll
    for (int e = 0; e < N; ++e) a1[e] = a1[e] * w1 + a2[e] * w2;
    m1 = mm;
}

template <int D, int GM>
__global__ void __launch_bounds__(kDecodeWarps * 32) decode_split_kernel(
    const uint16_t* __restrict__ q, const int32_t* __restrict__ d_hist, const uint16_t* __restrict__ k_cache,
    const uint16_t* __restrict__ v_cache, const float* __restrict__ cos_tab, const float* __restrict__ sin_tab,
    int Hq, int Hkv, int G, int passes, int max_len, int nsplit, float scale_log2, float* __restrict__ part_o,
    float* __restrict__ part_ml) {
    constexpr int LPR = D / 8;    // lanes per key row
    constexpr int RPW = 32 / LPR; // key rows per warp per load instruction
    constexpr int U = kDecodeUnroll;
    constexpr int KPI = kDecodeWarps * RPW * U;
    constexpr int HALF = D / 2;

    __shared__ float sm_m[kDecodeWarps][GM];
    __shared__ float sm_l[kDecodeWarps][GM];
    __shared__ float sm_acc[kDecodeWarps][GM][D];

    const int s = blockIdx.x;
    const int g = blockIdx.y / passes;
    const int pass = blockIdx.y % passes;
    const int b = blockIdx.z;
    const int h_begin = g * G + pass * GM;
    const int gcount = min(GM, G - pass * GM);
    const int hist = d_hist[b];
    if (hist < 0 || hist >= max_len) return;  // K1 has flagged it; sequence skipped
    const int nkeys = hist + 1;
    int per = (nkeys + nsplit - 1) / nsplit;
    per = max(per, 32);
    const int start = s * per;
    const int end = min(start + per, nkeys);

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int sub = lane % LPR;
    const int rowg = lane / LPR;
    const int d0 = sub * 8;

    float m[GM], l[GM], acc[GM][8];
#pragma unroll
    for (int h = 0; h < GM; ++h) {
        m[h] = -INFINITY;
        l[h] = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[h][e] = 0.f;
    }

    if (start < end) {
        // Rotated query (RoPE at position hist) for this thread's 8 elements, scaled by
        // scale*log2(e) so that dot products are log2-domain scores.
        float qf[GM][8];
        {
            const int jb = d0 % HALF;
            const float4* cp = reinterpret_cast<const float4*>(cos_tab + static_cast<size_t>(hist) * HALF + jb);
            const float4* sp = reinterpret_cast<const float4*>(sin_tab + static_cast<size_t>(hist) * HALF + jb);
            const float4 c0 = cp[0], c1 = cp[1], s0 = sp[0], s1 = sp[1];
            const float c[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
            const float sn[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
            const bool lower = d0 < HALF;
#pragma unroll
            for (int h = 0; h < GM; ++h) {
                if (h < gcount) {
                    const uint16_t* qrow = q + (static_cast<size_t>(b) * Hq + h_begin + h) * D;
                    float x[8], y[8];
                    unpack8(*reinterpret_cast<const uint4*>(qrow + d0), x);
                    unpack8(*reinterpret_cast<const uint4*>(qrow + (lower ? d0 + HALF : d0 - HALF)), y);
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        // lower half: a*c - b*s (a own, b partner); upper half: b*c + a*s (b own, a partner)
                        const float r = lower ? __fsub_rn(__fmul_rn(x[e], c[e]), __fmul_rn(y[e], sn[e]))
                                              : __fadd_rn(__fmul_rn(x[e], c[e]), __fmul_rn(y[e], sn[e]));
                        qf[h][e] = round_bf16(r) * scale_log2;
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 8; ++e) qf[h][e] = 0.f;
                }
            }
        }

        const size_t head_off = (static_cast<size_t>(b) * Hkv + g) * static_cast<size_t>(max_len) * D + d0;
        const uint16_t* kbase = k_cache + head_off;
        const uint16_t* vbase = v_cache + head_off;
        // The loop bound is uniform across the warp (all lanes take part in the shuffles).
        for (int kw = start + warp * U * RPW; kw < end; kw += KPI) {
            const int kb = kw + rowg;
            uint4 kr[U], vr[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int key = kb + u * RPW;
                if (key < end) {
                    kr[u] = ld_stream(kbase + static_cast<size_t>(key) * D);
                    vr[u] = ld_stream(vbase + static_cast<size_t>(key) * D);
                } else {
                    kr[u] = make_uint4(0, 0, 0, 0);
                    vr[u] = make_uint4(0, 0, 0, 0);
                }
            }
            float sc[U][GM];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                float kf[8];
                unpack8(kr[u], kf);
#pragma unroll
                for (int h = 0; h < GM; ++h) {
                    float part = 0.f;
#pragma unroll
                    for (int e = 0; e < 8; ++e) part = fmaf(qf[h][e], kf[e], part);
#pragma unroll
                    for (int off = LPR / 2; off > 0; off >>= 1) part += __shfl_xor_sync(0xFFFFFFFFu, part, off);
                    sc[u][h] = (kb + u * RPW < end) ? part : -INFINITY;
                }
            }
#pragma unroll
            for (int h = 0; h < GM; ++h) {
                float mx = sc[0][h];
#pragma unroll
                for (int u = 1; u < U; ++u) mx = fmaxf(mx, sc[u][h]);
                const float mn = fmaxf(m[h], mx);
                if (mn == -INFINITY) continue;
                const float alpha = fast_exp2(m[h] - mn);
                l[h] *= alpha;
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[h][e] *= alpha;
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const float pr = fast_exp2(sc[u][h] - mn);
                    l[h] += pr;
                    float vf[8];
                    unpack8(vr[u], vf);
#pragma unroll
                    for (int e = 0; e < 8; ++e) acc[h][e] = fmaf(pr, vf[e], acc[h][e]);
                }
                m[h] = mn;
            }
        }
        // merge the RPW row groups of the warp (lanes with equal `sub`)
#pragma unroll
        for (int off = LPR; off < 32; off <<= 1) {
#pragma unroll
            for (int h = 0; h < GM; ++h) {
                const float m2 = __shfl_xor_sync(0xFFFFFFFFu, m[h], off);
                const float l2 = __shfl_xor_sync(0xFFFFFFFFu, l[h], off);
                float a2[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) a2[e] = __shfl_xor_sync(0xFFFFFFFFu, acc[h][e], off);
                lse_merge(m[h], l[h], acc[h], m2, l2, a2);
            }
        }
    }
    // merge the warps through shared memory and write this split's partial
    if (rowg == 0) {
#pragma unroll
        for (int h = 0; h < GM; ++h) {
#pragma unroll
            for (int e = 0; e < 8; ++e) sm_acc[warp][h][d0 + e] = acc[h][e];
            if (sub == 0) {
                sm_m[warp][h] = m[h];
                sm_l[warp][h] = l[h];
            }
        }
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < gcount * D; idx += blockDim.x) {
        const int h = idx / D;
        const int d = idx % D;
        float mm = -INFINITY;
#pragma unroll
        for (int w = 0; w < kDecodeWarps; ++w) mm = fmaxf(mm, sm_m[w][h]);
        float ll = 0.f, aa = 0.f;
        if (mm != -INFINITY) {
#pragma unroll
            for (int w = 0; w < kDecodeWarps; ++w) {
                const float mw = sm_m[w][h];
                if (mw == -INFINITY) continue;
                const float wt = fast_exp2(mw - mm);
                ll += sm_l[w][h] * wt;
                aa += sm_acc[w][h][d] * wt;
            }
        }
        const size_t row = (static_cast<size_t>(b) * Hq + h_begin + h) * nsplit + s;
        part_o[row * D + d] = aa;
        if (d == 0) {
            part_ml[row * 2 + 0] = mm;
            part_ml[row * 2 + 1] = ll;
        }
    }
}

template <int D>
__global__ void __launch_bounds__(D) decode_combine_kernel(const float* __restrict__ part_o,
                                                           const float* __restrict__ part_ml,
                                                           const int32_t* __restrict__ d_hist, int Hq, int nsplit,
                                                           int max_len, uint16_t* __restrict__ out) {
    extern __shared__ float sm_w[];  // [nsplit] weights
    __shared__ float sm_inv_l;
    const int h = blockIdx.x;
    const int b = blockIdx.y;
    const int hist = d_hist[b];
    if (hist < 0 || hist >= max_len) return;
    const size_t row0 = (static_cast<size_t>(b) * Hq + h) * nsplit;
    if (threadIdx.x < 32) {
        float mm = -INFINITY;
        for (int s = threadIdx.x; s < nsplit; s += 32)
            if (part_ml[(row0 + s) * 2 + 1] > 0.f) mm = fmaxf(mm, part_ml[(row0 + s) * 2]);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) mm = fmaxf(mm, __shfl_xor_sync(0xFFFFFFFFu, mm, off));
        float ll = 0.f;
        for (int s = threadIdx.x; s < nsplit; s += 32) {
            const float ls = part_ml[(row0 + s) * 2 + 1];
            const float w = (ls > 0.f) ? fast_exp2(part_ml[(row0 + s) * 2] - mm) : 0.f;
            sm_w[s] = w;
            ll += ls * w;
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) ll += __shfl_xor_sync(0xFFFFFFFFu, ll, off);
        if (threadIdx.x == 0) sm_inv_l = 1.f / ll;
    }
    __syncthreads();
    const int d = threadIdx.x;
    float a = 0.f;
    for (int s = 0; s < nsplit; ++s) {
        const float w = sm_w[s];
        if (w != 0.f) a = fmaf(w, part_o[(row0 + s) * D + d], a);
    }
    out[(static_cast<size_t>(b) * Hq + h) * D + d] =
        __bfloat16_as_ushort(__float2bfloat16_rn(a * sm_inv_l));
}

template <int D, int GM>
void launch_split(const Shape& s, dim3 grid, const uint16_t* q, const int32_t* d_hist, const uint16_t* kc,
                  const uint16_t* vc, const float* cos_tab, const float* sin_tab, int G, int passes, int nsplit,
                  float scale_log2, float* part_o, float* part_ml, cudaStream_t st) {
    decode_split_kernel<D, GM><<<grid, kDecodeWarps * 32, 0, st>>>(q, d_hist, kc, vc, cos_tab, sin_tab,
                                                                   s.n_q_heads, s.n_kv_heads, G, passes,
                                                                   s.max_len, nsplit, scale_log2, part_o, part_ml);
}

template <int D>
void launch_split_d(const Shape& s, const uint16_t* q, const int32_t* d_hist, const uint16_t* kc,
                    const uint16_t* vc, const float* cos_tab, const float* sin_tab, int nsplit, float scale_log2,
                    float* part_o, float* part_ml, cudaStream_t st) {
    const int G = s.n_q_heads / s.n_kv_heads;
    const int gm = G <= 1 ? 1 : G <= 2 ? 2 : G <= 4 ? 4 : 8;
    const int passes = (G + gm - 1) / gm;
    const dim3 grid(static_cast<unsigned>(nsplit), static_cast<unsigned>(s.n_kv_heads * passes),
                    static_cast<unsigned>(s.batch));
    switch (gm) {
        case 1: launch_split<D, 1>(s, grid, q, d_hist, kc, vc, cos_tab, sin_tab, G, passes, nsplit, scale_log2, part_o, part_ml, st); break;
        case 2: launch_split<D, 2>(s, grid, q, d_hist, kc, vc, cos_tab, sin_tab, G, passes, nsplit, scale_log2, part_o, part_ml, st); break;
        case 4: launch_split<D, 4>(s, grid, q, d_hist, kc, vc, cos_tab, sin_tab, G, passes, nsplit, scale_log2, part_o, part_ml, st); break;
        default: launch_split<D, 8>(s, grid, q, d_hist, kc, vc, cos_tab, sin_tab, G, passes, nsplit, scale_log2, part_o, part_ml, st); break;
    }
}

}  // namespace

cudaError_t launch_decode_split(const Shape& s, const uint16_t* q, const int32_t* d_hist, const uint16_t* k_cache,
                                const uint16_t* v_cache, const float* cos_tab, const float* sin_tab, float* part_o,
                                float* part_ml, int nsplit, cudaStream_t st) {
    const float scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(s.head_dim)));
    if (s.head_dim == 128)
        launch_split_d<128>(s, q, d_hist, k_cache, v_cache, cos_tab, sin_tab, nsplit, scale_log2, part_o, part_ml, st);
    else
        launch_split_d<64>(s, q, d_hist, k_cache, v_cache, cos_tab, sin_tab, nsplit, scale_log2, part_o, part_ml, st);
    return cudaGetLastError();
}

cudaError_t launch_decode_combine(const Shape& s, const int32_t* d_hist, const float* part_o, const float* part_ml,
                                  int nsplit, uint16_t* out, cudaStream_t st) {
    const dim3 grid(static_cast<unsigned>(s.n_q_heads), static_cast<unsigned>(s.batch));
    const size_t smem = sizeof(float) * static_cast<size_t>(nsplit);
    if (s.head_dim == 128)
        decode_combine_kernel<128><<<grid, 128, smem, st>>>(part_o, part_ml, d_hist, s.n_q_heads, nsplit, s.max_len, out);
    else
        decode_combine_kernel<64><<<grid, 64, smem, st>>>(part_o, part_ml, d_hist, s.n_q_heads, nsplit, s.max_len, out);
    return cudaGetLastError();
}

}  // namespace attn

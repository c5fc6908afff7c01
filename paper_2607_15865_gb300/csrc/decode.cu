// decode.cu -- K3 split-KV decode attention (with the new token's RoPE + append fused
// in) and K4 log-sum-exp combine.
//
// Decode (Section 4.4): one new query per sequence b at position p = hist_len[b]
// attends to cache slots [0, p] of its kv head; its own k/v go to slot p (the
// in-place "Concat" of Listing 2, Section 4.6.3).  The length mask of the paper is
// given as hist_len on the device; slots past p are never used.
//
// K3: CTA (split s, kv head g [x head pass], sequence b) owns keys
// [s*per, min((s+1)*per, p+1)), per = max(ceil((p+1)/nsplit), 64) computed on the
// device.  It streams them once for all query heads of the group:
//   * thread 0 issues TMA tensor loads of 64-key K and V tiles (128-byte swizzle)
//     into a 3-stage shared-memory ring (two CTAs per SM keep ~200 KB in flight);
//   * QK: one key per thread over a quarter of D, the rotated queries (scale *
//     log2(e) folded in) read from shared memory, partial sums to shared memory;
//   * softmax: one warp per query head merges the partials, keeps the running
//     (max, sum) in the log2 domain and writes the tile's P;
//   * PV: one 16-byte V chunk per thread over a quarter of the tile's keys,
//     accumulators rescaled by 2^(m_old - m_new);
//   * the split whose range holds slot p rotates the new k (RoPE from the table,
//     the same float arithmetic and bf16 rounding as K1), writes k and v to slot p
//     and substitutes them for that row of the loaded tile.
// Each split writes its unnormalised partial (m, l, acc[D]) per head.
// K4: per (query head, sequence): m* = max m_s, l = sum l_s 2^(m_s-m*),
// out = sum acc_s 2^(m_s-m*) / l -> bf16; a programmatic dependent launch of K3.
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>

#include "internal.h"
#include "sm100_ptx.cuh"

namespace attn {
namespace {

constexpr int KT = 64;        // keys per tile
constexpr int NSTAGE = 3;     // TMA ring depth
constexpr int NTHREADS = 256;
constexpr int NSLICE = 4;     // D slices of the QK phase

template <int D, int GM>
struct DecLayout {
    static constexpr int DCH = D / 64;                 // 128-byte column boxes per row
    static constexpr int BOX = KT * 128;               // bytes of one [KT x 64] box
    static constexpr int TILE = DCH * BOX;             // one K (or V) tile
    static constexpr int STAGE = 2 * TILE;
    static constexpr int OFF_Q = NSTAGE * STAGE;                    // float q[GM][D]
    static constexpr int OFF_PART = OFF_Q + GM * D * 4;             // float part[NSLICE][GM][KT]
    static constexpr int OFF_P = OFF_PART + NSLICE * GM * KT * 4;   // float P[KT][8]
    static constexpr int OFF_ALPHA = OFF_P + KT * 8 * 4;            // float alpha[8]
    static constexpr int OFF_ML = OFF_ALPHA + 8 * 4;                // float m[8], l[8]
    static constexpr int OFF_KNEW = OFF_ML + 16 * 4;                // bf16 k_new[D], v_new[D]
    static constexpr int OFF_BAR = OFF_KNEW + 2 * D * 2;
    static constexpr int BYTES = OFF_BAR + NSTAGE * 8;
    static constexpr int ALLOC = BYTES + 1024;
    static constexpr int NKG = NTHREADS / (D / 8);     // key groups of the PV phase
    static constexpr int KPT = KT / NKG;               // keys per PV thread per tile
    static_assert((NTHREADS / 32) * GM * D * 4 <= NSTAGE * STAGE, "the final reduction reuses the ring");
    static_assert(2 * (ALLOC + 1024) <= 233472, "two CTAs per SM");
};

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ float bf16_at(const uint16_t* p) { return __uint_as_float(static_cast<uint32_t>(*p) << 16); }
__device__ __forceinline__ uint16_t to_bf16(float x) { return __bfloat16_as_ushort(__float2bfloat16_rn(x)); }

// Byte offset of the 16-byte chunk c (dims 8c..8c+7) of row r in a tile stored as
// 128-byte-swizzled [KT x 64] boxes (TMA SWIZZLE_128B).
__device__ __forceinline__ uint32_t swz(int r, int c) {
    return static_cast<uint32_t>((c >> 3) * (KT * 128) + r * 128 + (((c & 7) ^ (r & 7)) << 4));
}

// RoPE of element d of a head vector with the table row of its position (pairs j,
// j + D/2); each product and the difference/sum rounded to float separately.
template <int D>
__device__ __forceinline__ float rope_elem(const uint16_t* x, int d, const float* cos_row, const float* sin_row) {
    constexpr int HALF = D / 2;
    const int j = d % HALF;
    const float c = cos_row[j], s = sin_row[j];
    if (d < HALF) return __fsub_rn(__fmul_rn(bf16_at(x + d), c), __fmul_rn(bf16_at(x + d + HALF), s));
    return __fadd_rn(__fmul_rn(bf16_at(x + d), c), __fmul_rn(bf16_at(x + d - HALF), s));
}

__device__ __forceinline__ void fma8(float (&acc)[8], float p, const uint4& w) {
    const float2 p2 = make_float2(p, p);
    float2 x;
    x = ffma2(p2, make_float2(bf_lo(w.x), bf_hi(w.x)), make_float2(acc[0], acc[1])); acc[0] = x.x; acc[1] = x.y;
    x = ffma2(p2, make_float2(bf_lo(w.y), bf_hi(w.y)), make_float2(acc[2], acc[3])); acc[2] = x.x; acc[3] = x.y;
    x = ffma2(p2, make_float2(bf_lo(w.z), bf_hi(w.z)), make_float2(acc[4], acc[5])); acc[4] = x.x; acc[5] = x.y;
    x = ffma2(p2, make_float2(bf_lo(w.w), bf_hi(w.w)), make_float2(acc[6], acc[7])); acc[6] = x.x; acc[7] = x.y;
}

template <int D, int GM>
__global__ void __launch_bounds__(NTHREADS, 2) decode_split_kernel(
    const __grid_constant__ CUtensorMap map_k, const __grid_constant__ CUtensorMap map_v,
    const uint16_t* __restrict__ q, const uint16_t* __restrict__ k_new, const uint16_t* __restrict__ v_new,
    const int32_t* __restrict__ d_hist, int hist_add, uint16_t* __restrict__ k_cache, uint16_t* __restrict__ v_cache,
    const float* __restrict__ cos_tab, const float* __restrict__ sin_tab, int Hq, int Hkv, int G, int passes,
    int max_len, int nsplit, float scale_log2, float* __restrict__ part_o, float* __restrict__ part_ml,
    int* __restrict__ err, uint64_t wait_ns) {
    using L = DecLayout<D, GM>;
    constexpr int HALF = D / 2;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* gb = smem_raw + (base - raw);
    float* qs = reinterpret_cast<float*>(gb + L::OFF_Q);
    float* part = reinterpret_cast<float*>(gb + L::OFF_PART);
    float* P = reinterpret_cast<float*>(gb + L::OFF_P);
    float* alpha_s = reinterpret_cast<float*>(gb + L::OFF_ALPHA);
    float* ml_s = reinterpret_cast<float*>(gb + L::OFF_ML);
    uint16_t* knew_s = reinterpret_cast<uint16_t*>(gb + L::OFF_KNEW);
    uint16_t* vnew_s = knew_s + D;

    const int s = blockIdx.x;
    const int g = blockIdx.y / passes;
    const int pass = blockIdx.y % passes;
    const int b = blockIdx.z;
    const int h0 = g * G + pass * GM;
    const int gcount = min(GM, G - pass * GM);
    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;

    const int hist = decode_hist(d_hist, b, hist_add);
    if (hist < 0 || hist >= max_len) {
        if (s == 0 && blockIdx.y == 0 && tid == 0) atomicOr(err, kDevErrHistRange);
        return;  // sequence skipped: nothing written
    }
    const int nkeys = hist + 1;
    const int per = max((nkeys + nsplit - 1) / nsplit, KT);
    const int start = s * per;
    const int end = min(start + per, nkeys);
    const size_t row0 = (static_cast<size_t>(b) * Hq + h0) * nsplit + s;  // head h adds h*nsplit
    if (start >= end) {  // an empty split: weight 0 in the combine
        if (tid < gcount) {
            part_ml[(row0 + static_cast<size_t>(tid) * nsplit) * 2 + 0] = -INFINITY;
            part_ml[(row0 + static_cast<size_t>(tid) * nsplit) * 2 + 1] = 0.f;
        }
        return;
    }
    const int ntiles = (end - start + KT - 1) / KT;
    const int kv_row = b * Hkv + g;
    auto bar = [&](int st) -> uint32_t { return base + L::OFF_BAR + 8u * static_cast<uint32_t>(st); };
    int n_issued = 0;  // tiles issued so far (thread 0 only)
    auto issue = [&](int j) {
        const int st = j % NSTAGE;
        const uint32_t kdst = base + st * L::STAGE;
        // a refill overwrites a stage the CTA accessed through the generic proxy
        if (j >= NSTAGE) fence_proxy_async_smem();
        mbar_arrive_expect_tx(bar(st), L::STAGE);
#pragma unroll
        for (int c = 0; c < L::DCH; ++c) {
            tma_load_3d(kdst + c * L::BOX, &map_k, c * 64, start + j * KT, kv_row, bar(st));
            tma_load_3d(kdst + L::TILE + c * L::BOX, &map_v, c * 64, start + j * KT, kv_row, bar(st));
        }
        n_issued = j + 1;
    };
    if (tid == 0) {
        for (int st = 0; st < NSTAGE; ++st) mbar_init(bar(st), 1);
        fence_mbar_init();
    }
    __syncthreads();
    if (tid == 0) {
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_v);
        for (int j = 0; j < min(NSTAGE, ntiles); ++j) issue(j);
    }

    // Prologue: rotated queries (scaled into the log2 domain) and, for the split that
    // owns slot `hist`, the new token's rotated k and its v, appended to the cache.
    const float* cos_row = cos_tab + static_cast<size_t>(hist) * HALF;
    const float* sin_row = sin_tab + static_cast<size_t>(hist) * HALF;
    for (int idx = tid; idx < GM * D; idx += NTHREADS) {
        const int h = idx / D, d = idx % D;
        float v = 0.f;
        if (h < gcount) {
            const uint16_t* qrow = q + (static_cast<size_t>(b) * Hq + h0 + h) * D;
            v = __bfloat162float(__float2bfloat16_rn(rope_elem<D>(qrow, d, cos_row, sin_row))) * scale_log2;
        }
        qs[idx] = v;
    }
    const bool own_new = hist >= start && hist < end;
    if (own_new && tid < D) {
        const uint16_t* krow = k_new + static_cast<size_t>(kv_row) * D;
        const uint16_t kr = to_bf16(rope_elem<D>(krow, tid, cos_row, sin_row));
        const uint16_t vv = v_new[static_cast<size_t>(kv_row) * D + tid];
        knew_s[tid] = kr;
        vnew_s[tid] = vv;
        if (pass == 0) {
            const size_t dst = (static_cast<size_t>(kv_row) * max_len + hist) * D + tid;
            k_cache[dst] = kr;
            v_cache[dst] = vv;
        }
    }
    float m_run = -INFINITY, l_run = 0.f;  // warp h < gcount: running state of head h
    float acc[GM][8];
#pragma unroll
    for (int h = 0; h < GM; ++h)
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[h][e] = 0.f;
    __syncthreads();

    bool ok = true;
    const int qk_key = tid % KT;
    const int qk_slice = tid / KT;
    const int pv_chunk = tid % (D / 8);
    const int pv_group = tid / (D / 8);
    int j = 0;
    for (; j < ntiles; ++j) {
        const int st = j % NSTAGE;
        ok = mbar_wait(bar(st), static_cast<uint32_t>(j / NSTAGE) & 1u, nullptr, wait_ns);
        if (__syncthreads_or(!ok)) {
            ok = false;
            break;
        }
        uint8_t* ks = gb + st * L::STAGE;
        uint8_t* vs = ks + L::TILE;
        const int kt0 = start + j * KT;
        if (own_new && hist >= kt0 && hist < kt0 + KT) {  // CTA-uniform
            const int r = hist - kt0;
            if (tid < D / 8) {
                *reinterpret_cast<uint4*>(ks + swz(r, tid)) = reinterpret_cast<const uint4*>(knew_s)[tid];
                *reinterpret_cast<uint4*>(vs + swz(r, tid)) = reinterpret_cast<const uint4*>(vnew_s)[tid];
            }
            __syncthreads();
        }
        // ---- QK: one key, one quarter of D, every head of the pass
        {
            float2 a2[GM];
#pragma unroll
            for (int h = 0; h < GM; ++h) a2[h] = make_float2(0.f, 0.f);
#pragma unroll
            for (int cc = 0; cc < D / 32; ++cc) {
                const int c = qk_slice * (D / 32) + cc;
                const uint4 kw = *reinterpret_cast<const uint4*>(ks + swz(qk_key, c));
                const float2 k0 = make_float2(bf_lo(kw.x), bf_hi(kw.x));
                const float2 k1 = make_float2(bf_lo(kw.y), bf_hi(kw.y));
                const float2 k2 = make_float2(bf_lo(kw.z), bf_hi(kw.z));
                const float2 k3 = make_float2(bf_lo(kw.w), bf_hi(kw.w));
#pragma unroll
                for (int h = 0; h < GM; ++h) {
                    const float4 qa = *reinterpret_cast<const float4*>(qs + h * D + c * 8);
                    const float4 qb = *reinterpret_cast<const float4*>(qs + h * D + c * 8 + 4);
                    a2[h] = ffma2(make_float2(qa.x, qa.y), k0, a2[h]);
                    a2[h] = ffma2(make_float2(qa.z, qa.w), k1, a2[h]);
                    a2[h] = ffma2(make_float2(qb.x, qb.y), k2, a2[h]);
                    a2[h] = ffma2(make_float2(qb.z, qb.w), k3, a2[h]);
                }
            }
#pragma unroll
            for (int h = 0; h < GM; ++h) part[(qk_slice * GM + h) * KT + qk_key] = a2[h].x + a2[h].y;
        }
        __syncthreads();
        // every thread is past the PV of tile j-1: refill its ring stage
        if (tid == 0 && j >= 1 && j - 1 + NSTAGE < ntiles) issue(j - 1 + NSTAGE);
        // ---- softmax: warp h owns head h
        if (warp < gcount) {
            const int h = warp;
            float sc[2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int r = lane + 32 * u;
                float v = 0.f;
#pragma unroll
                for (int sl = 0; sl < NSLICE; ++sl) v += part[(sl * GM + h) * KT + r];
                sc[u] = (kt0 + r < end) ? v : -INFINITY;
            }
            float mx = fmaxf(sc[0], sc[1]);
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, off));
            const float m_new = fmaxf(m_run, mx);          // finite: the tile has a valid key
            const float alpha = fast_exp2(m_run - m_new);  // 0 on the first tile
            const float p0 = fast_exp2(sc[0] - m_new);
            const float p1 = fast_exp2(sc[1] - m_new);
            float sum = p0 + p1;
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, off);
            l_run = l_run * alpha + sum;
            m_run = m_new;
            P[lane * 8 + h] = p0;
            P[(lane + 32) * 8 + h] = p1;
            if (lane == 0) alpha_s[h] = alpha;
        }
        __syncthreads();
        // ---- PV: one 16-byte chunk of V per thread over KPT keys of the tile
#pragma unroll
        for (int h = 0; h < GM; ++h) {
            const float a = alpha_s[h < gcount ? h : 0];
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[h][e] *= a;
        }
#pragma unroll
        for (int i = 0; i < L::KPT; ++i) {
            const int r = pv_group + i * L::NKG;
            if (kt0 + r < end) {  // rows past the split's end may hold anything (never multiplied)
                const uint4 vw = *reinterpret_cast<const uint4*>(vs + swz(r, pv_chunk));
                const float4 pa = *reinterpret_cast<const float4*>(P + r * 8);
                const float4 pb = *reinterpret_cast<const float4*>(P + r * 8 + 4);
                const float pr[8] = {pa.x, pa.y, pa.z, pa.w, pb.x, pb.y, pb.z, pb.w};
#pragma unroll
                for (int h = 0; h < GM; ++h) fma8(acc[h], pr[h], vw);
            }
        }
    }
    if (!ok) {
        if (tid == 0) {
            atomicOr(err, kDevErrTimeout);
            // every copy issued must land before the CTA exits
            for (int t = max(0, n_issued - NSTAGE); t < n_issued; ++t)
                mbar_wait(bar(t % NSTAGE), static_cast<uint32_t>(t / NSTAGE) & 1u, nullptr);
        }
        __syncthreads();
        return;
    }
    // ---- merge the key groups (they share the CTA's running max) and write the partial:
    // first the groups inside a warp (shuffles), then the 8 warps through shared memory
#pragma unroll
    for (int off = D / 8; off < 32; off <<= 1)
#pragma unroll
        for (int h = 0; h < GM; ++h)
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[h][e] += __shfl_xor_sync(0xFFFFFFFFu, acc[h][e], off);
    __syncthreads();  // every thread is past the last tile; the ring is idle
    float* red = reinterpret_cast<float*>(gb);  // [8 warps][GM][D]
    if (lane < D / 8) {
#pragma unroll
        for (int h = 0; h < GM; ++h) {
            float4* dst = reinterpret_cast<float4*>(red + (warp * GM + h) * D + pv_chunk * 8);
            dst[0] = make_float4(acc[h][0], acc[h][1], acc[h][2], acc[h][3]);
            dst[1] = make_float4(acc[h][4], acc[h][5], acc[h][6], acc[h][7]);
        }
    }
    if (warp < gcount && lane == 0) {
        ml_s[warp] = m_run;
        ml_s[8 + warp] = l_run;
    }
    __syncthreads();
    for (int idx = tid; idx < gcount * D; idx += NTHREADS) {
        const int h = idx / D, d = idx % D;
        float a = 0.f;
#pragma unroll
        for (int w = 0; w < NTHREADS / 32; ++w) a += red[(w * GM + h) * D + d];
        const size_t row = row0 + static_cast<size_t>(h) * nsplit;
        part_o[row * D + d] = a;
        if (d == 0) {
            part_ml[row * 2 + 0] = ml_s[h];
            part_ml[row * 2 + 1] = ml_s[8 + h];
        }
    }
}

template <int D>
__global__ void __launch_bounds__(256) decode_combine_kernel(const float* __restrict__ part_o,
                                                             const float* __restrict__ part_ml,
                                                             const int32_t* __restrict__ d_hist, int hist_add, int Hq,
                                                             int nsplit,
                                                             int max_len, uint16_t* __restrict__ out) {
    constexpr int PER_LANE = D / 32;
    __shared__ float sm_w[256];
    __shared__ float sm_red[8][D];
    __shared__ float sm_inv_l;
    asm volatile("griddepcontrol.wait;" ::: "memory");  // K3's partials are complete and visible
    const int h = blockIdx.x;
    const int b = blockIdx.y;
    const int hist = decode_hist(d_hist, b, hist_add);
    if (hist < 0 || hist >= max_len) return;
    const size_t row0 = (static_cast<size_t>(b) * Hq + h) * nsplit;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp == 0) {
        float mm = -INFINITY;
        for (int s = lane; s < nsplit; s += 32)
            if (part_ml[(row0 + s) * 2 + 1] > 0.f) mm = fmaxf(mm, part_ml[(row0 + s) * 2]);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) mm = fmaxf(mm, __shfl_xor_sync(0xFFFFFFFFu, mm, off));
        float ll = 0.f;
        for (int s = lane; s < nsplit; s += 32) {
            const float ls = part_ml[(row0 + s) * 2 + 1];
            const float w = (ls > 0.f) ? fast_exp2(part_ml[(row0 + s) * 2] - mm) : 0.f;
            sm_w[s] = w;
            ll += ls * w;
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) ll += __shfl_xor_sync(0xFFFFFFFFu, ll, off);
        if (lane == 0) sm_inv_l = 1.f / ll;
    }
    __syncthreads();
    float a[PER_LANE];
#pragma unroll
    for (int e = 0; e < PER_LANE; ++e) a[e] = 0.f;
    for (int s = warp; s < nsplit; s += 8) {
        const float w = sm_w[s];
        if (w != 0.f) {  // empty splits' accumulators are never read
            const float* src = part_o + (row0 + s) * D + lane * PER_LANE;
#pragma unroll
            for (int e = 0; e < PER_LANE; ++e) a[e] = fmaf(w, src[e], a[e]);
        }
    }
#pragma unroll
    for (int e = 0; e < PER_LANE; ++e) sm_red[warp][lane * PER_LANE + e] = a[e];
    __syncthreads();
    for (int d = threadIdx.x; d < D; d += 256) {
        float t = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) t += sm_red[w][d];
        out[(static_cast<size_t>(b) * Hq + h) * D + d] = to_bf16(t * sm_inv_l);
    }
}

template <int D, int GM>
cudaError_t launch_split_t(const Shape& s, const DecodeMaps& maps, dim3 grid, const uint16_t* q,
                           const uint16_t* k_new, const uint16_t* v_new, const int32_t* d_hist, int hist_add,
                           uint16_t* kc, uint16_t* vc, const float* cos_tab, const float* sin_tab, int G, int passes,
                           int nsplit,
                           float scale_log2, float* part_o, float* part_ml, int* err, cudaStream_t st, uint64_t wait_ns) {
    decode_split_kernel<D, GM><<<grid, NTHREADS, DecLayout<D, GM>::ALLOC, st>>>(
        maps.k, maps.v, q, k_new, v_new, d_hist, hist_add, kc, vc, cos_tab, sin_tab, s.n_q_heads, s.n_kv_heads, G,
        passes,
        s.max_len, nsplit, scale_log2, part_o, part_ml, err, wait_ns);
    return cudaGetLastError();
}

template <int D>
cudaError_t launch_split_d(const Shape& s, const DecodeMaps& maps, const uint16_t* q, const uint16_t* k_new,
                           const uint16_t* v_new, const int32_t* d_hist, int hist_add, uint16_t* kc, uint16_t* vc,
                           const float* cos_tab, const float* sin_tab, int nsplit, float* part_o, float* part_ml,
                           int* err, cudaStream_t st, uint64_t wait_ns) {
    const float scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(D)));
    const int G = s.n_q_heads / s.n_kv_heads;
    const int passes = (G + 7) / 8;
    const int gm = (G + passes - 1) / passes;
    const dim3 grid(static_cast<unsigned>(nsplit), static_cast<unsigned>(s.n_kv_heads * passes),
                    static_cast<unsigned>(s.batch));
    switch (gm) {
#define ATTN_SPLIT_CASE(N)                                                                                     \
    case N:                                                                                                    \
        return launch_split_t<D, N>(s, maps, grid, q, k_new, v_new, d_hist, hist_add, kc, vc, cos_tab, sin_tab, G, \
                                    passes, nsplit, scale_log2, part_o, part_ml, err, st, wait_ns);
        ATTN_SPLIT_CASE(1) ATTN_SPLIT_CASE(2) ATTN_SPLIT_CASE(3) ATTN_SPLIT_CASE(4)
        ATTN_SPLIT_CASE(5) ATTN_SPLIT_CASE(6) ATTN_SPLIT_CASE(7) ATTN_SPLIT_CASE(8)
#undef ATTN_SPLIT_CASE
        default:
            return cudaErrorInvalidValue;
    }
}

template <int D, int GM>
cudaError_t set_smem_attr() {
    return cudaFuncSetAttribute(decode_split_kernel<D, GM>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                DecLayout<D, GM>::ALLOC);
}

}  // namespace

cudaError_t configure_decode() {
    cudaError_t e = cudaSuccess;
#define ATTN_CFG(D, N) \
    if (e == cudaSuccess) e = set_smem_attr<D, N>();
    ATTN_CFG(128, 1) ATTN_CFG(128, 2) ATTN_CFG(128, 3) ATTN_CFG(128, 4)
    ATTN_CFG(128, 5) ATTN_CFG(128, 6) ATTN_CFG(128, 7) ATTN_CFG(128, 8)
    ATTN_CFG(64, 1) ATTN_CFG(64, 2) ATTN_CFG(64, 3) ATTN_CFG(64, 4)
    ATTN_CFG(64, 5) ATTN_CFG(64, 6) ATTN_CFG(64, 7) ATTN_CFG(64, 8)
#undef ATTN_CFG
    return e;
}

int decode_num_splits(const Shape& s, int num_sms, int max_splits) {
    const int G = s.n_q_heads / s.n_kv_heads;
    const long items = static_cast<long>(s.batch) * s.n_kv_heads * ((G + 7) / 8);
    const long slots = 2L * num_sms;  // two CTAs per SM
    const long cap = std::max(1L, std::min<long>(max_splits, (s.max_len + KT - 1) / KT));
    // the smallest split count whose CTAs fill whole waves to >= 90%, else the best seen
    long best = 1;
    double best_eff = 0.0;
    for (long ns = 1; ns <= cap; ++ns) {
        const long ctas = items * ns;
        if (ctas < slots && ns < cap) continue;  // not enough CTAs to fill the GPU yet
        const double eff = static_cast<double>(ctas) / static_cast<double>(slots * ((ctas + slots - 1) / slots));
        if (eff >= 0.9) return static_cast<int>(ns);
        if (eff > best_eff) {
            best_eff = eff;
            best = ns;
        }
    }
    return static_cast<int>(best);
}

cudaError_t make_decode_maps(PFN_encodeTiled encode, const Shape& s, const uint16_t* k_cache,
                             const uint16_t* v_cache, DecodeMaps* maps) {
    const cuuint64_t D = static_cast<cuuint64_t>(s.head_dim);
    const cuuint64_t dims[3] = {D, static_cast<cuuint64_t>(s.max_len),
                                static_cast<cuuint64_t>(s.batch) * s.n_kv_heads};
    const cuuint64_t strides[2] = {D * 2, D * 2 * static_cast<cuuint64_t>(s.max_len)};
    const cuuint32_t box[3] = {64, KT, 1};
    const cuuint32_t estr[3] = {1, 1, 1};
    for (int i = 0; i < 2; ++i) {
        const CUresult r = encode(i == 0 ? &maps->k : &maps->v, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3,
                                  const_cast<uint16_t*>(i == 0 ? k_cache : v_cache), dims, strides, box, estr,
                                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    }
    return cudaSuccess;
}

cudaError_t launch_decode_split(const Shape& s, const DecodeMaps& maps, const uint16_t* q, const uint16_t* k_new,
                                const uint16_t* v_new, const int32_t* d_hist, int hist_add, uint16_t* k_cache,
                                uint16_t* v_cache, const float* cos_tab, const float* sin_tab, float* part_o,
                                float* part_ml, int nsplit, int* err, cudaStream_t st, uint64_t wait_ns) {
    if (s.head_dim == 128)
        return launch_split_d<128>(s, maps, q, k_new, v_new, d_hist, hist_add, k_cache, v_cache, cos_tab, sin_tab,
                                   nsplit, part_o, part_ml, err, st, wait_ns);
    return launch_split_d<64>(s, maps, q, k_new, v_new, d_hist, hist_add, k_cache, v_cache, cos_tab, sin_tab, nsplit,
                              part_o, part_ml, err, st, wait_ns);
}

cudaError_t launch_decode_combine(const Shape& s, const int32_t* d_hist, int hist_add, const float* part_o,
                                  const float* part_ml, int nsplit, uint16_t* out, cudaStream_t st) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(s.n_q_heads), static_cast<unsigned>(s.batch));
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (s.head_dim == 128)
        return cudaLaunchKernelEx(&cfg, decode_combine_kernel<128>, part_o, part_ml, d_hist, hist_add, s.n_q_heads, nsplit,
                                  s.max_len, out);
    return cudaLaunchKernelEx(&cfg, decode_combine_kernel<64>, part_o, part_ml, d_hist, hist_add, s.n_q_heads, nsplit,
                              s.max_len, out);
}

}  // namespace attn

// flash_fwd.cu -- K2: causal flash attention for prefill and prefill_kv on sm_103a.
//
// What it computes (Section 4.2-4.3; FAttention of Section 2.2 with the causal
// mask of Section 4.6.1): for the chunk's query rows i at positions p = hist + i
// and every query head h, out[b, i, h, :] = softmax_j(q_rot . k_j / sqrt(D)) v_j
// over cache slots j <= p of kv head h / G.  The caches already hold the chunk's
// rotated keys and values (K1 runs first), so the history and the new tokens are
// one contiguous key range [0, hist + chunk) -- the "Concat" of Listing 2 is the
// in-place layout itself.  prefill is the same kernel with hist = 0 (the paper's
// with_history template, Section 4.2).
//
// Design (one CTA = one 128-row query tile of one head; 192 threads):
//   warp 4      TMA producer: the q tile (4-D map straight from q [B,S,Hq,D]),
//               then K and V tiles of 128 keys into a 2-stage ring (128-byte
//               swizzle; rows past hist+chunk are zero-filled by the map bounds,
//               so unwritten cache slots are never read);
//   warp 5      tcgen05 issuer: S = Q K^T into one of two TMEM score buffers
//               (M=128, N=128, K=16 steps), then O += P V into the TMEM
//               accumulator (V as an MN-major operand);
//   warps 0-3   one thread per query row (= TMEM lane): RoPE of the q row in
//               shared memory before the first MMA (cos/sin gathered by position,
//               Section 4.6.2, float arithmetic, bf16 rounding as K1), then per
//               KV tile: scores from TMEM, causal mask by index compare (no mask
//               tensor), online softmax in the log2 domain, P as bf16 into a
//               swizzled shared buffer (double-buffered), rescale of the O row in
//               TMEM when the running maximum grew; finally O / l -> bf16 -> out.
// The MMA of tile j+1 overlaps the softmax of tile j (two score buffers).
// Every wait is bounded; on expiry the CTA records kDevErrTimeout, lets its
// in-flight copies and MMAs finish, releases TMEM and exits.
#include <cuda_bf16.h>

#include <cmath>

#include "internal.h"
#include "sm100_ptx.cuh"

namespace attn {
namespace {

constexpr int BM = 128;  // query rows per tile (TMEM lanes)
constexpr int BN = 128;  // keys per KV tile
constexpr int kThreads = 192;
constexpr int kWarpTma = 4;
constexpr int kWarpMma = 5;
constexpr uint32_t kTmemCols = 512;  // S0 [0,128) S1 [128,256) O [256,256+D)

enum Bar {
    B_QFULL, B_QREADY,
    B_KFULL0, B_KFULL1, B_KEMPTY0, B_KEMPTY1,
    B_VFULL0, B_VFULL1, B_VEMPTY0, B_VEMPTY1,
    B_SFULL0, B_SFULL1, B_PFULL0, B_PFULL1,
    B_PVDONE, B_DRAIN, NBAR
};

template <int D>
struct Layout {
    static constexpr int DCH = D / 64;          // 64-column (128-byte) chunks of a row
    static constexpr int CHUNK = 128 * 128;     // bytes of one 128-row x 128-byte chunk
    static constexpr int Q_BYTES = DCH * CHUNK;
    static constexpr int KV_BYTES = DCH * CHUNK;
    static constexpr int P_BYTES = (BN / 64) * CHUNK;
    static constexpr int OFF_Q = 0;
    static constexpr int OFF_K = OFF_Q + Q_BYTES;
    static constexpr int OFF_V = OFF_K + 2 * KV_BYTES;
    static constexpr int OFF_P = OFF_V + 2 * KV_BYTES;
    static constexpr int OFF_BAR = OFF_P + 2 * P_BYTES;
    static constexpr int OFF_TMEM = OFF_BAR + NBAR * 8;
    static constexpr int OFF_ABORT = OFF_TMEM + 8;
    static constexpr int BYTES = OFF_ABORT + 8;
    static constexpr int ALLOC = BYTES + 1024;  // slack to align the base to 1024 bytes
};
static_assert(Layout<128>::ALLOC <= 232448, "shared memory budget of one CTA");

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    const __nv_bfloat162 t = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&t);
}

// Byte offset of the 16-byte unit holding columns [8u, 8u+8) of row r inside a
// 128-row tile stored as 128-byte-swizzled 64-column chunks (TMA SWIZZLE_128B).
__device__ __forceinline__ uint32_t sw128_offset(int row, int col) {
    const int chunk = col >> 6;
    const int unit = (col & 63) >> 3;
    return static_cast<uint32_t>(chunk * (128 * 128) + row * 128 + ((unit ^ (row & 7)) << 4));
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    flash_fwd_kernel(const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_k,
                     const __grid_constant__ CUtensorMap map_v, int S, int H, int Hq, int Hkv, int n_qtiles,
                     float scale_log2, const float* __restrict__ cos_tab, const float* __restrict__ sin_tab,
                     uint16_t* __restrict__ out, int* __restrict__ err) {
    using L = Layout<D>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* gbase = smem_raw + (base - raw);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(gbase + L::OFF_ABORT);
    const uint32_t* tmem_holder = reinterpret_cast<const uint32_t*>(gbase + L::OFF_TMEM);
    auto bar = [&](int i) -> uint32_t { return base + L::OFF_BAR + 8u * static_cast<uint32_t>(i); };

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    // Longest rows first across every (head, sequence): with a causal mask the last
    // query tiles see the most keys, so they are dispatched before all shorter ones.
    const int heads_x_batch = static_cast<int>(gridDim.x) / n_qtiles;  // Hq * B
    const int lin = static_cast<int>(blockIdx.x);
    const int qt = n_qtiles - 1 - lin / heads_x_batch;
    const int h = (lin % heads_x_batch) % Hq;
    const int b = (lin % heads_x_batch) / Hq;
    const int g = h / (Hq / Hkv);
    const int q0 = qt * BM;
    const int rows_valid = min(BM, S - q0);
    const int n_kv = (H + q0 + rows_valid + BN - 1) / BN;

    if (threadIdx.x == 0) {
        *abort_flag = 0;
        mbar_init(bar(B_QFULL), 1);
        mbar_init(bar(B_QREADY), BM);
        for (int st = 0; st < 2; ++st) {
            mbar_init(bar(B_KFULL0 + st), 1);
            mbar_init(bar(B_KEMPTY0 + st), 1);
            mbar_init(bar(B_VFULL0 + st), 1);
            mbar_init(bar(B_VEMPTY0 + st), 1);
            mbar_init(bar(B_SFULL0 + st), 1);
            mbar_init(bar(B_PFULL0 + st), BM);
        }
        mbar_init(bar(B_PVDONE), 1);
        mbar_init(bar(B_DRAIN), 1);
        fence_mbar_init();
    }
    if (warp == kWarpMma) {
        tmem_alloc(base + L::OFF_TMEM, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;

    if (warp == kWarpTma) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            tma_prefetch_desc(&map_q);
            tma_prefetch_desc(&map_k);
            tma_prefetch_desc(&map_v);
            mbar_arrive_expect_tx(bar(B_QFULL), L::Q_BYTES);
#pragma unroll
            for (int c = 0; c < L::DCH; ++c)
                tma_load_4d(base + L::OFF_Q + c * L::CHUNK, &map_q, c * 64, h, q0, b, bar(B_QFULL));
            const int kv_row = b * Hkv + g;
            int issued_k[2] = {0, 0}, issued_v[2] = {0, 0};
            bool ok = true;
            for (int j = 0; j < n_kv; ++j) {
                const int st = j & 1;
                const uint32_t ph_free = static_cast<uint32_t>((j - 2) >> 1) & 1u;
                if (j >= 2 && !mbar_wait(bar(B_KEMPTY0 + st), ph_free, abort_flag)) { ok = false; break; }
                mbar_arrive_expect_tx(bar(B_KFULL0 + st), L::KV_BYTES);
#pragma unroll
                for (int c = 0; c < L::DCH; ++c)
                    tma_load_3d(base + L::OFF_K + st * L::KV_BYTES + c * L::CHUNK, &map_k, c * 64, j * BN, kv_row,
                                bar(B_KFULL0 + st));
                ++issued_k[st];
                if (j >= 2 && !mbar_wait(bar(B_VEMPTY0 + st), ph_free, abort_flag)) { ok = false; break; }
                mbar_arrive_expect_tx(bar(B_VFULL0 + st), L::KV_BYTES);
#pragma unroll
                for (int c = 0; c < L::DCH; ++c)
                    tma_load_3d(base + L::OFF_V + st * L::KV_BYTES + c * L::CHUNK, &map_v, c * 64, j * BN, kv_row,
                                bar(B_VFULL0 + st));
                ++issued_v[st];
            }
            if (!ok) {
                *abort_flag = 1;
                atomicOr(err, kDevErrTimeout);
            }
            // Every copy this thread issued must have landed before the CTA may exit.
            mbar_wait(bar(B_QFULL), 0, nullptr);
            for (int st = 0; st < 2; ++st) {
                if (issued_k[st]) mbar_wait(bar(B_KFULL0 + st), static_cast<uint32_t>(issued_k[st] - 1) & 1u, nullptr);
                if (issued_v[st]) mbar_wait(bar(B_VFULL0 + st), static_cast<uint32_t>(issued_v[st] - 1) & 1u, nullptr);
            }
        }
    } else if (warp == kWarpMma) {
        // ------------------------------------------------------------ tcgen05 issuer
        if (lane == 0) {
            constexpr uint32_t kIdS = idesc_bf16_f32(BM, BN, false, false);
            constexpr uint32_t kIdPV = idesc_bf16_f32(BM, D, false, true);
            const uint32_t sQ = base + L::OFF_Q;
            const uint32_t o_tmem = tmem + 2 * BN;
            auto issue_pv = [&](int jj) -> bool {
                const int st = jj & 1;
                const uint32_t ph = static_cast<uint32_t>(jj >> 1) & 1u;
                if (!mbar_wait(bar(B_PFULL0 + st), ph, abort_flag)) return false;
                if (!mbar_wait(bar(B_VFULL0 + st), ph, abort_flag)) return false;
                tc_fence_after();
                const uint32_t sP = base + L::OFF_P + st * L::P_BYTES;
                const uint32_t sV = base + L::OFF_V + st * L::KV_BYTES;
#pragma unroll
                for (int kk = 0; kk < BN / 16; ++kk) {
                    const uint64_t a = smem_desc_sw128(sP + (kk >> 2) * L::CHUNK + (kk & 3) * 32, 16, 1024);
                    const uint64_t bd = smem_desc_sw128(sV + kk * 16 * 128, L::CHUNK, 1024);
                    umma_ss(o_tmem, a, bd, kIdPV, (jj > 0 || kk > 0) ? 1u : 0u);
                }
                umma_commit(bar(B_PVDONE));
                umma_commit(bar(B_VEMPTY0 + st));
                return true;
            };
            bool ok = mbar_wait(bar(B_QREADY), 0, abort_flag);
            if (ok) {
                tc_fence_after();
                for (int j = 0; j < n_kv; ++j) {
                    const int st = j & 1;
                    const uint32_t ph = static_cast<uint32_t>(j >> 1) & 1u;
                    if (!mbar_wait(bar(B_KFULL0 + st), ph, abort_flag)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t sK = base + L::OFF_K + st * L::KV_BYTES;
                    const uint32_t s_tmem = tmem + st * BN;
#pragma unroll
                    for (int kk = 0; kk < D / 16; ++kk) {
                        const uint32_t off = (kk >> 2) * L::CHUNK + (kk & 3) * 32;
                        umma_ss(s_tmem, smem_desc_sw128(sQ + off, 16, 1024), smem_desc_sw128(sK + off, 16, 1024),
                                kIdS, kk > 0 ? 1u : 0u);
                    }
                    umma_commit(bar(B_SFULL0 + st));
                    umma_commit(bar(B_KEMPTY0 + st));
                    if (j >= 1 && !issue_pv(j - 1)) { ok = false; break; }
                }
                if (ok) ok = issue_pv(n_kv - 1);
            }
            if (!ok) {
                *abort_flag = 1;
                atomicOr(err, kDevErrTimeout);
            }
            // All tensor-core work issued here must finish before TMEM is released.
            umma_commit(bar(B_DRAIN));
            mbar_wait(bar(B_DRAIN), 0, nullptr);
        }
    } else {
        // ------------------------------------------------------------ softmax / epilogue warps
        constexpr int HALF = D / 2;
        const int t = threadIdx.x;  // query row in the tile == TMEM lane
        const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
        bool ok = mbar_wait(bar(B_QFULL), 0, abort_flag);
        ok = __all_sync(0xFFFFFFFFu, ok);
        if (ok && t < rows_valid) {
            // RoPE of this query row in place (pairs j, j + D/2), as K1 does for keys.
            const int pos = H + q0 + t;
            const float* crow = cos_tab + static_cast<size_t>(pos) * HALF;
            const float* srow = sin_tab + static_cast<size_t>(pos) * HALF;
#pragma unroll
            for (int u = 0; u < HALF / 8; ++u) {
                const int jlo = 8 * u;
                uint4* plo = reinterpret_cast<uint4*>(gbase + L::OFF_Q + sw128_offset(t, jlo));
                uint4* phi = reinterpret_cast<uint4*>(gbase + L::OFF_Q + sw128_offset(t, jlo + HALF));
                const uint4 xa = *plo, xb = *phi;
                const float4 c0 = *reinterpret_cast<const float4*>(crow + jlo);
                const float4 c1 = *reinterpret_cast<const float4*>(crow + jlo + 4);
                const float4 s0 = *reinterpret_cast<const float4*>(srow + jlo);
                const float4 s1 = *reinterpret_cast<const float4*>(srow + jlo + 4);
                const float c[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
                const float s[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
                const uint32_t wa[4] = {xa.x, xa.y, xa.z, xa.w};
                const uint32_t wb[4] = {xb.x, xb.y, xb.z, xb.w};
                uint32_t ya[4], yb[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    float lo[2], hi[2];
#pragma unroll
                    for (int k2 = 0; k2 < 2; ++k2) {
                        const float a = k2 ? bf_hi(wa[e]) : bf_lo(wa[e]);
                        const float bb = k2 ? bf_hi(wb[e]) : bf_lo(wb[e]);
                        const float cc = c[2 * e + k2], ss = s[2 * e + k2];
                        lo[k2] = __fsub_rn(__fmul_rn(a, cc), __fmul_rn(bb, ss));
                        hi[k2] = __fadd_rn(__fmul_rn(bb, cc), __fmul_rn(a, ss));
                    }
                    ya[e] = pack_bf16(lo[0], lo[1]);
                    yb[e] = pack_bf16(hi[0], hi[1]);
                }
                *plo = make_uint4(ya[0], ya[1], ya[2], ya[3]);
                *phi = make_uint4(yb[0], yb[1], yb[2], yb[3]);
            }
        }
        fence_proxy_async_smem();
        mbar_arrive(bar(B_QREADY));

        const int pos_row = H + q0 + t;  // last key this row may see
        const int min_pos = H + q0;      // smallest row position of the tile
        float m_run = -INFINITY;         // running maximum, log2 domain
        float l_run = 0.f;
        for (int j = 0; j < n_kv && ok; ++j) {
            const int st = j & 1;
            const uint32_t ph = static_cast<uint32_t>(j >> 1) & 1u;
            ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_SFULL0 + st), ph, abort_flag));
            if (!ok) break;
            tc_fence_after();
            uint32_t r[BN / 32][32];
#pragma unroll
            for (int c = 0; c < BN / 32; ++c) tmem_ld32(tmem + lane_base + st * BN + 32 * c, r[c]);
            tmem_wait_ld();
            const int kb = j * BN;
            float mx = -INFINITY;
            if (kb + BN - 1 > min_pos) {  // the tile crosses the diagonal: mask by index
#pragma unroll
                for (int c = 0; c < BN / 32; ++c)
#pragma unroll
                    for (int e = 0; e < 32; ++e) {
                        float v = __uint_as_float(r[c][e]);
                        v = (kb + 32 * c + e > pos_row) ? -INFINITY : v;
                        r[c][e] = __float_as_uint(v);
                        mx = fmaxf(mx, v);
                    }
            } else {
#pragma unroll
                for (int c = 0; c < BN / 32; ++c)
#pragma unroll
                    for (int e = 0; e < 32; ++e) mx = fmaxf(mx, __uint_as_float(r[c][e]));
            }
            // Lazy rescaling: P is taken relative to a reference max m_run that only moves
            // when the row max exceeds it by more than 2^8 (P <= 256 otherwise, exact in
            // bf16/fp32 ranges), so O and l are rescaled rarely; the result is unchanged.
            const float m_cand = fmaxf(m_run, mx * scale_log2);
            const bool move = m_cand > m_run + 8.f;  // always true on the first tile
            const float m_new = move ? m_cand : m_run;
            const float alpha = move ? fast_exp2(m_run - m_new) : 1.f;
            const float neg_m = -m_new;
            float rowsum = 0.f;
            uint8_t* pbuf = gbase + L::OFF_P + st * L::P_BYTES;
#pragma unroll
            for (int u8 = 0; u8 < BN / 8; ++u8) {
                const int c = u8 >> 2;
                const int e0 = (u8 & 3) * 8;
                float p[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    p[e] = fast_exp2(fmaf(__uint_as_float(r[c][e0 + e]), scale_log2, neg_m));
                    rowsum += p[e];
                }
                *reinterpret_cast<uint4*>(pbuf + sw128_offset(t, 8 * u8)) =
                    make_uint4(pack_bf16(p[0], p[1]), pack_bf16(p[2], p[3]), pack_bf16(p[4], p[5]),
                               pack_bf16(p[6], p[7]));
            }
            l_run = l_run * alpha + rowsum;
            if (j >= 1) {
                // O holds the sum through tile j-1 once PV(j-1) completes; rescale it.
                ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_PVDONE), static_cast<uint32_t>(j - 1) & 1u, abort_flag));
                if (!ok) break;
                tc_fence_after();
                if (__any_sync(0xFFFFFFFFu, alpha < 1.f)) {
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) {
                        uint32_t o[32];
                        const uint32_t ta = tmem + lane_base + 2 * BN + 32 * c;
                        tmem_ld32(ta, o);
                        tmem_wait_ld();
#pragma unroll
                        for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
                        tmem_st32(ta, o);
                    }
                    tmem_wait_st();
                }
            }
            m_run = m_new;
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(bar(B_PFULL0 + st));
        }
        if (ok) ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_PVDONE), static_cast<uint32_t>(n_kv - 1) & 1u, abort_flag));
        if (ok) {
            tc_fence_after();
            const float inv_l = 1.f / l_run;
            uint16_t* orow = out + ((static_cast<size_t>(b) * S + q0 + t) * Hq + h) * D;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t o[32];
                tmem_ld32(tmem + lane_base + 2 * BN + 32 * c, o);
                tmem_wait_ld();
                if (t < rows_valid) {
#pragma unroll
                    for (int v4 = 0; v4 < 4; ++v4) {
                        const float* f = reinterpret_cast<const float*>(o) + 8 * v4;
                        *reinterpret_cast<uint4*>(orow + 32 * c + 8 * v4) =
                            make_uint4(pack_bf16(f[0] * inv_l, f[1] * inv_l), pack_bf16(f[2] * inv_l, f[3] * inv_l),
                                       pack_bf16(f[4] * inv_l, f[5] * inv_l), pack_bf16(f[6] * inv_l, f[7] * inv_l));
                    }
                }
            }
        } else {
            *abort_flag = 1;
            atomicOr(err, kDevErrTimeout);
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kWarpMma) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

template <int D>
cudaError_t launch_d(const Shape& s, const FlashMaps& maps, int hist, int chunk, const float* cos_tab,
                     const float* sin_tab, uint16_t* out, int* err, cudaStream_t st) {
    const int n_qtiles = (chunk + BM - 1) / BM;
    const float scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(D)));
    const dim3 grid(static_cast<unsigned>(n_qtiles) * s.n_q_heads * s.batch);
    flash_fwd_kernel<D><<<grid, kThreads, Layout<D>::ALLOC, st>>>(maps.q, maps.k, maps.v, chunk, hist, s.n_q_heads,
                                                                   s.n_kv_heads, n_qtiles, scale_log2, cos_tab,
                                                                   sin_tab, out, err);
    return cudaGetLastError();
}

}  // namespace

cudaError_t configure_flash_fwd() {
    cudaError_t e = cudaFuncSetAttribute(flash_fwd_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Layout<128>::ALLOC);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(flash_fwd_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                Layout<64>::ALLOC);
}

cudaError_t launch_flash_fwd(const Shape& s, const FlashMaps& maps, int hist, int chunk, const float* cos_tab,
                             const float* sin_tab, uint16_t* out, int* err, int /*num_sms*/, cudaStream_t st) {
    if (s.head_dim == 128) return launch_d<128>(s, maps, hist, chunk, cos_tab, sin_tab, out, err, st);
    return launch_d<64>(s, maps, hist, chunk, cos_tab, sin_tab, out, err, st);
}

}  // namespace attn

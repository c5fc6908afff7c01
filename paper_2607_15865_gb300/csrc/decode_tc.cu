// decode_tc.cu -- K3 for head_dim 128: split-KV decode attention on the tensor cores.
//
// Decode (Section 4.4): one new query per sequence b at position p = hist_len[b]
// attends to cache slots [0, p] of its kv head; its own k/v go to slot p (the
// in-place "Concat" of Listing 2, Section 4.6.3).
//
// With grouped-query attention the G query heads of a kv head read the same keys,
// so a CTA's work is a contraction [G x D] x [D x keys] -- done here with tcgen05
// in swapped form so that the 128 keys of a tile fill the MMA's M dimension:
//   S^T [128 keys x 16] = K_tile [128 x D] . Q^T       (Q: G heads, zero-padded to 16)
//   O^T [D x 16]      += V_tile^T [D x 128] . P^T [128 x 16]
// Both accumulate in TMEM.  CTA (split s, kv head g, sequence b) owns keys
// [s*per, min((s+1)*per, p+1)), per computed on the device from p.  192 threads:
//   warps 0-3  one thread per key of the tile: scores from TMEM, per-head tile
//              max (shuffles + one exchange), lazy running max, P^T (bf16) into
//              shared memory; per-thread partial row sums; the epilogue (one
//              thread per output dimension d) writes the split's partial
//              (m, l, acc[D]) per head for K4 to merge;
//   warp 4     TMA producer: K and V tiles of 128 keys (128-byte swizzle) into a
//              3-stage ring, 64 KB per stage;
//   warp 5     tcgen05 issuer (S^T into one of two TMEM buffers, then O^T += ...).
// The split that owns slot p rotates the new k (RoPE from the table, the same
// float arithmetic and bf16 rounding as K1), writes k and v to slot p, uses
// q.k_new computed on the CUDA cores as that key's score and writes v_new over
// the loaded V row.  V rows past the split's end are zeroed before the PV MMA
// (the slots past hist_len may hold anything, and 0 * NaN would poison O).
// Every wait is bounded; on expiry the CTA records kDevErrTimeout, lets its
// copies and MMAs finish, releases TMEM and exits.
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>

#include "internal.h"
#include "sm100_ptx.cuh"

namespace attn {
namespace {

constexpr int D = 128;
constexpr int KT = 128;     // keys per tile (MMA M)
constexpr int NH = 16;      // padded query heads (MMA N)
constexpr int KST = 2;      // K ring stages (a K tile is free once S^T of it completes)
constexpr int VST = 4;      // V ring stages (a V tile is held until its PV completes)
constexpr int kThreads = 192;
constexpr int kWarpTma = 4;
constexpr int kWarpMma = 5;
constexpr uint32_t kTmemCols = 64;  // S^T x2 [0,32), O^T [32,48)
constexpr uint32_t TM_O = 32;

enum Bar { B_QREADY, B_KFULL0, B_KFULL1, B_KEMPTY0, B_KEMPTY1, B_VFULL0, B_VFULL1, B_VFULL2, B_VFULL3,
           B_VEMPTY0, B_VEMPTY1, B_VEMPTY2, B_VEMPTY3, B_SFULL0, B_SFULL1, B_PFULL0, B_PFULL1, B_PVDONE, B_OFULL,
           B_DRAIN, NBAR };

struct L {
    static constexpr int BOX = KT * 128;           // [128 keys x 64 dims] bf16, 16 KB
    static constexpr int TILE = 2 * BOX;           // one K (or V) tile, 32 KB
    static constexpr int OFF_K = 0;                // K ring
    static constexpr int OFF_V = KST * TILE;       // V ring
    static constexpr int OFF_Q = OFF_V + VST * TILE;  // Q^T [16 heads x 128] bf16, 2 x 2 KB
    static constexpr int OFF_P = OFF_Q + 2 * NH * 128;          // P^T [16 x 128 keys] x 2 buffers
    static constexpr int OFF_RED = OFF_P + 2 * 2 * NH * 128;    // float red[4 warps][16]
    static constexpr int OFF_NEWS = OFF_RED + 4 * NH * 4;       // float score of the new key [16]
    static constexpr int OFF_LS = OFF_NEWS + NH * 4;            // float l partials [4 warps][16]
    static constexpr int OFF_M = OFF_LS + 4 * NH * 4;           // float m [16]
    static constexpr int OFF_VNEW = OFF_M + NH * 4;             // bf16 v_new [128]
    static constexpr int OFF_BAR = OFF_VNEW + D * 2;
    static constexpr int OFF_TMEM = OFF_BAR + NBAR * 8;
    static constexpr int OFF_ABORT = OFF_TMEM + 8;
    static constexpr int BYTES = OFF_ABORT + 8;
    static constexpr int ALLOC = BYTES + 1024;
};
static_assert(L::ALLOC <= 232448, "shared memory of one CTA");

__device__ __forceinline__ float bf16_at(const uint16_t* p) { return __uint_as_float(static_cast<uint32_t>(*p) << 16); }
__device__ __forceinline__ uint16_t to_bf16(float x) { return __bfloat16_as_ushort(__float2bfloat16_rn(x)); }

// Byte offset of element (row, col) in a [rows x 128] bf16 tile stored as two
// 128-byte-swizzled 64-column chunks of `rows` rows (chunk stride rows * 128 bytes).
__device__ __forceinline__ uint32_t sw_elem(int row, int col, int rows) {
    return static_cast<uint32_t>((col >> 6) * rows * 128 + row * 128 + ((((col & 63) >> 3) ^ (row & 7)) << 4) +
                                 (col & 7) * 2);
}

__device__ __forceinline__ float rope_elem(const uint16_t* x, int d, const float* cos_row, const float* sin_row) {
    constexpr int HALF = D / 2;
    const int j = d % HALF;
    const float c = cos_row[j], s = sin_row[j];
    if (d < HALF) return __fsub_rn(__fmul_rn(bf16_at(x + d), c), __fmul_rn(bf16_at(x + d + HALF), s));
    return __fadd_rn(__fmul_rn(bf16_at(x + d), c), __fmul_rn(bf16_at(x + d - HALF), s));
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}

__device__ __forceinline__ void named_sync_128() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// Barrier 1 over the 128 softmax threads that also returns the OR of `pred`.
__device__ __forceinline__ bool named_or_128(bool pred) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, 1, 128, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"(static_cast<uint32_t>(pred))
        : "memory");
    return r != 0;
}

__global__ void __launch_bounds__(kThreads, 1) decode_tc_kernel(
    const __grid_constant__ CUtensorMap map_k, const __grid_constant__ CUtensorMap map_v,
    const uint16_t* __restrict__ q, const uint16_t* __restrict__ k_new, const uint16_t* __restrict__ v_new,
    const int32_t* __restrict__ d_hist, uint16_t* __restrict__ k_cache, uint16_t* __restrict__ v_cache,
    const float* __restrict__ cos_tab, const float* __restrict__ sin_tab, int Hq, int Hkv, int max_len, int nsplit,
    float scale_log2, float* __restrict__ part_o, float* __restrict__ part_ml, int* __restrict__ err) {
    constexpr int HALF = D / 2;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* gb = smem_raw + (base - raw);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(gb + L::OFF_ABORT);
    float* red = reinterpret_cast<float*>(gb + L::OFF_RED);
    float* news = reinterpret_cast<float*>(gb + L::OFF_NEWS);
    float* ls = reinterpret_cast<float*>(gb + L::OFF_LS);
    float* msh = reinterpret_cast<float*>(gb + L::OFF_M);
    uint16_t* vnew_s = reinterpret_cast<uint16_t*>(gb + L::OFF_VNEW);
    auto bar = [&](int i) -> uint32_t { return base + L::OFF_BAR + 8u * static_cast<uint32_t>(i); };

    const int G = Hq / Hkv;
    const int s = blockIdx.x;
    const int g = blockIdx.y;
    const int b = blockIdx.z;
    const int h0 = g * G;
    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;

    const int hist = d_hist[b];
    if (hist < 0 || hist >= max_len) {
        if (s == 0 && g == 0 && tid == 0) atomicOr(err, kDevErrHistRange);
        return;  // sequence skipped: nothing written
    }
    const int nkeys = hist + 1;
    const int per = max((nkeys + nsplit - 1) / nsplit, KT);
    const int start = s * per;
    const int end = min(start + per, nkeys);
    const size_t row0 = (static_cast<size_t>(b) * Hq + h0) * nsplit + s;  // head h adds h * nsplit
    if (start >= end) {  // an empty split: weight 0 in the combine
        if (tid < G) {
            part_ml[(row0 + static_cast<size_t>(tid) * nsplit) * 2 + 0] = -INFINITY;
            part_ml[(row0 + static_cast<size_t>(tid) * nsplit) * 2 + 1] = 0.f;
        }
        return;
    }
    const int ntiles = (end - start + KT - 1) / KT;
    const int kv_row = b * Hkv + g;
    const bool own_new = hist >= start && hist < end;

    if (tid == 0) {
        *abort_flag = 0;
        mbar_init(bar(B_QREADY), 128);
        for (int st = 0; st < KST; ++st) {
            mbar_init(bar(B_KFULL0 + st), 1);
            mbar_init(bar(B_KEMPTY0 + st), 1);
        }
        for (int st = 0; st < VST; ++st) {
            mbar_init(bar(B_VFULL0 + st), 1);
            mbar_init(bar(B_VEMPTY0 + st), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(B_SFULL0 + i), 1);
            mbar_init(bar(B_PFULL0 + i), 128);
        }
        mbar_init(bar(B_PVDONE), 1);
        mbar_init(bar(B_OFULL), 1);
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
    const uint32_t tmem = *reinterpret_cast<const uint32_t*>(gb + L::OFF_TMEM);

    if (warp == kWarpTma) {
        // ------------------------------------------------------------ TMA producer (lane 0: K, lane 1: V)
        if (lane < 2) {
            const bool is_k = lane == 0;
            const CUtensorMap* map = is_k ? &map_k : &map_v;
            const int nst = is_k ? KST : VST;
            const int full0 = is_k ? B_KFULL0 : B_VFULL0;
            const int empty0 = is_k ? B_KEMPTY0 : B_VEMPTY0;
            const uint32_t ring = base + (is_k ? L::OFF_K : L::OFF_V);
            tma_prefetch_desc(map);
            int issued = 0;
            bool ok = true;
            for (int j = 0; j < ntiles; ++j) {
                const int st = j % nst;
                if (j >= nst && !mbar_wait(bar(empty0 + st), static_cast<uint32_t>(j / nst - 1) & 1u, abort_flag)) {
                    ok = false;
                    break;
                }
                mbar_arrive_expect_tx(bar(full0 + st), L::TILE);
#pragma unroll
                for (int c = 0; c < 2; ++c)
                    tma_load_3d(ring + st * L::TILE + c * L::BOX, map, c * 64, start + j * KT, kv_row, bar(full0 + st));
                issued = j + 1;
            }
            if (!ok) {
                *abort_flag = 1;
                atomicOr(err, kDevErrTimeout);
                for (int t = max(0, issued - nst); t < issued; ++t)
                    mbar_wait(bar(full0 + t % nst), static_cast<uint32_t>(t / nst) & 1u, nullptr);
            }
        }
    } else if (warp == kWarpMma) {
        // ------------------------------------------------------------ tcgen05 issuer
        if (lane == 0) {
            constexpr uint32_t kIdQK = idesc_bf16_f32(KT, NH, false, false);
            constexpr uint32_t kIdPV = idesc_bf16_f32(D, NH, true, false);
            const uint32_t sQ = base + L::OFF_Q;
            auto issue_pv = [&](int jj) -> bool {
                if (!mbar_wait(bar(B_PFULL0 + (jj & 1)), static_cast<uint32_t>(jj >> 1) & 1u, abort_flag)) return false;
                if (!mbar_wait(bar(B_VFULL0 + jj % VST), static_cast<uint32_t>(jj / VST) & 1u, abort_flag)) return false;
                tc_fence_after();
                const uint32_t sV = base + L::OFF_V + (jj % VST) * L::TILE;
                const uint32_t sP = base + L::OFF_P + (jj & 1) * (2 * NH * 128);
#pragma unroll
                for (int kk = 0; kk < KT / 16; ++kk)
                    umma_ss(tmem + TM_O, smem_desc_sw128(sV + kk * 16 * 128, L::BOX, 1024),
                            smem_desc_sw128(sP + (kk >> 2) * NH * 128 + (kk & 3) * 32, 16, 1024), kIdPV,
                            (jj > 0 || kk > 0) ? 1u : 0u);
                umma_commit(bar(B_PVDONE));
                umma_commit(bar(B_VEMPTY0 + jj % VST));
                return true;
            };
            bool ok = mbar_wait(bar(B_QREADY), 0, abort_flag);
            if (ok) {
                tc_fence_after();
                for (int j = 0; j < ntiles; ++j) {
                    const int ks = j % KST;
                    if (!mbar_wait(bar(B_KFULL0 + ks), static_cast<uint32_t>(j / KST) & 1u, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sK = base + L::OFF_K + ks * L::TILE;
#pragma unroll
                    for (int kk = 0; kk < D / 16; ++kk) {
                        const uint32_t off = (kk >> 2) * L::BOX + (kk & 3) * 32;
                        umma_ss(tmem + (j & 1) * NH, smem_desc_sw128(sK + off, 16, 1024),
                                smem_desc_sw128(sQ + (kk >> 2) * NH * 128 + (kk & 3) * 32, 16, 1024), kIdQK,
                                kk > 0 ? 1u : 0u);
                    }
                    umma_commit(bar(B_SFULL0 + (j & 1)));
                    umma_commit(bar(B_KEMPTY0 + ks));  // K is consumed once S^T(j) completes
                    if (j >= 1 && !issue_pv(j - 1)) {
                        ok = false;
                        break;
                    }
                }
                if (ok) ok = issue_pv(ntiles - 1);
                if (ok) umma_commit(bar(B_OFULL));  // the epilogue's signal: every PV is complete
            }
            if (!ok) {
                *abort_flag = 1;
                atomicOr(err, kDevErrTimeout);
            }
            umma_commit(bar(B_DRAIN));
            mbar_wait(bar(B_DRAIN), 0, nullptr);
        }
    } else {
        // ------------------------------------------------------------ softmax / epilogue (one thread per key)
        const int t = tid;  // key row of a tile; output dimension in the epilogue
        const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
        uint8_t* qs = gb + L::OFF_Q;
        const float* cos_row = cos_tab + static_cast<size_t>(hist) * HALF;
        const float* sin_row = sin_tab + static_cast<size_t>(hist) * HALF;
        // Q^T: row h = rotated q of head h0 + h (bf16), zero rows past G; P^T buffers zeroed.
        // Each thread owns dimension t of every head: all loads first, then the math.
        const int tp = t < HALF ? t + HALF : t - HALF;  // RoPE partner dimension
        const float c_t = cos_row[t % HALF], s_t = sin_row[t % HALF];
        float qx[NH], qy[NH];
#pragma unroll
        for (int h = 0; h < NH; ++h) {
            const uint16_t* qrow = q + (static_cast<size_t>(b) * Hq + h0 + min(h, G - 1)) * D;
            qx[h] = bf16_at(qrow + t);
            qy[h] = bf16_at(qrow + tp);
        }
        float qhat[NH];
#pragma unroll
        for (int h = 0; h < NH; ++h) {
            const float r = t < HALF ? __fsub_rn(__fmul_rn(qx[h], c_t), __fmul_rn(qy[h], s_t))
                                     : __fadd_rn(__fmul_rn(qx[h], c_t), __fmul_rn(qy[h], s_t));
            const uint16_t qb = h < G ? to_bf16(r) : 0;
            qhat[h] = __uint_as_float(static_cast<uint32_t>(qb) << 16);
            *reinterpret_cast<uint16_t*>(qs + sw_elem(h, t, NH)) = qb;
        }
        for (int i = t; i < 2 * NH * 128 / 16; i += 128)
            reinterpret_cast<uint4*>(gb + L::OFF_P)[i] = make_uint4(0, 0, 0, 0);
        if (own_new) {
            // the new token: rotated k to slot hist, v to slot hist and to shared memory, and
            // its score q.k_new per head (float, reduced over the 128 dimensions)
            const uint16_t kr = to_bf16(rope_elem(k_new + static_cast<size_t>(kv_row) * D, t, cos_row, sin_row));
            const uint16_t vv = v_new[static_cast<size_t>(kv_row) * D + t];
            const size_t dst = (static_cast<size_t>(kv_row) * max_len + hist) * D + t;
            k_cache[dst] = kr;
            v_cache[dst] = vv;
            vnew_s[t] = vv;
            const float kf = __uint_as_float(static_cast<uint32_t>(kr) << 16);
#pragma unroll
            for (int h = 0; h < NH; ++h) {
                float v = qhat[h] * kf;
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, off);
                if (lane == 0) red[warp * NH + h] = v;
            }
        }
        fence_proxy_async_smem();
        named_sync_128();
        if (own_new && t < NH) news[t] = red[t] + red[NH + t] + red[2 * NH + t] + red[3 * NH + t];
        mbar_arrive(bar(B_QREADY));
        named_sync_128();

        float m_run[NH], l_run[NH];
#pragma unroll
        for (int h = 0; h < NH; ++h) {
            m_run[h] = -INFINITY;
            l_run[h] = 0.f;
        }
        bool ok = true;
        for (int j = 0; j < ntiles; ++j) {
            ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_SFULL0 + (j & 1)), static_cast<uint32_t>(j >> 1) & 1u, abort_flag));
            if (!ok) break;
            tc_fence_after();
            uint32_t r[NH];
            tmem_ld16(tmem + lane_base + (j & 1) * NH, r);
            tmem_wait_ld();
            const int key = start + j * KT + t;
            const bool valid = key < end;
            float sc[NH];
#pragma unroll
            for (int h = 0; h < NH; ++h) {
                const float raw_s = (key == hist) ? news[h] : __uint_as_float(r[h]);
                sc[h] = (valid && h < G) ? raw_s * scale_log2 : -INFINITY;
            }
            // per-head tile max: warp shuffles, then the four warps through shared memory
#pragma unroll
            for (int h = 0; h < NH; ++h) {
                if (h < G) {  // uniform: padded heads are skipped
                    float mx = sc[h];
#pragma unroll
                    for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, off));
                    if (lane == 0) red[warp * NH + h] = mx;
                }
            }
            named_sync_128();
            bool any_move = false;
            float alpha[NH];
#pragma unroll
            for (int h = 0; h < NH; ++h) {
                const float tmx = h < G ? fmaxf(fmaxf(red[h], red[NH + h]), fmaxf(red[2 * NH + h], red[3 * NH + h]))
                                        : -INFINITY;
                const float m_cand = fmaxf(m_run[h], tmx);
                const bool move = m_cand > m_run[h] + 8.f;  // lazy: P stays <= 2^8 otherwise
                alpha[h] = move ? fast_exp2(m_run[h] - m_cand) : 1.f;
                if (move) m_run[h] = m_cand;
                any_move |= move;
            }
            named_sync_128();  // every warp has read `red` before the next tile overwrites it
            if (j > 0 && any_move) {  // the same decision in every thread (same tile maxima)
                // O^T holds PV through tile j-1 once PV(j-1) completed (S(j) completed after PV(j-2)).
                ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_PVDONE), static_cast<uint32_t>(j - 1) & 1u, abort_flag));
                if (!ok) break;
                tc_fence_after();
                uint32_t o[NH];
                tmem_ld16(tmem + lane_base + TM_O, o);
                tmem_wait_ld();
#pragma unroll
                for (int h = 0; h < NH; ++h) o[h] = __float_as_uint(__uint_as_float(o[h]) * alpha[h]);
                tmem_st16(tmem + lane_base + TM_O, o);
                tmem_wait_st();
            }
            // P^T (bf16, row = head, column = key of the tile); padded heads stay zero
            uint8_t* pbuf = gb + L::OFF_P + (j & 1) * (2 * NH * 128);
#pragma unroll
            for (int h = 0; h < NH; ++h) {
                l_run[h] *= alpha[h];
                if (h < G) {
                    const float m_ref = m_run[h] == -INFINITY ? 0.f : m_run[h];
                    const float p = fast_exp2(sc[h] - m_ref);
                    l_run[h] += p;
                    *reinterpret_cast<uint16_t*>(pbuf + sw_elem(h, t, NH)) = to_bf16(p);
                }
            }
            // V rows past the split's end may hold anything: zero them; the new token's v.
            // (Only the tile that holds them: wait for its V to land first.)
            uint8_t* vtile = gb + L::OFF_V + (j % VST) * L::TILE;
            const bool patch = named_or_128(!valid || key == hist);
            if (patch) {
                ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_VFULL0 + j % VST), static_cast<uint32_t>(j / VST) & 1u, abort_flag));
                if (!ok) break;
            }
            if (!valid) {
#pragma unroll
                for (int c = 0; c < 16; ++c)
                    *reinterpret_cast<uint4*>(vtile + sw_elem(t, 8 * c, KT)) = make_uint4(0, 0, 0, 0);
            } else if (key == hist) {
#pragma unroll
                for (int c = 0; c < 16; ++c)
                    *reinterpret_cast<uint4*>(vtile + sw_elem(t, 8 * c, KT)) = reinterpret_cast<const uint4*>(vnew_s)[c];
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(bar(B_PFULL0 + (j & 1)));
        }
        // (PVDONE could be two phases behind here -- PV(ntiles-2) may still run -- so
        // the epilogue waits on its own barrier, committed once after the last PV.)
        if (ok) ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_OFULL), 0u, abort_flag));
        if (ok) {
            // row sums: every thread holds a partial over its keys
#pragma unroll
            for (int h = 0; h < NH; ++h) {
                if (h < G) {
                    float v = l_run[h];
#pragma unroll
                    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, off);
                    if (lane == 0) ls[warp * NH + h] = v;
                }
            }
            if (t == 0) {  // every thread holds the same running maxima
#pragma unroll
                for (int h = 0; h < NH; ++h) msh[h] = m_run[h];
            }
            tc_fence_after();
            uint32_t o[NH];
            tmem_ld16(tmem + lane_base + TM_O, o);  // thread t = output dimension d
            tmem_wait_ld();
            named_sync_128();
            for (int h = 0; h < G; ++h) {
                const size_t row = row0 + static_cast<size_t>(h) * nsplit;
                part_o[row * D + t] = __uint_as_float(o[h]);
                if (t == 0) {
                    part_ml[row * 2 + 0] = msh[h];
                    part_ml[row * 2 + 1] = ls[h] + ls[NH + h] + ls[2 * NH + h] + ls[3 * NH + h];
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

}  // namespace

cudaError_t configure_decode_tc() {
    return cudaFuncSetAttribute(decode_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, L::ALLOC);
}

int decode_tc_num_splits(const Shape& s, int num_sms) {
    const long items = static_cast<long>(s.batch) * s.n_kv_heads;
    const long slots = num_sms;  // one CTA per SM
    const long cap = std::max(1L, std::min<long>(256, (s.max_len + KT - 1) / KT));
    long best = 1;
    double best_eff = 0.0;
    for (long ns = 1; ns <= cap; ++ns) {
        const long ctas = items * ns;
        if (ctas < slots && ns < cap) continue;
        const double eff = static_cast<double>(ctas) / static_cast<double>(slots * ((ctas + slots - 1) / slots));
        if (eff >= 0.9) return static_cast<int>(ns);
        if (eff > best_eff) {
            best_eff = eff;
            best = ns;
        }
    }
    return static_cast<int>(best);
}

cudaError_t make_decode_tc_maps(PFN_encodeTiled encode, const Shape& s, const uint16_t* k_cache,
                                const uint16_t* v_cache, DecodeMaps* maps) {
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(s.max_len),
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

cudaError_t launch_decode_tc(const Shape& s, const DecodeMaps& maps, const uint16_t* q, const uint16_t* k_new,
                             const uint16_t* v_new, const int32_t* d_hist, uint16_t* k_cache, uint16_t* v_cache,
                             const float* cos_tab, const float* sin_tab, float* part_o, float* part_ml, int nsplit,
                             int* err, cudaStream_t st) {
    const float scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(D)));
    const dim3 grid(static_cast<unsigned>(nsplit), static_cast<unsigned>(s.n_kv_heads), static_cast<unsigned>(s.batch));
    decode_tc_kernel<<<grid, kThreads, L::ALLOC, st>>>(maps.k, maps.v, q, k_new, v_new, d_hist, k_cache, v_cache,
                                                       cos_tab, sin_tab, s.n_q_heads, s.n_kv_heads, s.max_len, nsplit,
                                                       scale_log2, part_o, part_ml, err);
    return cudaGetLastError();
}

}  // namespace attn

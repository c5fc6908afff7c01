// w4_gemm.cu -- W4BF16 weight GEMM for the prefill-side projections (tcgen05), and the
// RMSNorm pre-pass of the block's chunk.
//
// A prefill chunk of T tokens turns the block's projections (Listing 1: q/k/v_proj, o_proj)
// into GEMMs, Y[T, N] = X[T, K] . W[N, K]^T, with W in the W4BF16 tile stream of
// attn_w4bf16_gemv (Section 5.1).  Reading: each weight is decoded once into the tensor
// cores' operand type, W_bf16 = bf16((q - z) * s), and the products accumulate in f32.
//
// Computed transposed, Y^T = W . X^T, so that the decoded weights are the MMA's A operand,
// which tcgen05 reads from tensor memory: each decode thread owns one feature row (one TMEM
// lane), decodes its 128 inputs of a group from the record in shared memory and stores the
// 64 bf16 pairs straight into TMEM -- no shared-memory round trip, no swizzle arithmetic, a
// row's scale and zero point read once per group.  X^T is the B operand, K-major from
// shared memory exactly as TMA lays out a 128-token x 64-input box of X.
//
// Persistent CTAs walk output tiles of 256 features (two M = 128 halves) x 128 tokens
// (the MMA's N), token tiles fastest.  448 threads:
//   warp 0, one lane   producer: per 128-input group one X tile (two 2-D TMA boxes, 128-byte
//                      swizzle; tokens past T read as zeros) and the 16 weight records of the
//                      tile's 256 features into a kStages ring: their codes as one 4-D TMA box
//                      with 64-byte swizzle (row r's 16-byte chunk c lands at chunk
//                      c ^ ((r >> 1) & 3), so the eight rows that a quarter-warp of decode
//                      threads reads at once sit in eight different bank groups), their
//                      scales and zero points as one 3-D box;
//   warp 1, one lane   tcgen05 issuer: per group and half, 8 MMAs 128 x 128 x 16 from the
//                      half's A buffer in TMEM and the X stage, into the half's accumulator;
//   warps 2-9          decode (warps 2-5 the first half's 128 features, 6-9 the second),
//                      into two A buffers per half (double-buffered across groups);
//   warps 10-13        epilogue: each thread one feature of each half, 128 tokens from TMEM,
//                      optionally the residual added in float, rounded to bf16, written
//                      to y or, split by feature, to y / y1 / y2.  Each half's accumulator is
//                      handed back as soon as it is read, so the next tile's MMAs of that
//                      half start while the epilogue finishes the other half.
// TMEM (512 columns): A buffers (half h, buffer b) at 64 (2h + b), accumulators at 256 + 128 h.
// Every wait is bounded (ATTN_DEVERR_TIMEOUT in *err, then the CTA drains and exits).
#include <cuda_bf16.h>

#include <algorithm>
#include <cstdint>
#include <map>
#include <mutex>

#include "internal.h"
#include "sm100_ptx.cuh"

namespace attn {
namespace {

constexpr int kThreads = 448;
constexpr int kWarpTma = 0, kWarpMma = 1, kWarpDec0 = 2, kWarpEpi0 = 10;
constexpr int kBT = 128;                    // tokens per tile (MMA N)
constexpr int kBF = 256;                    // features per tile (two MMA M = 128 halves)
constexpr int kStages = 4;
constexpr int kChunk = 128 * 128;           // 128 rows x 64 bf16 (128 bytes), swizzled
constexpr int kXStage = 2 * kChunk;         // X tile: 128 tokens x 128 inputs
constexpr int kRecBytes = 1072;             // one weight record: 16 rows x 128 inputs
constexpr int kRecs = kBF / 16;             // records per stage
constexpr int kWcStage = kRecs * 16 * 64;   // their codes: 256 rows x 64 bytes, 64-byte swizzle
constexpr int kWsStage = kRecs * 48;        // their scales and zero points: 16 x 48 bytes
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kTmA = 0, kTmAcc = 256;
constexpr uint64_t kWaitNs = 1000000000ull;

struct L {
    static constexpr int OFF_X = 0;
    static constexpr int OFF_WC = OFF_X + kStages * kXStage;
    static constexpr int OFF_WS = OFF_WC + kStages * kWcStage;
    static constexpr int OFF_BAR = OFF_WS + kStages * kWsStage;
    static constexpr int NBAR = 2 * kStages + 2 + 2 + 1 + 2 + 1;
    static constexpr int OFF_TMEM = OFF_BAR + 8 * NBAR;
    static constexpr int OFF_ABORT = OFF_TMEM + 16;
    static constexpr int BYTES = OFF_ABORT + 16;
    static constexpr int ALLOC = BYTES + 1024;  // the dynamic base is aligned up to 1024 in the kernel
};
static_assert(L::ALLOC <= 232448, "shared memory");
enum Bar {
    B_FULL0 = 0, B_EMPTY0 = kStages, B_AFULL0 = 2 * kStages, B_AEMPTY0 = B_AFULL0 + 2, B_ACCFULL = B_AEMPTY0 + 2,
    B_ACCEMPTY0 = B_ACCFULL + 1, B_DRAIN = B_ACCEMPTY0 + 2
};

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int c0, int c1, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
        : "memory");
}

__device__ __forceinline__ uint32_t bf16x2_sub(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("sub.rn.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}

__device__ __forceinline__ uint32_t bf16x2_mul(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}

// (128 + q) for the two codes of pair j of a word, as one three-input logic op.
__device__ __forceinline__ uint32_t code_pair(uint32_t w, int j, uint32_t mask, uint32_t magic) {
    uint32_t r;
    asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(r) : "r"(w >> (4 * j)), "r"(mask), "r"(magic));
    return r;
}

// Work units: units [0, n_full) are whole output tiles (tile = unit); the tiles after them
// are cut into their two 128-feature halves, one unit each, so that the last round of the
// persistent CTAs ends more evenly.  Returns the tile and the mask of its halves (a half
// past N is never on).
__device__ __forceinline__ int unit_tile(int u, int n_full, int n_tt, int N, int& hmask) {
    int tile = u;
    hmask = 3;
    if (u >= n_full) {
        tile = n_full + ((u - n_full) >> 1);
        hmask = 1 << ((u - n_full) & 1);
    }
    if ((tile / n_tt) * kBF + 128 >= N) hmask &= 1;
    return tile;
}

__global__ void __launch_bounds__(kThreads, 1) w4_gemm_kernel(const __grid_constant__ CUtensorMap map_x,
                                                              const __grid_constant__ CUtensorMap map_wc,
                                                              const __grid_constant__ CUtensorMap map_ws, int n_full, int n_units,
                                                              int T, int N, int K,
                                                              uint16_t* __restrict__ y, int* err, const W4GemmEpi epi) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* gb = smem_raw + (base - raw);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(gb + L::OFF_ABORT);
    auto bar = [&](int i) -> uint32_t { return base + L::OFF_BAR + 8u * static_cast<uint32_t>(i); };
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int ngroup = K / 128;
    const int n_tt = (T + kBT - 1) / kBT;

    if (tid == 0) {
        *abort_flag = 0;
        for (int s = 0; s < kStages; ++s) {
            mbar_init(bar(B_FULL0 + s), 1);
            mbar_init(bar(B_EMPTY0 + s), 1 + 8);  // the MMA commit and the eight decode warps
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(bar(B_AFULL0 + b), 8);
            mbar_init(bar(B_AEMPTY0 + b), 1);
            mbar_init(bar(B_ACCEMPTY0 + b), 4);  // per half: the four epilogue warps
        }
        mbar_init(bar(B_ACCFULL), 1);
        mbar_init(bar(B_DRAIN), 1);
        fence_mbar_init();
        tma_prefetch_desc(&map_x);
        tma_prefetch_desc(&map_wc);
        tma_prefetch_desc(&map_ws);
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
        if (lane == 0) {
            uint32_t gs = 0;  // groups issued
            bool ok = true;
            for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
                int hmask;
                const int tile = unit_tile(u, n_full, n_tt, N, hmask);
                const int ft = tile / n_tt, tt = tile - ft * n_tt;
                const int f0 = ft * kBF, t0 = tt * kBT;
                for (int G = 0; G < ngroup; ++G, ++gs) {
                    const int s = static_cast<int>(gs % kStages);
                    if (gs >= kStages &&
                        !mbar_wait(bar(B_EMPTY0 + s), (gs / kStages - 1u) & 1u, abort_flag, kWaitNs)) {
                        ok = false;
                        break;
                    }
                    // (row tiles past N read as zeros; every box counts its full size)
                    mbar_arrive_expect_tx(bar(B_FULL0 + s), kXStage + kWcStage + kWsStage);
                    for (int c = 0; c < 2; ++c)
                        tma_load_2d(base + L::OFF_X + s * kXStage + c * kChunk, &map_x, G * 128 + c * 64, t0,
                                    bar(B_FULL0 + s));
                    tma_load_4d(base + L::OFF_WC + s * kWcStage, &map_wc, 0, 0, G, f0 / 16, bar(B_FULL0 + s));
                    tma_load_3d(base + L::OFF_WS + s * kWsStage, &map_ws, 0, G, f0 / 16, bar(B_FULL0 + s));
                }
            }
            if (!ok) {
                *abort_flag = 1;
                atomicOr(err, kDevErrTimeout);
            }
            // every copy issued must land before the CTA may exit
            for (uint32_t g = gs > kStages ? gs - kStages : 0; g < gs; ++g)
                mbar_wait(bar(B_FULL0 + g % kStages), (g / kStages) & 1u, nullptr, kWaitNs);
        }
    } else if (warp == kWarpMma) {
        if (lane == 0) {
            constexpr uint32_t kId = idesc_bf16_f32(128, kBT, false, false);
            constexpr uint32_t kHi = desc_hi_sw128(1024);
            const uint32_t x_lo0 = desc_lo_sw128(base + L::OFF_X, 16);
            uint32_t gs = 0;
            int tiles_done = 0;
            bool ok = true;
            for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x, ++tiles_done) {
                int hmask;
                unit_tile(u, n_full, n_tt, N, hmask);
                for (int G = 0; G < ngroup; ++G, ++gs) {
                    const int s = static_cast<int>(gs % kStages), b = static_cast<int>(gs & 1u);
                    if (!mbar_wait(bar(B_FULL0 + s), (gs / kStages) & 1u, abort_flag, kWaitNs) ||
                        !mbar_wait(bar(B_AFULL0 + b), (gs >> 1) & 1u, abort_flag, kWaitNs)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t xa = x_lo0 + ((s * kXStage) >> 4);
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        if (!((hmask >> h) & 1)) continue;
                        // the accumulator of half h is free once the epilogue read the previous tile's
                        if (G == 0 && tiles_done > 0 &&
                            !mbar_wait(bar(B_ACCEMPTY0 + h), static_cast<uint32_t>(tiles_done - 1) & 1u, abort_flag,
                                       kWaitNs)) {
                            ok = false;
                            break;
                        }
                        if (G == 0) tc_fence_after();
                        const uint32_t a_col = tmem + kTmA + 64u * (2 * h + b), d_col = tmem + kTmAcc + 128u * h;
#pragma unroll
                        for (int kk = 0; kk < 8; ++kk) {
                            const uint32_t c = ((kk >> 2) * kChunk + (kk & 3) * 32) >> 4;
                            umma_ts_w(d_col, a_col + 8u * kk, xa + c, kHi, kId, (G > 0 || kk > 0) ? 1u : 0u);
                        }
                    }
                    if (!ok) break;
                    umma_commit(bar(B_EMPTY0 + s));
                    umma_commit(bar(B_AEMPTY0 + b));
                }
                if (!ok) break;
                umma_commit(bar(B_ACCFULL));  // the tile's products are complete
            }
            if (!ok) {
                *abort_flag = 1;
                atomicOr(err, kDevErrTimeout);
            }
            umma_commit(bar(B_DRAIN));  // also after an abort: the MMAs issued so far complete on it
            mbar_wait(bar(B_DRAIN), 0u, nullptr, kWaitNs);
        }
    } else if (warp < kWarpEpi0) {
        // ------------------------------------------------ decode: one feature row per thread
        const int h = (warp - kWarpDec0) >> 2;        // half of the tile
        const int q = warp & 3;                       // TMEM lane quadrant of this warp
        const int fl = q * 32 + lane;                 // feature within the half (= TMEM lane)
        const int rrow = 128 * h + fl;                // feature within the tile
        const uint32_t magic = 0x43004300u, mask = 0x000F000Fu;
        uint32_t gs = 0;
        bool ok = true;
        for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
            int hmask;
            const int tile = unit_tile(u, n_full, n_tt, N, hmask);
            const int ft = tile / n_tt;
            const int f0 = ft * kBF;
            const bool have = f0 + rrow < N;   // this feature exists (N is a multiple of 16)
            const bool half_on = (hmask >> h) & 1;
            for (int G = 0; G < ngroup; ++G, ++gs) {
                const int s = static_cast<int>(gs % kStages), b = static_cast<int>(gs & 1u);
                bool w_ok = mbar_wait(bar(B_FULL0 + s), (gs / kStages) & 1u, abort_flag, kWaitNs);
                if (w_ok && gs >= 2)
                    w_ok = mbar_wait(bar(B_AEMPTY0 + b), ((gs >> 1) - 1u) & 1u, abort_flag, kWaitNs);
                ok = __all_sync(0xFFFFFFFFu, w_ok);
                if (!ok) break;
                if (half_on) {
                    uint32_t wv[16];
                    uint32_t zp = 0x43004300u, sp = 0u;
                    if (have) {
                        const uint8_t* row = gb + L::OFF_WC + s * kWcStage + rrow * 64;
                        const uint8_t* rec = gb + L::OFF_WS + s * kWsStage + (rrow >> 4) * 48;
                        const int sw = (rrow >> 1) & 3;  // the 64-byte swizzle of this row
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const uint4 u = *reinterpret_cast<const uint4*>(row + 16 * (i ^ sw));
                            wv[4 * i] = u.x;
                            wv[4 * i + 1] = u.y;
                            wv[4 * i + 2] = u.z;
                            wv[4 * i + 3] = u.w;
                        }
                        const uint32_t sc = *reinterpret_cast<const uint16_t*>(rec + (rrow & 15) * 2);
                        const uint32_t z = rec[32 + (rrow & 15)];
                        zp = (0x4300u + z) * 0x00010001u;  // (128 + z) in both halves
                        sp = sc * 0x00010001u;
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i) wv[i] = 0u;
                    }
                    // word i: inputs 8 i .. 8 i + 7; pair p: inputs 8 i + 2 p, + 1 -> TMEM column 4 i + p
                    const uint32_t a_col = tmem + (static_cast<uint32_t>(q * 32) << 16) + kTmA + 64u * (2 * h + b);
#pragma unroll
                    for (int half = 0; half < 2; ++half) {
                        uint32_t o[32];
#pragma unroll
                        for (int i = 0; i < 8; ++i)
#pragma unroll
                            for (int p = 0; p < 4; ++p)
                                o[4 * i + p] = bf16x2_mul(bf16x2_sub(code_pair(wv[8 * half + i], p, mask, magic), zp), sp);
                        tmem_st32(a_col + 32u * half, o);
                    }
                    tmem_wait_st();
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(bar(B_AFULL0 + b));
                    mbar_arrive(bar(B_EMPTY0 + s));
                }
            }
        }
        if (!ok && lane == 0) {
            *abort_flag = 1;
            atomicOr(err, kDevErrTimeout);
        }
    } else {
        // ------------------------------------------------ epilogue: one feature of each half per thread
        const int q = warp & 3;
        const int fl = q * 32 + lane;
        int tiles_done = 0;
        bool ok = true;
        for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x, ++tiles_done) {
            int hmask;
            const int tile = unit_tile(u, n_full, n_tt, N, hmask);
            const int ft = tile / n_tt, tt = tile - ft * n_tt;
            const int f0 = ft * kBF, t0 = tt * kBT;
            ok = __all_sync(0xFFFFFFFFu,
                            mbar_wait(bar(B_ACCFULL), static_cast<uint32_t>(tiles_done) & 1u, abort_flag, kWaitNs));
            if (!ok) break;
            tc_fence_after();
#pragma unroll 1
            for (int h = 0; h < 2; ++h) {
                const int n = f0 + 128 * h + fl;
                if ((hmask >> h) & 1) {
                    // destination of feature n: y, or a part of the split output
                    uint16_t* dst = y;
                    int stride = epi.n0, cc = n;
                    if (n >= epi.n1) {
                        dst = epi.y2;
                        stride = N - epi.n1;
                        cc = n - epi.n1;
                    } else if (n >= epi.n0) {
                        dst = epi.y1;
                        stride = epi.n1 - epi.n0;
                        cc = n - epi.n0;
                    }
                    const uint32_t d_col = tmem + (static_cast<uint32_t>(q * 32) << 16) + kTmAcc + 128u * h;
#pragma unroll 1
                    for (int c = 0; c < kBT / 32; ++c) {
                        const int tb = t0 + 32 * c;
                        // the residual of these 32 tokens, all loads in flight at once (h may be
                        // x: each element is read here before this thread writes it below)
                        uint32_t res[32];
                        if (epi.residual != nullptr && n < N) {
#pragma unroll
                            for (int e = 0; e < 32; ++e)
                                res[e] = tb + e < T ? static_cast<uint32_t>(
                                                          epi.residual[static_cast<size_t>(tb + e) * N + n])
                                                    : 0u;
                        }
                        uint32_t r[32];
                        tmem_ld32(d_col + 32u * c, r);
                        tmem_wait_ld();
                        if (c == kBT / 32 - 1) {
                            // this half's accumulator is read: the next tile's MMAs may overwrite it
                            tc_fence_before();
                            __syncwarp();
                            if (lane == 0) mbar_arrive(bar(B_ACCEMPTY0 + h));
                        }
                        if (n < N) {
#pragma unroll
                            for (int e = 0; e < 32; ++e) {
                                const int t = tb + e;
                                if (t < T) {
                                    float v = __uint_as_float(r[e]);
                                    if (epi.residual != nullptr) v += __uint_as_float(res[e] << 16);
                                    dst[static_cast<size_t>(t) * stride + cc] = __bfloat16_as_ushort(__float2bfloat16_rn(v));
                                }
                            }
                        }
                    }
                } else {
                    __syncwarp();
                    if (lane == 0) mbar_arrive(bar(B_ACCEMPTY0 + h));  // an absent half is free at once
                }
            }
        }
        if (!ok && lane == 0) {
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

// RMSNorm rows: one warp per row of K values.  Pass 1: per-lane float sums of squares over
// 16-byte chunks in order, then a shuffle tree (a fixed order); pass 2 re-reads the row
// (L1/L2) and writes bf16((x * r) * gamma).
__global__ void __launch_bounds__(256) rmsnorm_rows_kernel(const uint16_t* __restrict__ x,
                                                           const uint16_t* __restrict__ gamma, float eps, int T, int K,
                                                           uint16_t* __restrict__ xn) {
    const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (row >= T) return;
    const uint4* xr = reinterpret_cast<const uint4*>(x + static_cast<size_t>(row) * K);
    const int nchunk = K / 8;
    float ss = 0.f;
    for (int i = lane; i < nchunk; i += 32) {
        const uint4 v = xr[i];
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float a = __uint_as_float(w[e] << 16), b = __uint_as_float(w[e] & 0xFFFF0000u);
            ss = fmaf(a, a, ss);
            ss = fmaf(b, b, ss);
        }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, off);
    const float r = 1.0f / sqrtf(ss / static_cast<float>(K) + eps);
    const uint4* gr = reinterpret_cast<const uint4*>(gamma);
    uint4* out = reinterpret_cast<uint4*>(xn + static_cast<size_t>(row) * K);
    for (int i = lane; i < nchunk; i += 32) {
        const uint4 v = xr[i], g = gr[i];
        const uint32_t w[4] = {v.x, v.y, v.z, v.w}, gw[4] = {g.x, g.y, g.z, g.w};
        uint32_t o[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float lo = (__uint_as_float(w[e] << 16) * r) * __uint_as_float(gw[e] << 16);
            const float hi = (__uint_as_float(w[e] & 0xFFFF0000u) * r) * __uint_as_float(gw[e] & 0xFFFF0000u);
            o[e] = pack_bf16x2(lo, hi);
        }
        out[i] = make_uint4(o[0], o[1], o[2], o[3]);
    }
}

std::mutex g_mutex;
PFN_encodeTiled g_encode = nullptr;
constexpr int kMaxDevices = 64;
bool g_configured[kMaxDevices] = {};

// How many of the last tiles to cut into halves: the split that minimises the busiest
// CTA's work as the kernel deals units (unit u to CTA u mod grid), a half counted as 0.6
// of a tile (the x tile and the MMA issue do not halve).  Cached per (tiles, SMs).
int tail_halves(long long n_tiles, int sms) {
    static std::mutex mu;
    static std::map<std::pair<long long, int>, int> cache;
    {
        std::lock_guard<std::mutex> lock(mu);
        const auto it = cache.find({n_tiles, sms});
        if (it != cache.end()) return it->second;
    }
    int best_x = 0;
    double best = 1e300;
    for (int xs = 0; xs <= std::min<long long>(n_tiles, 3LL * sms); ++xs) {
        const long long units = n_tiles + xs;
        const long long g = std::min<long long>(units, sms);
        const long long n_full = n_tiles - xs;
        // CTA c gets full units c, c+g, ... below n_full and half units from n_full on
        double worst = 0.0;
        for (long long c = 0; c < std::min<long long>(g, 2LL * sms); ++c) {
            const long long nf = c < n_full ? (n_full - 1 - c) / g + 1 : 0;
            const long long first_h = c >= n_full ? c : c + nf * g;  // its first unit past n_full
            const long long nh = first_h < units ? (units - 1 - first_h) / g + 1 : 0;
            worst = std::max(worst, static_cast<double>(nf) + 0.6 * static_cast<double>(nh));
        }
        if (worst < best - 1e-9) {
            best = worst;
            best_x = xs;
        }
    }
    std::lock_guard<std::mutex> lock(mu);
    cache[{n_tiles, sms}] = best_x;
    return best_x;
}

}  // namespace

cudaError_t launch_rmsnorm_rows(const uint16_t* x, const uint16_t* gamma, float eps, int T, int K, uint16_t* xn,
                                cudaStream_t st) {
    rmsnorm_rows_kernel<<<(T + 7) / 8, 256, 0, st>>>(x, gamma, eps, T, K, xn);
    return cudaGetLastError();
}

cudaError_t launch_w4_gemm(const uint8_t* tiles, const uint16_t* x, int T, int N, int K, uint16_t* y, int* err,
                           cudaStream_t st, const W4GemmEpi* epi_in) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    {
        std::lock_guard<std::mutex> lock(g_mutex);
        if (g_encode == nullptr) {
            cudaDriverEntryPointQueryResult qres;
            void* fn = nullptr;
            e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &qres);
            if (e != cudaSuccess) return e;
            if (qres != cudaDriverEntryPointSuccess || fn == nullptr) return cudaErrorNotSupported;
            g_encode = reinterpret_cast<PFN_encodeTiled>(fn);
        }
        if (!g_configured[dev]) {
            e = cudaFuncSetAttribute(w4_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, L::ALLOC);
            if (e != cudaSuccess) return e;
            g_configured[dev] = true;
        }
    }
    CUtensorMap map, map_wc, map_ws;
    {
        const cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(T)};
        const cuuint64_t strides[1] = {static_cast<cuuint64_t>(K) * 2};
        const cuuint32_t box[2] = {64, static_cast<cuuint32_t>(kBT)};
        const cuuint32_t estr[2] = {1, 1};
        const CUresult r = g_encode(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t*>(x), dims, strides,
                                    box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    }
    // The tile stream as two views: record (row tile t, group g) at (t * K/128 + g) * 1072 bytes.
    //   codes  [row tile][group][16 rows][64 bytes]  (16-bit elements, box 32 x 16 x 1 x 16)
    //   scales and zero points [row tile][group][48 bytes] from byte 1024 of each record
    const cuuint64_t ng = static_cast<cuuint64_t>(K / 128), nt = static_cast<cuuint64_t>(N / 16);
    {
        const cuuint64_t dims[4] = {32, 16, ng, nt};
        const cuuint64_t strides[3] = {64, kRecBytes, kRecBytes * ng};
        const cuuint32_t box[4] = {32, 16, 1, static_cast<cuuint32_t>(kRecs)};
        const cuuint32_t estr[4] = {1, 1, 1, 1};
        const CUresult r = g_encode(&map_wc, CU_TENSOR_MAP_DATA_TYPE_UINT16, 4, const_cast<uint8_t*>(tiles), dims,
                                    strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
                                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    }
    {
        const cuuint64_t dims[3] = {24, ng, nt};
        const cuuint64_t strides[2] = {kRecBytes, kRecBytes * ng};
        const cuuint32_t box[3] = {24, 1, static_cast<cuuint32_t>(kRecs)};
        const cuuint32_t estr[3] = {1, 1, 1};
        const CUresult r = g_encode(&map_ws, CU_TENSOR_MAP_DATA_TYPE_UINT16, 3, const_cast<uint8_t*>(tiles) + 1024,
                                    dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                                    CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    }
    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const long long n_tiles = static_cast<long long>((T + kBT - 1) / kBT) * ((N + kBF - 1) / kBF);
    if (n_tiles > (1LL << 29)) return cudaErrorInvalidValue;
    const int best_x = tail_halves(n_tiles, sms);
    const int n_full = static_cast<int>(n_tiles - best_x), n_units = static_cast<int>(n_tiles + best_x);
    const unsigned grid = static_cast<unsigned>(std::min<long long>(n_units, sms));
    W4GemmEpi epi = {N, N, nullptr, nullptr, nullptr};
    if (epi_in != nullptr) epi = *epi_in;
    w4_gemm_kernel<<<grid, kThreads, L::ALLOC, st>>>(map, map_wc, map_ws, n_full, n_units, T, N, K, y, err, epi);
    return cudaGetLastError();
}

}  // namespace attn

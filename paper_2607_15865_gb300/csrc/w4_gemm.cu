// w4_gemm.cu -- W4BF16 weight GEMM for the prefill-side projections (tcgen05).
//
// A prefill chunk of T tokens turns the block's projections (Listing 1: q/k/v_proj, o_proj)
// into GEMMs, Y[T, N] = X[T, K] . W[N, K]^T, with W in the W4BF16 tile stream of
// attn_w4bf16_gemv (Section 5.1).  Reading: each weight is decoded once into the tensor
// cores' operand type, W_bf16 = bf16((q - z) * s), and the products accumulate in f32.
//
// One CTA computes a 128-token x 128-feature tile of Y, walking K one 128-input group at a
// time through a kStages ring:
//   * warp 0, one lane: the x tile of the group by two 2-D TMA loads (128 tokens x 64 inputs,
//     128-byte swizzle; rows past T read as zeros) and the 8 weight records of the group's
//     128 features by 8 bulk copies, all completing on the stage's mbarrier;
//   * warps 2..5: decode the records into the B operand, double-buffered in shared memory
//     in the same swizzled K-major layout the TMA gives x: per code word one shift and one
//     lop3 per pair of codes give (128 + q) bf16 pairs, a bf16x2 subtraction of (128 + z)
//     leaves q - z exactly, a bf16x2 multiply by s rounds each weight once; one 16-byte store
//     per word;
//   * warp 1, one lane: 8 tcgen05.mma (kind::f16, 128 x 128 x 16) per group into one TMEM
//     accumulator, committing the x stage and the B buffer back to their producers;
//   * warps 2..5 again: the epilogue, 32 TMEM lanes (tokens) each: optionally the residual
//     added in float, rounded to bf16, the columns optionally split three ways (q, k, v).
// rmsnorm_rows_kernel is the block's input_layernorm for a chunk: one factor per token,
// so it runs as a pre-pass over the chunk before the stacked QKV GEMM.
// Every wait is bounded (ATTN_DEVERR_TIMEOUT in *err, then the CTA drains and exits).
#include <cuda_bf16.h>

#include <cstdint>
#include <mutex>

#include "internal.h"
#include "sm100_ptx.cuh"

namespace attn {
namespace {

constexpr int kThreads = 192;
constexpr int kWarpTma = 0, kWarpMma = 1;  // warps 2..5 decode and run the epilogue
constexpr int kBM = 128, kBN = 128;
constexpr int kStages = 3;
constexpr int kChunk = 128 * 128;          // 128 rows x 64 bf16 (128 bytes), swizzled
constexpr int kXStage = 2 * kChunk;        // x tile: 128 tokens x 128 inputs
constexpr int kRecBytes = 1072;            // one weight record: 16 rows x 128 inputs
constexpr int kRecs = kBN / 16;            // records per stage
constexpr int kWStage = kRecs * kRecBytes;
constexpr int kBTile = 2 * kChunk;         // decoded weights: 128 features x 128 inputs
constexpr uint32_t kTmemCols = 128;
constexpr uint64_t kWaitNs = 1000000000ull;

struct L {
    static constexpr int OFF_X = 0;
    static constexpr int OFF_W = OFF_X + kStages * kXStage;
    static constexpr int OFF_B = ((OFF_W + kStages * kWStage + 1023) / 1024) * 1024;
    static constexpr int OFF_BAR = OFF_B + 2 * kBTile;
    static constexpr int NBAR = 2 * kStages + 4 + 1;  // FULL, EMPTY, BFULL x2, BEMPTY x2, ACC
    static constexpr int OFF_TMEM = OFF_BAR + 8 * NBAR;
    static constexpr int OFF_ABORT = OFF_TMEM + 16;
    static constexpr int BYTES = OFF_ABORT + 16;
    static constexpr int ALLOC = BYTES + 1024;  // the dynamic base is aligned up to 1024 in the kernel
};
static_assert(L::ALLOC <= 232448, "shared memory");
enum Bar { B_FULL0 = 0, B_EMPTY0 = kStages, B_BFULL0 = 2 * kStages, B_BEMPTY0 = 2 * kStages + 2, B_ACC = 2 * kStages + 4 };

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int c0, int c1, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
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

__global__ void __launch_bounds__(kThreads, 1) w4_gemm_kernel(const __grid_constant__ CUtensorMap map_x,
                                                              const uint8_t* __restrict__ tiles, int T, int N, int K,
                                                              uint16_t* __restrict__ y, int* err, const W4GemmEpi epi) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* gb = smem_raw + (base - raw);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(gb + L::OFF_ABORT);
    auto bar = [&](int i) -> uint32_t { return base + L::OFF_BAR + 8u * static_cast<uint32_t>(i); };
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n0 = blockIdx.x * kBN, m0 = blockIdx.y * kBM;
    const int ngroup = K / 128;
    const int nrec = min(kRecs, (N - n0 + 15) / 16);  // records of this feature tile

    if (tid == 0) {
        *abort_flag = 0;
        for (int s = 0; s < kStages; ++s) {
            mbar_init(bar(B_FULL0 + s), 1);
            mbar_init(bar(B_EMPTY0 + s), 1 + 4);  // the MMA commit and the four decode warps
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(bar(B_BFULL0 + b), 4);
            mbar_init(bar(B_BEMPTY0 + b), 1);
        }
        mbar_init(bar(B_ACC), 1);
        fence_mbar_init();
        tma_prefetch_desc(&map_x);
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
            int issued = 0;
            bool ok = true;
            for (int G = 0; G < ngroup; ++G) {
                const int s = G % kStages;
                if (G >= kStages &&
                    !mbar_wait(bar(B_EMPTY0 + s), static_cast<uint32_t>(G / kStages - 1) & 1u, abort_flag, kWaitNs)) {
                    ok = false;
                    break;
                }
                mbar_arrive_expect_tx(bar(B_FULL0 + s), kXStage + nrec * kRecBytes);
                for (int c = 0; c < 2; ++c)
                    tma_load_2d(base + L::OFF_X + s * kXStage + c * kChunk, &map_x, G * 128 + c * 64, m0,
                                bar(B_FULL0 + s));
                for (int r = 0; r < nrec; ++r) {
                    const size_t rec = static_cast<size_t>(n0 / 16 + r) * ngroup + G;
                    bulk_load(base + L::OFF_W + s * kWStage + r * kRecBytes, tiles + rec * kRecBytes, kRecBytes,
                              bar(B_FULL0 + s));
                }
                issued = G + 1;
            }
            if (!ok) {
                *abort_flag = 1;
                atomicOr(err, kDevErrTimeout);
            }
            // every copy issued must land before the CTA may exit
            for (int G = issued > kStages ? issued - kStages : 0; G < issued; ++G)
                mbar_wait(bar(B_FULL0 + G % kStages), static_cast<uint32_t>(G / kStages) & 1u, nullptr, kWaitNs);
        }
    } else if (warp == kWarpMma) {
        if (lane == 0) {
            constexpr uint32_t kId = idesc_bf16_f32(kBM, kBN, false, false);
            constexpr uint32_t kHi = desc_hi_sw128(1024);
            const uint32_t x_lo0 = desc_lo_sw128(base + L::OFF_X, 16);
            const uint32_t b_lo0 = desc_lo_sw128(base + L::OFF_B, 16);
            bool ok = true;
            for (int G = 0; G < ngroup; ++G) {
                const int s = G % kStages, b = G & 1;
                if (!mbar_wait(bar(B_FULL0 + s), static_cast<uint32_t>(G / kStages) & 1u, abort_flag, kWaitNs) ||
                    !mbar_wait(bar(B_BFULL0 + b), static_cast<uint32_t>(G >> 1) & 1u, abort_flag, kWaitNs)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t xa = x_lo0 + ((s * kXStage) >> 4), bb = b_lo0 + ((b * kBTile) >> 4);
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    const uint32_t c = ((kk >> 2) * kChunk + (kk & 3) * 32) >> 4;
                    umma_ss_w(tmem, xa + c, kHi, bb + c, kHi, kId, (G > 0 || kk > 0) ? 1u : 0u);
                }
                umma_commit(bar(B_EMPTY0 + s));
                umma_commit(bar(B_BEMPTY0 + b));
            }
            if (!ok) {
                *abort_flag = 1;
                atomicOr(err, kDevErrTimeout);
            }
            umma_commit(bar(B_ACC));  // also after an abort: the MMAs issued so far complete on it
            mbar_wait(bar(B_ACC), 0u, nullptr, kWaitNs);
        }
    } else {
        // ------------------------------------------------ decode warps, then the epilogue
        const int dt = tid - 64;  // 0..127
        const uint32_t magic = 0x43004300u, mask = 0x000F000Fu;
        bool ok = true;
        for (int G = 0; G < ngroup && ok; ++G) {
            const int s = G % kStages, b = G & 1;
            ok = mbar_wait(bar(B_FULL0 + s), static_cast<uint32_t>(G / kStages) & 1u, abort_flag, kWaitNs);
            if (ok && G >= 2)
                ok = mbar_wait(bar(B_BEMPTY0 + b), static_cast<uint32_t>((G >> 1) - 1) & 1u, abort_flag, kWaitNs);
            ok = __all_sync(0xFFFFFFFFu, ok);
            if (!ok) break;
            const uint8_t* ws = gb + L::OFF_W + s * kWStage;
            uint8_t* bt = gb + L::OFF_B + b * kBTile;
#pragma unroll 4
            for (int j = 0; j < 16; ++j) {
                const int wi = dt + 128 * j;
                const int n = wi >> 4, i16 = wi & 15;  // feature row, word of the group
                const int r = n >> 4, rr = n & 15;
                uint4 v = make_uint4(0u, 0u, 0u, 0u);
                if (r < nrec) {
                    const uint8_t* rec = ws + r * kRecBytes;
                    const uint32_t w = *reinterpret_cast<const uint32_t*>(rec + rr * 64 + i16 * 4);
                    const uint32_t sc = *reinterpret_cast<const uint16_t*>(rec + 1024 + rr * 2);
                    const uint32_t z = rec[1056 + rr];
                    const uint32_t zp = (0x4300u + z) * 0x00010001u;  // (128 + z) in both halves
                    const uint32_t sp = sc * 0x00010001u;
                    v.x = bf16x2_mul(bf16x2_sub(code_pair(w, 0, mask, magic), zp), sp);
                    v.y = bf16x2_mul(bf16x2_sub(code_pair(w, 1, mask, magic), zp), sp);
                    v.z = bf16x2_mul(bf16x2_sub(code_pair(w, 2, mask, magic), zp), sp);
                    v.w = bf16x2_mul(bf16x2_sub(code_pair(w, 3, mask, magic), zp), sp);
                }
                // inputs 8 i16 .. 8 i16 + 7 of row n: chunk i16 / 8, 16-byte unit (i16 % 8) ^ (n % 8)
                *reinterpret_cast<uint4*>(bt + (i16 >> 3) * kChunk + n * 128 + (((i16 & 7) ^ (n & 7)) << 4)) = v;
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(bar(B_BFULL0 + b));
                mbar_arrive(bar(B_EMPTY0 + s));
            }
        }
        if (!ok && lane == 0) {
            *abort_flag = 1;
            atomicOr(err, kDevErrTimeout);
        }
        // epilogue: this warp reads TMEM lanes 32 (warp % 4) .. + 31 (tokens)
        const bool acc_ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_ACC), 0u, abort_flag, kWaitNs));
        if (ok && acc_ok) {
            tc_fence_after();
            const int q = warp & 3;
            const int m = m0 + q * 32 + lane;
            for (int c = 0; c < kBN / 32; ++c) {
                uint32_t r[32];
                tmem_ld32(tmem + (static_cast<uint32_t>(q * 32) << 16) + 32u * c, r);
                tmem_wait_ld();
                const int col = n0 + 32 * c;
                if (m < T && col < N) {
                    // destination of these 32 columns: y, or a part of the split output
                    uint16_t* base_ptr = y;
                    int stride = epi.n0, cc = col;
                    if (col >= epi.n1) {
                        base_ptr = epi.y2;
                        stride = N - epi.n1;
                        cc = col - epi.n1;
                    } else if (col >= epi.n0) {
                        base_ptr = epi.y1;
                        stride = epi.n1 - epi.n0;
                        cc = col - epi.n0;
                    }
                    uint4* dst = reinterpret_cast<uint4*>(base_ptr + static_cast<size_t>(m) * stride + cc);
                    float f[32];
#pragma unroll
                    for (int e = 0; e < 32; ++e) f[e] = __uint_as_float(r[e]);
                    if (epi.residual != nullptr) {
                        const uint4* res = reinterpret_cast<const uint4*>(epi.residual + static_cast<size_t>(m) * N + col);
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            const uint4 rv = res[u];
                            const uint32_t w4[4] = {rv.x, rv.y, rv.z, rv.w};
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                f[8 * u + 2 * e] += __uint_as_float(w4[e] << 16);
                                f[8 * u + 2 * e + 1] += __uint_as_float(w4[e] & 0xFFFF0000u);
                            }
                        }
                    }
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        dst[u] = make_uint4(pack_bf16x2(f[8 * u + 0], f[8 * u + 1]), pack_bf16x2(f[8 * u + 2], f[8 * u + 3]),
                                            pack_bf16x2(f[8 * u + 4], f[8 * u + 5]), pack_bf16x2(f[8 * u + 6], f[8 * u + 7]));
                }
            }
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
    CUtensorMap map;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(T)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(K) * 2};
    const cuuint32_t box[2] = {64, static_cast<cuuint32_t>(kBM)};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = g_encode(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t*>(x), dims, strides, box,
                                estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    const dim3 grid(static_cast<unsigned>(N / kBN), static_cast<unsigned>((T + kBM - 1) / kBM));
    W4GemmEpi epi = {N, N, nullptr, nullptr, nullptr};
    if (epi_in != nullptr) epi = *epi_in;
    w4_gemm_kernel<<<grid, kThreads, L::ALLOC, st>>>(map, tiles, T, N, K, y, err, epi);
    return cudaGetLastError();
}

}  // namespace attn

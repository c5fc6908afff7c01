// w4_gemv.cu -- W4BF16 weight-only GEMV for the decode-side matmuls.
//
// The paper deploys every model with W4BF16 quantization, 4-bit weights and bf16
// activations (Section 5.1), and its decode throughput is the weight stream: each
// generated token reads every weight once (Section 5.2).  Grouped asymmetric codes
// (the GPTQ / AWQ form the paper's tool chain reads): weight row n, input k, group
// g = k / 128, code q in 0..15, zero point z in 0..15 and bf16 scale s per (n, g):
//   y[m, n] = sum_k x[m, k] * (q[n, k] - z[n, g]) * s[n, g]
// for the few activation rows m (at most 8 per launch) of a decode batch.  The kernel
// is built around the weight stream:
//   * the weights arrive as one stream of 1072-byte tiles, each 16 rows x one 128-input
//     group with the 16 rows' scales and zero points (tile (T, G) is record
//     T * K/128 + G).  A unit is one row-tile; one stage of a unit is up to
//     kTilesPerStage consecutive tiles (one contiguous bulk copy).  Each warp owns a
//     private ring of kStages stages in shared memory with one mbarrier each and keeps
//     kStages - 1 copies in flight ahead of the stage it decodes (across unit
//     boundaries): every warp reads contiguous memory, the bytes in flight do not live
//     in registers, and the ring bookkeeping is paid once per stage;
//   * decoding: with the code of input 8i + j at bit (0, 16, 4, 20, 8, 24, 12, 28)[j]
//     of word i, a shift and one masked OR of the bf16 pair 128.0 | 128.0 turn the
//     codes of inputs (k, k + 1) into the exact bf16 pair (128 + q_k, 128 + q_k+1).
//     Those pairs are the A fragments of mma.sync m16n8k16 (16 rows x 16 inputs),
//     whose B fragments are the x rows (staged once per CTA in fragment order) and
//     whose f32 accumulators give D = sum over the group of (128 + q) x.  (tcgen05.mma
//     reads A only from shared or tensor memory: the decoded tile would make a round
//     trip there, at 4x the HBM bytes, for a product only 8 columns wide);
//   * per group and row, y += s * (D - (128 + z) * sum of x over the group): exact
//     products, f32 sums (the tensor cores take the multiply-adds off the CUDA
//     cores, which then only decode, so up to 8 x rows cost the same as one);
//   * split-K inside the CTA when the rows are few: the 8 warps of a CTA work on
//     8 / KS units, KS warps per unit on a KS-th of its groups each, and the partial
//     sums meet in shared memory;
//   * a warp's first copies are issued before x is staged, so the prologue overlaps the
//     weight stream;
//   * fused around the product (Listing 1's block): an optional RMSNorm of x, applied to
//     the staged copy before the group sums; an optional residual added in f32 before the
//     bf16 rounding; and an optional split of the output columns into three arrays (q, k
//     and v of a fused QKV projection);
//   * launched as a programmatic dependent of the previous kernel on the stream: every
//     read of data that kernel may write (x) and every write (y) comes after
//     griddepcontrol.wait, and each CTA lets the next kernel start once it has begun.  With
//     early_weights the first weight copies are issued before the wait too (the caller
//     promises the previous kernel does not write the tiles), so a chain of GEMVs streams
//     the next matrix while the last CTAs of the previous one finish.
// Every wait is bounded: a tile that never lands sets ATTN_DEVERR_TIMEOUT in *err (when
// err is not null) and the warp stops decoding.
#include <cuda_bf16.h>

#include <cstdint>
#include <mutex>

#include "internal.h"
#include "sm100_ptx.cuh"

namespace attn {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
// 4 tiles per copy and a double-buffered ring measured best among 1..8 tiles per copy
// and 2..6 stages (deeper rings cost CTAs per SM and gained nothing)
constexpr int kTilesPerStage = 4;  // tiles (groups) per bulk copy
constexpr int kStages = 2;         // ring depth per warp
constexpr int kUnitRows = 16;      // rows per unit (the mma M)
constexpr int kTileBytes = 1072;   // 16 x 64 code bytes, 16 scales, 16 zero points
constexpr int kScaleOff = 1024, kZeroOff = 1056;
constexpr int kStageBytes = kTilesPerStage * kTileBytes;
constexpr int kRingBytes = kWarps * kStages * kStageBytes;
constexpr int kBarBytes = kWarps * kStages * 8;
constexpr int kRedFloats = 2 * kWarps * 32 * 4;  // split-K partials, double-buffered
constexpr long long kSmemLimit = 232448;         // opt-in shared memory per CTA (227 KB)
// what is left for x in fragment order (2K bytes per row) and its group sums (K/4 bytes)
constexpr long long kXBytes = kSmemLimit - kRingBytes - kBarBytes - kRedFloats * 4;
static_assert(kXBytes >= 16 * 1024, "the rings leave too little shared memory for x");
constexpr uint32_t kPairMagic = 0x43004300u;   // bf16 128.0 in both halves
constexpr uint32_t kPairMask = 0x000F000Fu;    // the low code of each 16-bit half
constexpr uint64_t kWaitNs = 1000000000ull;

// One contiguous global -> shared copy completing on `bar` (16-byte aligned, size a
// multiple of 16).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

__device__ __forceinline__ void cp_async_8(uint32_t dst, const void* src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(dst), "l"(src) : "memory");
}

__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// D += A (16 x 16, bf16, row) * B (16 x 8, bf16, col), f32 accumulators.
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                               uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// ((w >> 4j) & 0x000F000F) | 0x43004300 as one three-input logic op (LUT 0xEA: (a & b) | c).
__device__ __forceinline__ uint32_t code_pair(uint32_t w, int j, uint32_t mask, uint32_t magic) {
    uint32_t r;
    asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(r) : "r"(w >> (4 * j)), "r"(mask), "r"(magic));
    return r;
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

// Shared memory of one CTA: the rings, their barriers, the split-K partials, the group
// sums of x [ngroup][8] and x in fragment order [ngroup][8 mma][4 * MT lanes] (8 bytes
// each: x[g][128G + 32t + 8i + 4h + 0..3] for lane 4g + t of mma 2i + h).
__host__ __device__ constexpr size_t smem_bytes(int MT, int K) {
    return static_cast<size_t>(kRingBytes) + kBarBytes + kRedFloats * 4 + static_cast<size_t>(K / 128) * 8 * 4 +
           static_cast<size_t>(MT) * K * 2;
}

// One tile: D = sum over the group of (128 + q) x on the tensor cores, then
// acc += s * (D - (128 + z) * sum of x) for rows (g, g + 8) x columns (2t, 2t + 1).
// xb points at this lane's B fragments; lanes g >= MT read those of lane g mod MT, which
// only fills output columns >= MT, never stored.
template <int MT>
__device__ __forceinline__ void decode_tile(const uint8_t* st, const uint2* xb, const float* xs_g, int g, int t,
                                            uint32_t mask, uint32_t magic, float (&acc)[4]) {
    const uint4 c0 = *reinterpret_cast<const uint4*>(st + g * 64 + t * 16);
    const uint4 c8 = *reinterpret_cast<const uint4*>(st + (g + 8) * 64 + t * 16);
    // two accumulator chains (the even and the odd halves of each code word) halve the
    // dependent run of tensor-core ops
    float da[4] = {0.f, 0.f, 0.f, 0.f}, db[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint32_t w0 = i == 0 ? c0.x : i == 1 ? c0.y : i == 2 ? c0.z : c0.w;
        const uint32_t w8 = i == 0 ? c8.x : i == 1 ? c8.y : i == 2 ? c8.z : c8.w;
        const uint2 b0 = xb[(2 * i) * 4 * MT];
        const uint2 b1 = xb[(2 * i + 1) * 4 * MT];
        mma_bf16_16816(da, code_pair(w0, 0, mask, magic), code_pair(w8, 0, mask, magic), code_pair(w0, 1, mask, magic),
                       code_pair(w8, 1, mask, magic), b0.x, b0.y);
        mma_bf16_16816(db, code_pair(w0, 2, mask, magic), code_pair(w8, 2, mask, magic), code_pair(w0, 3, mask, magic),
                       code_pair(w8, 3, mask, magic), b1.x, b1.y);
    }
    const float d[4] = {da[0] + db[0], da[1] + db[1], da[2] + db[2], da[3] + db[3]};
    const uint16_t* scl = reinterpret_cast<const uint16_t*>(st + kScaleOff);
    const float s0 = bf16_lo(scl[g]), s8 = bf16_lo(scl[g + 8]);
    // 128 + z exactly: (2^23 + z) - (2^23 - 128)
    const float c0f = __uint_as_float(0x4B000000u | st[kZeroOff + g]) - 8388480.f;
    const float c8f = __uint_as_float(0x4B000000u | st[kZeroOff + g + 8]) - 8388480.f;
    const float2 xs = *reinterpret_cast<const float2*>(xs_g + 2 * t);
    acc[0] = fmaf(s0, fmaf(-c0f, xs.x, d[0]), acc[0]);
    acc[1] = fmaf(s0, fmaf(-c0f, xs.y, d[1]), acc[1]);
    acc[2] = fmaf(s8, fmaf(-c8f, xs.x, d[2]), acc[2]);
    acc[3] = fmaf(s8, fmaf(-c8f, xs.y, d[3]), acc[3]);
}

template <int MT>
__global__ void __launch_bounds__(kThreads) w4_gemv_kernel(const uint8_t* __restrict__ tiles,
                                                           const uint16_t* __restrict__ x, int M, int N, int K,
                                                           int KS, uint16_t* __restrict__ y, int* err,
                                                           int early_weights, W4Fused fz) {
    extern __shared__ __align__(1024) uint8_t smem[];
    const int ngroup = K / 128;
    const uint32_t ring = smem_u32(smem);
    const uint32_t bars = ring + kRingBytes;
    float* red = reinterpret_cast<float*>(smem + kRingBytes + kBarBytes);
    float* xsum = red + kRedFloats;
    uint2* xfrag = reinterpret_cast<uint2*>(xsum + ngroup * 8);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, t = lane & 3;

    if (!early_weights) griddep_wait();
    // each warp's ring: barriers, then its first kStages - 1 copies, in flight while x is staged
    if (lane == 0) {
        for (int s = 0; s < kStages; ++s) mbar_init(bars + 8 * (warp * kStages + s), 1);
        fence_mbar_init();
    }
    __syncwarp();
    const int units = (N + kUnitRows - 1) / kUnitRows;
    const int upc = kWarps / KS;  // units per CTA round
    const int blocks = (units + upc - 1) / upc;
    const int part = warp % KS, uslot = warp / KS;
    const int g0 = part * ngroup / KS, g1 = (part + 1) * ngroup / KS;
    const uint32_t my_ring = ring + warp * kStages * kStageBytes;
    // the bf16 128.0 pair, kept in a register for the three-input logic op
    uint32_t magic = kPairMagic;
    asm volatile("" : "+r"(magic));
    const uint32_t my_bars = bars + 8 * warp * kStages;

    // issue side: the next stage to load, kStages - 1 ahead of the one decoded
    int iblk = blockIdx.x, iG = g0, islot = 0;
    bool ivalid = iblk < blocks && iblk * upc + uslot < units;
    bool failed = false;
    int outstanding = 0;
    auto issue = [&]() {
        const int nt = min(kTilesPerStage, g1 - iG);
        if (lane == 0) {
            const size_t rec = static_cast<size_t>(iblk * upc + uslot) * ngroup + iG;
            const uint32_t bar = my_bars + 8 * islot;
            mbar_arrive_expect_tx(bar, nt * kTileBytes);
            bulk_load(my_ring + islot * kStageBytes, tiles + rec * kTileBytes, nt * kTileBytes, bar);
        }
        ++outstanding;
        islot = islot + 1 == kStages ? 0 : islot + 1;
        iG += nt;
        if (iG == g1) {
            iG = g0;
            iblk += gridDim.x;
            ivalid = iblk < blocks && iblk * upc + uslot < units;
        }
    };
    for (int s = 0; s < kStages - 1 && ivalid; ++s) issue();
    if (early_weights) griddep_wait();  // x and y belong to the stream order from here on
    griddep_launch_dependents();

    // x in fragment order (asynchronous 8-byte copies, rows past M zero)
    const uint32_t xfrag_s = smem_u32(xfrag);
    for (int i = tid; i < ngroup * 8 * 4 * MT; i += kThreads) {
        const int slot = i % (4 * MT), ge = i / (4 * MT);
        const int e = ge & 7, G = ge >> 3, m = slot >> 2, tt = slot & 3;
        if (m < M)
            cp_async_8(xfrag_s + 8 * i, x + static_cast<size_t>(m) * K + 128 * G + 32 * tt + 8 * (e >> 1) + 4 * (e & 1));
        else
            xfrag[i] = make_uint2(0u, 0u);
    }
    cp_async_wait_all();
    __syncthreads();
    if (fz.gamma != nullptr) {
        // RMSNorm of each row of x (Listing 1 "input_layernorm"): r = 1 / sqrt(mean(x^2) + eps),
        // then x * r * gamma rounded to bf16 in place.  A thread's fragment slot, and so its row,
        // is the same for all its elements (the stride divides by 4 * MT).
        const int slot = tid % (4 * MT), m = slot >> 2;
        float ss = 0.f;
        for (int i = tid; i < ngroup * 8 * 4 * MT; i += kThreads) {
            const uint2 v = xfrag[i];
            const float a = bf16_lo(v.x), b = bf16_hi(v.x), c = bf16_lo(v.y), d = bf16_hi(v.y);
            ss = fmaf(a, a, fmaf(b, b, fmaf(c, c, fmaf(d, d, ss))));
        }
        // lanes of one row: those that differ in the two low lane bits or in bits >= 4 * MT
        ss += __shfl_xor_sync(0xFFFFFFFFu, ss, 1);
        ss += __shfl_xor_sync(0xFFFFFFFFu, ss, 2);
        for (int off = 4 * MT; off < 32; off <<= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, off);
        if ((lane & 3) == 0 && lane < 4 * MT) red[warp * 8 + m] = ss;
        __syncthreads();
        if (tid < MT) {
            float tot = 0.f;
            for (int w = 0; w < kWarps; ++w) tot += red[w * 8 + tid];
            red[kWarps * 8 + tid] = 1.f / sqrtf(tot / static_cast<float>(K) + fz.eps);
        }
        __syncthreads();
        const float r = red[kWarps * 8 + m];
        for (int i = tid; i < ngroup * 8 * 4 * MT; i += kThreads) {
            if (m >= M) break;
            const int ge = i / (4 * MT), e = ge & 7, G = ge >> 3, tt = slot & 3;
            const int k0 = 128 * G + 32 * tt + 8 * (e >> 1) + 4 * (e & 1);
            const uint2 gm = *reinterpret_cast<const uint2*>(fz.gamma + k0);
            const uint2 v = xfrag[i];
            xfrag[i] = make_uint2(pack_bf16x2(bf16_lo(v.x) * r * bf16_lo(gm.x), bf16_hi(v.x) * r * bf16_hi(gm.x)),
                                  pack_bf16x2(bf16_lo(v.y) * r * bf16_lo(gm.y), bf16_hi(v.y) * r * bf16_hi(gm.y)));
        }
        __syncthreads();
    }
    // group sums of x, one (group, row) per thread
    for (int i = tid; i < ngroup * 8; i += kThreads) {
        const int G = i >> 3, m = i & 7;
        float s = 0.f;
        if (m < M) {
            const uint2* p = xfrag + static_cast<size_t>(G) * 8 * 4 * MT + 4 * m;
#pragma unroll 8
            for (int e = 0; e < 8; ++e)
#pragma unroll
                for (int tt = 0; tt < 4; ++tt) {
                    const uint2 v = p[e * 4 * MT + tt];
                    s += (bf16_lo(v.x) + bf16_hi(v.x)) + (bf16_lo(v.y) + bf16_hi(v.y));
                }
        }
        xsum[i] = s;
    }
    __syncthreads();

    int cslot = 0;
    uint32_t cphase = 0;
    int rb = 0;  // split-K buffer
    for (int blk = blockIdx.x; blk < blocks; blk += gridDim.x) {
        const int unit = blk * upc + uslot;
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
        if (unit < units) {
            for (int G = g0; G < g1; G += kTilesPerStage) {
                if (ivalid && !failed) {
                    __syncwarp();  // every lane is done with the slot the copy overwrites
                    issue();
                }
                if (!failed) {
                    const bool landed = mbar_wait(my_bars + 8 * cslot, cphase, nullptr, kWaitNs);
                    failed = __any_sync(0xFFFFFFFFu, !landed);
                    if (failed && err != nullptr && lane == 0) atomicOr(err, kDevErrTimeout);
                }
                if (!failed) {  // (the slot of a failed wait stays current for the drain below)
                    --outstanding;
                    const uint8_t* st = smem + (my_ring - ring) + cslot * kStageBytes;
                    const int nt = min(kTilesPerStage, g1 - G);
                    const uint2* xb = xfrag + static_cast<size_t>(G) * 8 * 4 * MT + (lane & (4 * MT - 1));
                    if (nt == kTilesPerStage) {
#pragma unroll
                        for (int tt = 0; tt < kTilesPerStage; ++tt)
                            decode_tile<MT>(st + tt * kTileBytes, xb + tt * 8 * 4 * MT, xsum + (G + tt) * 8, g, t,
                                            kPairMask, magic, acc);
                    } else {
                        for (int tt = 0; tt < nt; ++tt)
                            decode_tile<MT>(st + tt * kTileBytes, xb + tt * 8 * 4 * MT, xsum + (G + tt) * 8, g, t,
                                            kPairMask, magic, acc);
                    }
                    cslot = cslot + 1 == kStages ? 0 : cslot + 1;
                    if (cslot == 0) cphase ^= 1u;
                }
            }
        }
        if (KS > 1) {
            float4* rr = reinterpret_cast<float4*>(red) + (rb * kWarps + warp) * 32 + lane;
            *rr = make_float4(acc[0], acc[1], acc[2], acc[3]);
            __syncthreads();
            if (part == 0) {
                for (int p = 1; p < KS; ++p) {
                    const float4 o = rr[p * 32];
                    acc[0] += o.x;
                    acc[1] += o.y;
                    acc[2] += o.z;
                    acc[3] += o.w;
                }
            }
            rb ^= 1;
        }
        if (part == 0 && unit < units) {
            const int r0 = unit * kUnitRows + g, n0 = 2 * t;
#pragma unroll
            for (int v = 0; v < 4; ++v) {
                // weight row `row` is output column `row` of x row `n`
                const int row = r0 + ((v & 2) ? 8 : 0), n = n0 + (v & 1);
                if (n < M && row < N) {
                    float o = acc[v];
                    if (fz.residual != nullptr) o += bf16_lo(fz.residual[static_cast<size_t>(n) * N + row]);
                    uint16_t* dst = row < fz.n0   ? y + static_cast<size_t>(n) * fz.n0 + row
                                    : row < fz.n1 ? fz.y1 + static_cast<size_t>(n) * (fz.n1 - fz.n0) + (row - fz.n0)
                                                  : fz.y2 + static_cast<size_t>(n) * (N - fz.n1) + (row - fz.n1);
                    *dst = __bfloat16_as_ushort(__float2bfloat16_rn(o));
                }
            }
        }
    }
    // after a timeout: let the copies still in flight (the failed one and those issued
    // after it) land, each wait bounded, before the warp exits
    if (failed) {
        for (int s = 0; s < outstanding && s < kStages; ++s) {
            mbar_wait(my_bars + 8 * cslot, cphase, nullptr, kWaitNs);
            cslot = cslot + 1 == kStages ? 0 : cslot + 1;
            if (cslot == 0) cphase ^= 1u;
        }
    }
}

// Per device: the SM count and, per MT, whether the shared-memory limit is raised and the
// CTAs per SM at the last shared-memory size asked for (the host side stays cheap when a
// decode loop calls the same shapes over and over).
constexpr int kMaxDevices = 64;
std::mutex g_mutex;
int g_sms[kMaxDevices] = {};
bool g_configured[kMaxDevices][4] = {};
size_t g_occ_smem[kMaxDevices][4] = {};
int g_occ[kMaxDevices][4] = {};

template <int MT>
cudaError_t launch_t(const uint8_t* tiles, const uint16_t* x, int M, int N, int K, uint16_t* y, int* err,
                     bool early_weights, const W4Fused& fz, cudaStream_t st) {
    constexpr int mi = MT == 1 ? 0 : MT == 2 ? 1 : MT == 4 ? 2 : 3;
    auto kern = w4_gemv_kernel<MT>;
    const size_t smem = smem_bytes(MT, K);
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    {
        std::lock_guard<std::mutex> lock(g_mutex);
        if (g_sms[dev] == 0) {
            e = cudaDeviceGetAttribute(&g_sms[dev], cudaDevAttrMultiProcessorCount, dev);
            if (e != cudaSuccess) return e;
        }
        if (!g_configured[dev][mi]) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(kSmemLimit));
            if (e != cudaSuccess) return e;
            g_configured[dev][mi] = true;
        }
    }
    int per_sm = 0, nsm = 0;
    {
        std::lock_guard<std::mutex> lock(g_mutex);
        per_sm = g_occ_smem[dev][mi] == smem ? g_occ[dev][mi] : 0;
        nsm = g_sms[dev];
    }
    if (per_sm == 0) {
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, smem);
        if (e != cudaSuccess) return e;
        if (per_sm < 1) return cudaErrorInvalidConfiguration;
        std::lock_guard<std::mutex> lock(g_mutex);
        g_occ_smem[dev][mi] = smem;
        g_occ[dev][mi] = per_sm;
    }

    // Split-K factor: the fewest stages on the busiest warp.  Grid: every resident CTA slot
    // (so that the SMs get equal numbers of CTAs, whose round counts differ by at most one).
    const long long units = (static_cast<long long>(N) + kUnitRows - 1) / kUnitRows;
    const int ngroup = K / 128;
    const long long grid_max = static_cast<long long>(nsm) * per_sm;
    int best_ks = 1;
    long long best_t = -1, best_blocks = 0;
    for (int ks = 1; ks <= kWarps && ks <= ngroup; ks *= 2) {
        const long long blocks = (units + kWarps / ks - 1) / (kWarps / ks);
        const long long rounds = (blocks + grid_max - 1) / grid_max;
        const long long per_part = (ngroup + ks - 1) / ks;
        const long long tsteps = rounds * ((per_part + kTilesPerStage - 1) / kTilesPerStage);
        if (best_t < 0 || tsteps < best_t) {
            best_t = tsteps;
            best_ks = ks;
            best_blocks = blocks;
        }
    }
    const unsigned grid = static_cast<unsigned>(best_blocks < grid_max ? best_blocks : grid_max);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, tiles, x, M, N, K, best_ks, y, err, early_weights ? 1 : 0, fz);
}

}  // namespace

int w4_gemv_max_rows(int K) {
    const long long per_row = static_cast<long long>(K) * 2;
    const long long avail = kXBytes - static_cast<long long>(K / 128) * 8 * 4;
    if (avail < per_row) return 0;
    const long long fit = avail / per_row;
    return fit >= 8 ? 8 : fit >= 4 ? 4 : fit >= 2 ? 2 : 1;
}

cudaError_t launch_w4_gemv(const uint8_t* tiles, const uint16_t* x, int M, int N, int K, uint16_t* y, int* err,
                           bool early_weights, const W4Fused& fz, cudaStream_t st) {
    if (M <= 1) return launch_t<1>(tiles, x, M, N, K, y, err, early_weights, fz, st);
    if (M <= 2) return launch_t<2>(tiles, x, M, N, K, y, err, early_weights, fz, st);
    if (M <= 4) return launch_t<4>(tiles, x, M, N, K, y, err, early_weights, fz, st);
    return launch_t<8>(tiles, x, M, N, K, y, err, early_weights, fz, st);
}

}  // namespace attn

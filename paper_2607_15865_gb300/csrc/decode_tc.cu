// decode_tc.cu -- K3 for head_dim 128: split-KV decode attention on the tensor cores,
// with the merge of the splits fused in.
//
// Decode (Section 4.4): one new query per sequence b at position p = hist_len[b]
// attends to cache slots [0, p] of its kv head; its own k/v go to slot p (the
// in-place "Concat" of Listing 2, Section 4.6.3).  The same kernel takes ntok new
// tokens per sequence (multi-token decode, e.g. verifying a speculative draft): token
// i at position p + i attends to slots [0, p + i], causally among the new tokens.
//
// With grouped-query attention the G query heads of a kv head read the same keys,
// so a CTA's work is a contraction [C x D] x [D x keys], C = G x ntok columns (query
// head, new token) -- done here with tcgen05 in swapped form so that the 128 keys of
// a tile fill the MMA's M dimension:
//   S^T [128 keys x 16] = K_tile [128 x D] . Q^T       (Q: C columns, zero-padded to 16)
//   O^T [D x 16]      += V_tile^T [D x 128] . P^T [128 x 16]
// Both accumulate in TMEM.  The T = ceil((p+ntok)/128) key tiles of a sequence are
// claimed by the nsplit CTAs of its item (b, kv head, column group): in a one-wave grid
// split s starts with tile s, in a larger one only split 0 has a fixed first tile; every
// other tile is a ticket from the item's counter, so CTAs that stream faster take more
// tiles, splits dispatched late help the items that still have tiles, and no CTA loads
// keys that another one owns.
// 192 threads:
//   warps 0-3  one thread per key of the tile: scores from TMEM, masking, P^T (bf16)
//              into shared memory, per-thread partial row sums.  The running max m
//              moves lazily: a tile whose scores all stay within 2^8 of m (checked
//              with one OR-barrier) is exponentiated against m as it is; otherwise
//              the per-column tile maxima are reduced (a halving butterfly: 16
//              shuffles for 16 columns) and O^T is rescaled.  Epilogue: one thread
//              per output dimension d;
//   warp 4     TMA producer: K and V tiles of 128 keys (128-byte swizzle) into
//              rings of 2 (K) and 4 (V) stages of 32 KB;
//   warp 5     tcgen05 issuer; it also owns the new tokens: it rotates their k (RoPE
//              from the table, the same float arithmetic and bf16 rounding as K1),
//              writes k and v to their slots of the cache and into the shared-memory
//              copies of the tiles that hold those slots (zeroing the V rows past the
//              last new slot: slots past it may hold anything, and 0 * NaN would poison
//              O), so the MMA itself produces the new keys' scores.
// Merge of the splits that took tiles, each holding a partial (m, l, acc[D]) per column:
//   out = sum_s 2^(m_s - M) acc_s / sum_s 2^(m_s - M) l_s,  M = max_s m_s,
// in one of three ways, each its own instantiation (MODE):
//   one wave, global: split s writes its partial at slot s and counts itself; the last
//     of the min(nsplit, T) splits with tiles merges;
//   one wave, cluster (when a cluster per item fits on the device at once): the item's
//     splits are one thread-block cluster; each stages its partial in shared memory and,
//     after a cluster barrier, merges a share of the dimensions from its peers' staging;
//   several waves: a split writes its partial to a slot it takes from a counter and adds
//     (1 contributor, its tile count) to the item's done word; the split whose addition
//     completes T tiles merges the slots.
// A split that took all T tiles writes the normalised output itself.  Every wait is
// bounded; on expiry the CTA records kDevErrTimeout, lets its copies and MMAs finish,
// releases TMEM and still takes part in the merge (its count, or the cluster barriers).
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>

#include "internal.h"
#include "sm100_ptx.cuh"

namespace attn {
namespace {

constexpr int D = 128;
constexpr int KT = 128;     // keys per tile (MMA M)
constexpr int NH = 16;      // padded columns of Q^T (MMA N): query heads x new tokens
constexpr int kMaxTok = 16;  // new tokens per sequence in one launch (heads x tokens <= NH)
// The kernel is built for MAXTOK = 1 (plain decode) and kMaxTok (multi-token decode): the
// issuer keeps the new tokens' rotated k and v in registers, unrolled over MAXTOK, and
// sixteen unrolled slots cost a single-token decode about 2 us.
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
    static constexpr int OFF_K = 0;                // K ring (the merge's weights reuse it)
    static constexpr int OFF_V = KST * TILE;       // V ring
    static constexpr int OFF_Q = OFF_V + VST * TILE;  // Q^T [16 heads x 128] bf16, 2 x 2 KB
    static constexpr int OFF_P = OFF_Q + 2 * NH * 128;          // P^T [16 x 128 keys] x 2 buffers
    static constexpr int OFF_RED = OFF_P + 2 * 2 * NH * 128;    // float tile maxima [16 heads][4 warps]
    static constexpr int OFF_LS = OFF_RED + NH * 4 * 4;         // float l partials [16 heads][4 warps]
    static constexpr int OFF_META = OFF_LS + NH * 4 * 4;       // int tile index per local tile, ring of 8
    static constexpr int OFF_BAR = OFF_META + 8 * 4;
    static constexpr int OFF_TMEM = OFF_BAR + NBAR * 8;
    static constexpr int OFF_ABORT = OFF_TMEM + 4;
    static constexpr int OFF_LAST = OFF_ABORT + 4;
    // int [8] at OFF_LAST: merge flag, merged slots, this CTA's partial slot, tiles it
    // claimed, a helper split's first ticket
    static constexpr int OFF_CROW = OFF_LAST + 32;  // size_t [16]: partial row (slot 0) of column c
    static constexpr int OFF_OROW = OFF_CROW + NH * 8;  // size_t [16]: q / out row of column c
    static constexpr int BYTES = OFF_OROW + NH * 8;
    static constexpr int ALLOC = BYTES + 1024;
};
static_assert(L::ALLOC <= 232448, "shared memory of one CTA");
static_assert((kThreads / 32) * NH * 8 + (kThreads / 32) * NH * D * 4 <= KST * L::TILE,
              "merge buffers fit in the K ring");

__device__ __forceinline__ float bf16_at(const uint16_t* p) { return __uint_as_float(static_cast<uint32_t>(*p) << 16); }
__device__ __forceinline__ uint16_t to_bf16(float x) { return __bfloat16_as_ushort(__float2bfloat16_rn(x)); }

// Byte offset of element (row, col) in a [rows x 128] bf16 tile stored as two
// 128-byte-swizzled 64-column chunks of `rows` rows (chunk stride rows * 128 bytes).
__device__ __forceinline__ uint32_t sw_elem(int row, int col, int rows) {
    return static_cast<uint32_t>((col >> 6) * rows * 128 + row * 128 + ((((col & 63) >> 3) ^ (row & 7)) << 4) +
                                 (col & 7) * 2);
}

template <int N>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, uint32_t (&r)[N]) {
    static_assert(N == 8 || N == 16, "8 or 16 columns");
    if constexpr (N == 16) {
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
            "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
            : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
              "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
            : "r"(taddr));
    } else {
        asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                     : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                     : "r"(taddr));
    }
}

template <int N>
__device__ __forceinline__ void tmem_st_cols(uint32_t taddr, const uint32_t (&r)[N]) {
    static_assert(N == 8 || N == 16, "8 or 16 columns");
    if constexpr (N == 16) {
        asm volatile(
            "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
            "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
            "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
            "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
            : "memory");
    } else {
        asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"r"(taddr),
                     "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
                     : "memory");
    }
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

// Reduction of N values per lane over the 32 lanes of a warp by recursive halving:
// at each step a lane keeps half of its values, sends the other half to its partner
// and combines (N - 1 shuffles for N -> 1), then the remaining lane bits reduce
// plainly.  Returns the reduction of value index halving_owner<N>(lane) over all
// 32 lanes; v is clobbered.
template <int N, bool kMax>
__device__ __forceinline__ float warp_reduce_halving(float (&v)[N], int lane) {
    static_assert(N == 8 || N == 16, "8 or 16 values");
#pragma unroll
    for (int half = N / 2, mask = 16; half >= 1; half >>= 1, mask >>= 1) {
        const bool upper = (lane & mask) != 0;
#pragma unroll
        for (int i = 0; i < half; ++i) {
            const float keep = upper ? v[i + half] : v[i];
            const float send = upper ? v[i] : v[i + half];
            const float got = __shfl_xor_sync(0xFFFFFFFFu, send, mask);
            v[i] = kMax ? fmaxf(keep, got) : keep + got;
        }
    }
    float r = v[0];
    constexpr int kRest = (N == 16) ? 1 : 2;  // lane bits not used by the halving steps
#pragma unroll
    for (int mask = kRest; mask > 0; mask >>= 1) {
        const float got = __shfl_xor_sync(0xFFFFFFFFu, r, mask);
        r = kMax ? fmaxf(r, got) : r + got;
    }
    return r;
}

// Value index whose reduction lane `lane` holds after warp_reduce_halving<N>, and
// whether that lane is the first of the lanes holding it.
template <int N>
__device__ __forceinline__ int halving_owner(int lane) {
    return N == 16 ? (lane >> 1) : (lane >> 2);
}
template <int N>
__device__ __forceinline__ bool halving_leader(int lane) {
    return N == 16 ? (lane & 1) == 0 : (lane & 3) == 0;
}

// NHP: columns the softmax processes (8 when G * ntok <= 8, else 16); the MMA always
// runs N = 16 with the rows of Q^T past the CTA's C columns zero.  With more than 16
// columns (G * ntok > 16) the grid's z dimension is (sequence, column group): every column
// group streams the same key tiles, which its sibling CTAs read at about the same time, so
// the repeats come from L2.
// MODE: how the splits of an item meet.  kModeGlobal (one wave): each split with tiles
// writes its partial (m, l, acc) at slot s in global memory and the last of them merges;
// kModeCluster (one wave): the item's splits are one thread-block cluster and merge through
// distributed shared memory; kModeWaves: the grid is several waves (s0 < nsplit), with
// helper splits and slot and visit counters.  Each is its own instantiation, so that a
// launch runs only the code of its mode.
constexpr int kModeGlobal = 0, kModeCluster = 1, kModeWaves = 2;
template <int NHP, int MAXTOK, int MODE>
__global__ void __launch_bounds__(kThreads, 1) decode_tc_kernel(
    const __grid_constant__ CUtensorMap map_k, const __grid_constant__ CUtensorMap map_v,
    const uint16_t* __restrict__ q, const uint16_t* __restrict__ k_new, const uint16_t* __restrict__ v_new,
    const int32_t* __restrict__ d_hist, int hist_add, int ntok, uint16_t* __restrict__ k_cache,
    uint16_t* __restrict__ v_cache, const float* __restrict__ cos_tab, const float* __restrict__ sin_tab, int Hq, int Hkv,
    int max_len, int nsplit,
    float scale_log2, float* __restrict__ part_o, float* __restrict__ part_ml, int* __restrict__ counters,
    uint16_t* __restrict__ out, int* __restrict__ err, int producer_early, uint64_t wait_ns, int ncg, int spec,
    int s0) {
    constexpr bool WAVES = MODE == kModeWaves;
    constexpr int HALF = D / 2;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* gb = smem_raw + (base - raw);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(gb + L::OFF_ABORT);
    float* red = reinterpret_cast<float*>(gb + L::OFF_RED);
    float* ls = reinterpret_cast<float*>(gb + L::OFF_LS);
    auto bar = [&](int i) -> uint32_t { return base + L::OFF_BAR + 8u * static_cast<uint32_t>(i); };

    const int G = Hq / Hkv;
    // Columns: global column c = token c / G, head h0 + c % G, of G * ntok; this CTA takes the
    // 16-column group cg, columns c0 .. c0 + C - 1 (its local column h is global column c0 + h).
    // Grid (split, kv head, sequence x column group) for one wave; for several waves (s0 <
    // nsplit) (kv head, sequence x column group, split), so that every item's split 0 is
    // dispatched before any split 1, and so on: the later splits start as SMs free up and
    // help the items that still have tiles.
    constexpr bool wave_grid = WAVES;
    const int s = wave_grid ? blockIdx.z : blockIdx.x;
    const int g = wave_grid ? blockIdx.x : blockIdx.y;
    const int bz = static_cast<int>(wave_grid ? blockIdx.y : blockIdx.z);
    const int b = bz / ncg;
    const int cg = bz - b * ncg;
    const int c0 = cg * NH;
    const int C = min(NH, G * ntok - c0);
    const int h0 = g * G;
    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;
    // The lengths, q and the new k/v are the caller's inputs: complete when this grid
    // starts (it is a dependent launch only after another decode step, which lets its
    // dependents start only once its own predecessors are complete).
    const int hist = decode_hist(d_hist, b, hist_add);  // in flight while the barriers and TMEM are set up
    const int kv_row = b * Hkv + g;
    const bool multi = nsplit > 1;
    // Several waves (s0 < nsplit): helper splits may claim after their item is merged, so
    // slots are taken from a counter and every split records its visit; in one wave the
    // splits with tiles are exactly s < min(nsplit, T), each using slot s.
    const bool waves = WAVES && multi;
    int* lastv = reinterpret_cast<int*>(gb + L::OFF_LAST);  // [0] merge flag [1] slots [2] slot [3] claimed
    const int n_items = static_cast<int>(wave_grid ? gridDim.x * gridDim.y : gridDim.y * gridDim.z);
    // Counters of this item (sequence, kv head, column group): tile claims, partial slots and
    // visits (ints, then 64-bit (contributors << 32 | tiles done) words from an even offset);
    // all zero between launches: the last split to visit resets the first three, the merging
    // split the fourth.
    const int ctr_row = kv_row * ncg + cg;
    int* claim_ctr = counters + ctr_row;
    int* slot_ctr = counters + n_items + ctr_row;
    int* visit_ctr = counters + 2 * n_items + ctr_row;
    unsigned long long* done_ctr = reinterpret_cast<unsigned long long*>(counters + ((3 * n_items + 1) & ~1)) + ctr_row;
    // A helper split (s >= s0: a grid of several waves) first asks its item's counter for a
    // tile.  If none is left -- the item is done, or its tiles are all taken -- the CTA
    // records its visit and leaves before any set-up.  When the batch's lengths are within
    // 10% of each other (read by one warp, batches of up to 1024) there is nothing to even
    // out, and helpers leave without asking: the splits 0 then finish their items alone and
    // write the outputs without a merge.  (After the previous decode step the counters are
    // touched only once that step is complete.)
    int first_ticket = 0;
    if (WAVES && multi && s >= s0) {
        if (warp == 0) {
            if (producer_early == 0) griddep_wait();
            const int batch = static_cast<int>(gridDim.y) / ncg;
            int tmax = 0, tsum = 0;
            if (batch <= 1024) {
                for (int bb = lane; bb < batch; bb += 32) {
                    const int hb = decode_hist(d_hist, bb, hist_add);
                    const int tb = hb >= 0 && hb <= max_len - ntok ? (hb + ntok + KT - 1) / KT : 0;
                    tmax = max(tmax, tb);
                    tsum += tb;
                }
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) {
                    tmax = max(tmax, __shfl_xor_sync(0xFFFFFFFFu, tmax, off));
                    tsum += __shfl_xor_sync(0xFFFFFFFFu, tsum, off);
                }
            }
            const bool even = batch <= 1024 && 10LL * tmax * batch <= 11LL * tsum;
            if (lane == 0) {
                int t = -1;
                if (hist >= 0 && hist <= max_len - ntok) {
                    if (!even) t = s0 + atomicAdd(claim_ctr, 1);
                    if (t >= (hist + ntok + KT - 1) / KT) t = -1;
                    if (t < 0 && atomicAdd(visit_ctr, 1) == nsplit - 1) {
                        *claim_ctr = 0;
                        *slot_ctr = 0;
                        *visit_ctr = 0;
                    }
                }
                lastv[4] = t;
            }
        }
        __syncthreads();
        first_ticket = lastv[4];
        if (first_ticket < 0) return;  // (a skipped sequence also leaves here, touching nothing)
    }
    // The producer sets up the barriers and, unless the previous kernel may have written the
    // cache (a decode step right after another, spec = 0), issues the copies of its first
    // tile, tile s, before the length is known: the K slot's arrival is held back until the
    // producer knows whether tile s holds keys of the sequence (the copies read in-range
    // slots or the map's zero fill either way; a tile past the sequence is not used).
    const bool spec_first = spec != 0 && s < s0 && s * KT < max_len;
    if (warp == kWarpTma && lane == 0) {
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
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_v);
        if (spec_first) {
            mbar_expect_tx(bar(B_KFULL0), L::TILE);
#pragma unroll
            for (int c = 0; c < 2; ++c)
                tma_load_3d(base + L::OFF_K + c * L::BOX, &map_k, c * 64, s * KT, kv_row, bar(B_KFULL0));
            mbar_arrive_expect_tx(bar(B_VFULL0), L::TILE);
#pragma unroll
            for (int c = 0; c < 2; ++c)
                tma_load_3d(base + L::OFF_V + c * L::BOX, &map_v, c * 64, s * KT, kv_row, bar(B_VFULL0));
        }
    }

    if (tid < NH) {
        const int c = c0 + min(tid, C - 1);
        const size_t r = (static_cast<size_t>(b) * ntok + c / G) * Hq + h0 + c % G;
        reinterpret_cast<size_t*>(gb + L::OFF_OROW)[tid] = r;
        reinterpret_cast<size_t*>(gb + L::OFF_CROW)[tid] = r * nsplit;
    }
    if (warp == kWarpMma) {
        tmem_alloc(base + L::OFF_TMEM, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<const uint32_t*>(gb + L::OFF_TMEM);
    // Dependent launch after the previous decode step: the setup above overlaps that step's
    // tail; its cache append, merge counters and partials are read or reused only after
    // this wait.  The next step may start only after it.
    // With producer_early (a dependent launch after the kernel that writes q and the new k/v)
    // the TMA warp skips this wait: it reads only the lengths, the tile counters and cache
    // tiles, which that kernel does not write (the new tokens' rows are patched in shared
    // memory), so the history streams in while that kernel finishes.  It waits before the
    // merge, and the CTA releases its own dependents only from threads that have waited.
    const bool early = producer_early != 0 && warp == kWarpTma;
    if (!early) {
        griddep_wait();
        griddep_launch_dependents();
    }

    const bool hist_ok = hist >= 0 && hist <= max_len - ntok;
    if (!hist_ok && s == 0 && g == 0 && cg == 0 && tid == 0) atomicOr(err, kDevErrHistRange);
    const int nkeys = hist + ntok;        // slots [0, hist) and the new tokens' [hist, hist + ntok)
    const int T = (nkeys + KT - 1) / KT;  // key tiles of the sequence; tile T-1 holds the last new slot
    // Splits s < s0 start with tile s; every other tile is claimed from the item's counter
    // (tickets s0, s0 + 1, ...).  A split that gets no tile writes nothing.
    // Rows of column c (token c / G, head h0 + c % G), tabulated once in the prologue:
    // q / out row (b * ntok + c / G) * Hq + h0 + c % G, and partial row of slot 0 that
    // times nsplit (slot sp adds sp).  Columns past C repeat column C - 1.
    const size_t* crow = reinterpret_cast<const size_t*>(gb + L::OFF_CROW);
    const size_t* orow = reinterpret_cast<const size_t*>(gb + L::OFF_OROW);
    int* meta = reinterpret_cast<int*>(gb + L::OFF_META);  // tile index of local tile j at [j % 8]; -1 ends

    if (!hist_ok) {
        // sequence skipped: nothing written (the speculative copies land before the CTA ends)
        if (spec_first && warp == kWarpTma && lane == 0) {
            mbar_arrive(bar(B_KFULL0));
            mbar_wait(bar(B_KFULL0), 0u, nullptr);
            mbar_wait(bar(B_VFULL0), 0u, nullptr);
        }
    } else if (warp == kWarpTma) {
        // ------------------------------------------------------------ TMA producer (lane 0)
        // Tiles are claimed, not fixed: split s < s0 starts with tile s, then takes tickets
        // s0, s0+1, ... from the item's tile counter until they run past T, so CTAs that
        // stream faster take more tiles and splits that start late find the tiles taken.  The
        // next ticket is claimed while the current tile's copies are issued.  A split that
        // gets a tile takes a partial slot; every split records its visit once its claims are
        // over.  One thread feeds both rings: the V slot of tile j frees (PV(j-4) done)
        // before the K slot does (S(j-2) done).
        if (lane == 0) {
            // (one wave with a single split that has tiles: it walks them in order, touching
            // no counter, as does the only split of an item)
            const bool claims = waves || (multi && min(nsplit, T) > 1);
            auto take = [&]() { return s0 + atomicAdd(claim_ctr, 1); };
            int cur = !multi ? 0 : (s < s0 ? min(s, T) : first_ticket);
            int claimed = cur < T ? 1 : 0;
            int nxt = !claims ? cur + 1 : (cur < T ? take() : T);
            int issued_k = 0, issued_v = 0;
            bool ok = true;
            auto advance = [&]() {
                cur = nxt;
                if (cur < T) {
                    ++claimed;
                    nxt = claims ? take() : cur + 1;
                }
            };
            for (int j = 0;; ++j) {
                const int tile = cur < T ? cur : -1;
                const int ks = j % KST, vs = j % VST;
                if (j >= KST && !mbar_wait(bar(B_KEMPTY0 + ks), static_cast<uint32_t>(j / KST - 1) & 1u, abort_flag, wait_ns)) {
                    ok = false;
                    break;
                }
                meta[j % 8] = tile;
                if (j == 0 && spec_first) {
                    // tile s is in flight: its K slot's arrival publishes meta[0]
                    mbar_arrive(bar(B_KFULL0));
                    issued_k = issued_v = 1;
                    if (tile < 0) {  // tile s holds no keys of the sequence: the copies still land
                        mbar_wait(bar(B_VFULL0), 0u, nullptr);
                        break;
                    }
                    advance();
                    continue;
                }
                if (tile < 0) {  // no more tiles: complete the K slot's phase without data
                    mbar_arrive(bar(B_KFULL0 + ks));
                    break;
                }
                mbar_arrive_expect_tx(bar(B_KFULL0 + ks), L::TILE);
#pragma unroll
                for (int c = 0; c < 2; ++c)
                    tma_load_3d(base + L::OFF_K + ks * L::TILE + c * L::BOX, &map_k, c * 64, tile * KT, kv_row,
                                bar(B_KFULL0 + ks));
                issued_k = j + 1;
                if (j >= VST && !mbar_wait(bar(B_VEMPTY0 + vs), static_cast<uint32_t>(j / VST - 1) & 1u, abort_flag, wait_ns)) {
                    ok = false;
                    break;
                }
                mbar_arrive_expect_tx(bar(B_VFULL0 + vs), L::TILE);
#pragma unroll
                for (int c = 0; c < 2; ++c)
                    tma_load_3d(base + L::OFF_V + vs * L::TILE + c * L::BOX, &map_v, c * 64, tile * KT, kv_row,
                                bar(B_VFULL0 + vs));
                issued_v = j + 1;
                advance();
            }
            if (!ok) {
                *abort_flag = 1;
                atomicOr(err, kDevErrTimeout);
                for (int t = max(0, issued_k - KST); t < issued_k; ++t)
                    mbar_wait(bar(B_KFULL0 + t % KST), static_cast<uint32_t>(t / KST) & 1u, nullptr);
                for (int t = max(0, issued_v - VST); t < issued_v; ++t)
                    mbar_wait(bar(B_VFULL0 + t % VST), static_cast<uint32_t>(t / VST) & 1u, nullptr);
                if (claims) {
                    // take every ticket still unclaimed (and count it, unprocessed), so that the
                    // item's tiles are all accounted for and its merge and reset still happen
                    const int first = s0 + atomicAdd(claim_ctr, T);
                    if (first < T) claimed += T - first;
                }
            }
            // a partial slot for a split with tiles, taken before its visit (read after the CTA
            // barrier of the merge, as is the claim count)
            lastv[2] = waves && claimed > 0 ? atomicAdd(slot_ctr, 1) : s;
            lastv[3] = claimed;
            if (waves && atomicAdd(visit_ctr, 1) == nsplit - 1) {
                // every split of the item has made its last claim: reset for the next launch
                *claim_ctr = 0;
                *slot_ctr = 0;
                *visit_ctr = 0;
            }
        }
        if (early) griddep_wait();
    } else if (warp == kWarpMma) {
        // ------------------------------------------------------------ tcgen05 issuer (+ the new tokens)
        // Lane l handles dimensions 4l .. 4l+3 of each new token tt (slot hist + tt, rotated
        // at that position by every CTA; written by the CTA that gets the slot's tile).
        const int last_row = (hist + ntok - 1) - (T - 1) * KT;  // row of the last new slot in tile T-1
        uint2 k_rot[MAXTOK], v_val[MAXTOK];
#pragma unroll
        for (int tt = 0; tt < MAXTOK; ++tt) {
            if (tt >= ntok) break;
            const int d0 = 4 * lane;
            const int dp = d0 < HALF ? d0 + HALF : d0 - HALF;  // RoPE partner dimensions
            const size_t src = (static_cast<size_t>(b * ntok + tt) * Hkv + g) * D;
            const uint2 kx = *reinterpret_cast<const uint2*>(k_new + src + d0);
            const uint2 ky = *reinterpret_cast<const uint2*>(k_new + src + dp);
            v_val[tt] = *reinterpret_cast<const uint2*>(v_new + src + d0);
            const size_t pos = static_cast<size_t>(hist + tt);
            const float4 c4 = *reinterpret_cast<const float4*>(cos_tab + pos * HALF + d0 % HALF);
            const float4 s4 = *reinterpret_cast<const float4*>(sin_tab + pos * HALF + d0 % HALF);
            const float xs[4] = {__uint_as_float(kx.x << 16), __uint_as_float(kx.x & 0xFFFF0000u),
                                 __uint_as_float(kx.y << 16), __uint_as_float(kx.y & 0xFFFF0000u)};
            const float ys[4] = {__uint_as_float(ky.x << 16), __uint_as_float(ky.x & 0xFFFF0000u),
                                 __uint_as_float(ky.y << 16), __uint_as_float(ky.y & 0xFFFF0000u)};
            const float cs[4] = {c4.x, c4.y, c4.z, c4.w}, ss[4] = {s4.x, s4.y, s4.z, s4.w};
            uint32_t kb[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float r = d0 < HALF ? __fsub_rn(__fmul_rn(xs[e], cs[e]), __fmul_rn(ys[e], ss[e]))
                                          : __fadd_rn(__fmul_rn(xs[e], cs[e]), __fmul_rn(ys[e], ss[e]));
                kb[e] = to_bf16(r);
            }
            k_rot[tt] = make_uint2(kb[0] | (kb[1] << 16), kb[2] | (kb[3] << 16));
        }
        constexpr uint32_t kIdQK = idesc_bf16_f32(KT, NH, false, false);
        constexpr uint32_t kIdPV = idesc_bf16_f32(D, NH, true, false);
        const uint32_t sQ = base + L::OFF_Q;
        auto wait_all = [&](int barrier, uint32_t parity) -> bool {
            return __all_sync(0xFFFFFFFFu, mbar_wait(bar(barrier), parity, abort_flag, wait_ns));
        };
        auto issue_pv = [&](int jj) -> bool {
            if (!wait_all(B_PFULL0 + (jj & 1), static_cast<uint32_t>(jj >> 1) & 1u)) return false;
            if (!wait_all(B_VFULL0 + jj % VST, static_cast<uint32_t>(jj / VST) & 1u)) return false;
            const uint32_t sV = base + L::OFF_V + (jj % VST) * L::TILE;
            const int vtile = meta[jj % 8];
            if (vtile * KT + KT > hist) {
                // the new tokens' v into their rows of this tile; in tile T-1 the rows past the
                // last new slot zeroed (those slots may hold anything, and 0 * NaN would poison O)
                uint8_t* vt = gb + L::OFF_V + (jj % VST) * L::TILE;
#pragma unroll
                for (int tt = 0; tt < MAXTOK; ++tt)
                    if (tt < ntok && (hist + tt) / KT == vtile)
                        *reinterpret_cast<uint2*>(vt + sw_elem(hist + tt - vtile * KT, 4 * lane, KT)) = v_val[tt];
                if (vtile == T - 1)
                    for (int i = (last_row + 1) * 16 + lane; i < KT * 16; i += 32)
                        *reinterpret_cast<uint4*>(vt + sw_elem(i >> 4, 8 * (i & 15), KT)) = make_uint4(0, 0, 0, 0);
                fence_proxy_async_smem();
            }
            __syncwarp();
            if (lane == 0) {
                tc_fence_after();
                const uint32_t sP = base + L::OFF_P + (jj & 1) * (2 * NH * 128);
#pragma unroll
                for (int kk = 0; kk < KT / 16; ++kk)
                    umma_ss(tmem + TM_O, smem_desc_sw128(sV + kk * 16 * 128, L::BOX, 1024),
                            smem_desc_sw128(sP + (kk >> 2) * NH * 128 + (kk & 3) * 32, 16, 1024), kIdPV,
                            (jj > 0 || kk > 0) ? 1u : 0u);
                umma_commit(bar(B_PVDONE));
                umma_commit(bar(B_VEMPTY0 + jj % VST));
            }
            __syncwarp();
            return true;
        };
        bool ok = wait_all(B_QREADY, 0);
        int n = 0;  // tiles this CTA processes
        if (ok) {
            for (int j = 0;; ++j) {
                const int ks = j % KST;
                if (!wait_all(B_KFULL0 + ks, static_cast<uint32_t>(j / KST) & 1u)) {
                    ok = false;
                    break;
                }
                const int tile = meta[j % 8];
                if (tile < 0) {
                    n = j;
                    break;
                }
                const uint32_t sK = base + L::OFF_K + ks * L::TILE;
                if (tile * KT + KT > hist) {  // new tokens in this tile: to the cache, rotated k into their rows
#pragma unroll
                    for (int tt = 0; tt < MAXTOK; ++tt) {
                        if (tt < ntok && (hist + tt) / KT == tile) {
                            const size_t dst = (static_cast<size_t>(kv_row) * max_len + hist + tt) * D + 4 * lane;
                            *reinterpret_cast<uint2*>(k_cache + dst) = k_rot[tt];
                            *reinterpret_cast<uint2*>(v_cache + dst) = v_val[tt];
                            *reinterpret_cast<uint2*>(gb + L::OFF_K + ks * L::TILE +
                                                      sw_elem(hist + tt - tile * KT, 4 * lane, KT)) = k_rot[tt];
                        }
                    }
                    fence_proxy_async_smem();
                }
                __syncwarp();
                if (lane == 0) {
                    tc_fence_after();
#pragma unroll
                    for (int kk = 0; kk < D / 16; ++kk) {
                        const uint32_t off = (kk >> 2) * L::BOX + (kk & 3) * 32;
                        umma_ss(tmem + (j & 1) * NH, smem_desc_sw128(sK + off, 16, 1024),
                                smem_desc_sw128(sQ + (kk >> 2) * NH * 128 + (kk & 3) * 32, 16, 1024), kIdQK,
                                kk > 0 ? 1u : 0u);
                    }
                    umma_commit(bar(B_SFULL0 + (j & 1)));
                    umma_commit(bar(B_KEMPTY0 + ks));  // K is consumed once S^T(j) completes
                }
                __syncwarp();
                if (j >= 1 && !issue_pv(j - 1)) {
                    ok = false;
                    break;
                }
            }
            if (ok) {
                // the softmax learns the count from the same end marker: S buffer n's phase
                // completes without an MMA (S(n-2) on that buffer was consumed: PFULL(n-2) seen)
                if (lane == 0) mbar_arrive(bar(B_SFULL0 + (n & 1)));
                if (n > 0) ok = issue_pv(n - 1);
                if (ok && n > 0 && lane == 0) umma_commit(bar(B_OFULL));  // every PV is complete
            }
        }
        if (!ok && lane == 0) {
            *abort_flag = 1;
            atomicOr(err, kDevErrTimeout);
        }
        if (lane == 0) {
            umma_commit(bar(B_DRAIN));
            mbar_wait(bar(B_DRAIN), 0, nullptr);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ softmax / epilogue (one thread per key)
        const int t = tid;  // key row of a tile; output dimension in the epilogue
        const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
        {
            // Q^T: row c = rotated q of token c / G, head h0 + c % G (bf16) at position
            // hist + c / G; zero rows past C; P^T buffers zeroed.  Each thread owns dimension t
            // of every column: all loads first, then the math.
            uint8_t* qs = gb + L::OFF_Q;
            const int tp = t < HALF ? t + HALF : t - HALF;  // RoPE partner dimension
            float qx[NHP], qy[NHP], c_t[NHP], s_t[NHP];
#pragma unroll
            for (int c = 0; c < NHP; ++c) {
                const int cc = min(c, C - 1);
                const uint16_t* qrow = q + orow[cc] * D;
                qx[c] = bf16_at(qrow + t);
                qy[c] = bf16_at(qrow + tp);
                const size_t pos = static_cast<size_t>(hist + (c0 + cc) / G);
                c_t[c] = cos_tab[pos * HALF + t % HALF];
                s_t[c] = sin_tab[pos * HALF + t % HALF];
            }
#pragma unroll
            for (int c = 0; c < NH; ++c) {
                uint16_t qb = 0;
                if (c < NHP && c < C) {
                    const float r = t < HALF ? __fsub_rn(__fmul_rn(qx[c], c_t[c]), __fmul_rn(qy[c], s_t[c]))
                                             : __fadd_rn(__fmul_rn(qx[c], c_t[c]), __fmul_rn(qy[c], s_t[c]));
                    qb = to_bf16(r);
                }
                *reinterpret_cast<uint16_t*>(qs + sw_elem(c, t, NH)) = qb;
            }
            for (int i = t; i < 2 * NH * 128 / 16; i += 128)
                reinterpret_cast<uint4*>(gb + L::OFF_P)[i] = make_uint4(0, 0, 0, 0);
            fence_proxy_async_smem();
            mbar_arrive(bar(B_QREADY));
        }

        float m_run[NHP], l_run[NHP];
#pragma unroll
        for (int h = 0; h < NHP; ++h) {
            m_run[h] = -INFINITY;
            l_run[h] = 0.f;
        }
        bool ok = true;
        int n = 0;  // tiles processed
        // The four softmax warps meet at named barriers (the lazy-max test, the tile maxima,
        // the epilogue): a wait that ran out in one warp is made known to all four through a
        // barrier that every one of them reaches, before any of them leaves the loop, so that
        // no warp is left waiting at a barrier the others never reach.
        for (int j = 0;; ++j) {
            ok = !named_or_128(!mbar_wait(bar(B_SFULL0 + (j & 1)), static_cast<uint32_t>(j >> 1) & 1u, abort_flag, wait_ns));
            if (!ok) break;
            const int tile = meta[j % 8];
            if (tile < 0) {
                n = j;
                break;
            }
            tc_fence_after();
            uint32_t r[NHP];
            tmem_ld_cols<NHP>(tmem + lane_base + (j & 1) * NH, r);
            tmem_wait_ld();
            // key tile * KT + t is visible to global column c (token c / G) iff it is <= hist + c / G,
            // i.e. iff c >= (key - hist) * G (always for a history key: key - hist < 0)
            const int kg = (tile * KT + t - hist) * G - c0;
            float sc[NHP];
            bool exceed = false;
#pragma unroll
            for (int h = 0; h < NHP; ++h) {
                sc[h] = (h < C && h >= kg) ? __uint_as_float(r[h]) * scale_log2 : -INFINITY;
                exceed |= sc[h] > m_run[h] + 8.f;  // lazy: P stays <= 2^8 otherwise
            }
            if (named_or_128(exceed)) {
                // per-head tile maxima: halving butterfly in the warp, then the four warps.
                // (`red` is rewritten only after the next tile's OR-barrier, which every
                // thread reaches after its reads below.)
                float mx[NHP];
#pragma unroll
                for (int h = 0; h < NHP; ++h) mx[h] = sc[h];
                const float wm = warp_reduce_halving<NHP, true>(mx, lane);
                if (halving_leader<NHP>(lane)) red[halving_owner<NHP>(lane) * 4 + warp] = wm;
                named_sync_128();
                bool any_move = false;
                float alpha[NHP];
#pragma unroll
                for (int h = 0; h < NHP; ++h) {
                    const float4 r4 = reinterpret_cast<const float4*>(red)[h];
                    const float tmx = fmaxf(fmaxf(r4.x, r4.y), fmaxf(r4.z, r4.w));
                    const bool move = tmx > m_run[h] + 8.f;
                    alpha[h] = move ? fast_exp2(m_run[h] - tmx) : 1.f;
                    if (move) m_run[h] = tmx;
                    any_move |= move;
                    l_run[h] *= alpha[h];
                }
                if (j > 0 && any_move) {  // the same decision in every thread (same tile maxima)
                    // O^T holds PV through tile j-1 once PV(j-1) completed (S(j) completed after PV(j-2)).
                    ok = !named_or_128(!mbar_wait(bar(B_PVDONE), static_cast<uint32_t>(j - 1) & 1u, abort_flag, wait_ns));
                    if (!ok) break;
                    tc_fence_after();
                    uint32_t o[NHP];
                    tmem_ld_cols<NHP>(tmem + lane_base + TM_O, o);
                    tmem_wait_ld();
#pragma unroll
                    for (int h = 0; h < NHP; ++h) o[h] = __float_as_uint(__uint_as_float(o[h]) * alpha[h]);
                    tmem_st_cols<NHP>(tmem + lane_base + TM_O, o);
                    tmem_wait_st();
                }
            }
            // P^T (bf16, row = head, column = key of the tile); padded heads stay zero
            uint8_t* pbuf = gb + L::OFF_P + (j & 1) * (2 * NH * 128);
#pragma unroll
            for (int h = 0; h < NHP; ++h) {
                if (h < C) {
                    const float m_ref = m_run[h] == -INFINITY ? 0.f : m_run[h];
                    const float p = fast_exp2(sc[h] - m_ref);
                    l_run[h] += p;
                    *reinterpret_cast<uint16_t*>(pbuf + sw_elem(h, t, NH)) = to_bf16(p);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(bar(B_PFULL0 + (j & 1)));
        }
        if (ok && n > 0) {
            // (PVDONE could be two phases behind here -- PV(n-2) may still run -- so the
            // epilogue waits on its own barrier, committed once after the last PV.)
            ok = !named_or_128(!mbar_wait(bar(B_OFULL), 0u, abort_flag, wait_ns));
        }
        if (ok && n > 0) {
            // row sums: every thread holds a partial over its keys
            const float wl = warp_reduce_halving<NHP, false>(l_run, lane);
            if (halving_leader<NHP>(lane)) ls[halving_owner<NHP>(lane) * 4 + warp] = wl;
            tc_fence_after();
            uint32_t o[NHP];
            tmem_ld_cols<NHP>(tmem + lane_base + TM_O, o);  // thread t = output dimension d
            tmem_wait_ld();
            named_sync_128();
            // the output (one split with tiles), the partial (m, l, acc) at slot s (global
            // merge), or (m, l, acc) staged in the idle V ring: read by the cluster's merge, or
            // written out below once the producer has taken this CTA's partial slot (waves)
            float* st_o = reinterpret_cast<float*>(gb + L::OFF_V);
            float2* st_ml = reinterpret_cast<float2*>(gb + L::OFF_V + NH * D * 4);
            const bool alone = !multi || (!waves && T == 1);
#pragma unroll
            for (int h = 0; h < NHP; ++h) {
                if (h < C) {
                    const float4 l4 = reinterpret_cast<const float4*>(ls)[h];
                    const float l_tot = (l4.x + l4.y) + (l4.z + l4.w);
                    if (alone) {
                        out[orow[h] * D + t] = to_bf16(__uint_as_float(o[h]) / l_tot);
                    } else if constexpr (MODE == kModeGlobal) {
                        const size_t row = crow[h] + s;
                        part_o[row * D + t] = __uint_as_float(o[h]);
                        if (t == 0) reinterpret_cast<float2*>(part_ml)[row] = make_float2(m_run[h], l_tot);
                    } else {
                        st_o[h * D + t] = __uint_as_float(o[h]);
                        if (t == 0) st_ml[h] = make_float2(m_run[h], l_tot);
                    }
                }
            }
        } else if (!ok) {
            *abort_flag = 1;
            atomicOr(err, kDevErrTimeout);
        }
    }

    // ---------------------------------------------------------------- merge of the splits
    if constexpr (MODE == kModeCluster) {
        // The nsplit CTAs of an item form a thread-block cluster (rank = split s).
        // The splits with tiles (s < min(nsplit, T)) have staged (m, l, acc) in shared
        // memory; after a cluster barrier every CTA merges its share of the dimensions,
        // reading its peers' staging directly, then waits at a second barrier until its own
        // staging has been read.  (T is the same in every CTA of the cluster, so all or none
        // of them take part.)
        if (hist_ok && multi && T > 1) {
            tc_fence_before();
            cluster_sync();
            if (s == 0 && tid == 0) *claim_ctr = 0;  // every split has made its last claim
            const int nw = min(nsplit, T);
            const int ds = (D + nsplit - 1) / nsplit;  // dimensions merged by this CTA
            const int d0 = s * ds, nd = max(0, min(D, d0 + ds) - d0);
            const uint32_t st_base = base + L::OFF_V;
            for (int p = tid; p < C * nd; p += kThreads) {
                const int h = p / nd, d = d0 + (p - h * nd);
                float mr[16], lr[16], orr[16];
#pragma unroll
                for (int r = 0; r < 16; ++r) {
                    if (r < nw) {
                        const uint32_t rb = mapa_shared(st_base, static_cast<uint32_t>(r));
                        const float2 ml = ld_dsmem_f32x2(rb + NH * D * 4 + h * 8);
                        mr[r] = ml.x;
                        lr[r] = ml.y;
                        orr[r] = ld_dsmem_f32(rb + (h * D + d) * 4);
                    }
                }
                float mm = -INFINITY;
#pragma unroll
                for (int r = 0; r < 16; ++r)
                    if (r < nw && lr[r] > 0.f) mm = fmaxf(mm, mr[r]);
                float l_tot = 0.f, acc = 0.f;
#pragma unroll
                for (int r = 0; r < 16; ++r)
                    if (r < nw && lr[r] > 0.f) {
                        const float wgt = fast_exp2(mr[r] - mm);
                        l_tot = fmaf(wgt, lr[r], l_tot);
                        acc = fmaf(wgt, orr[r], acc);
                    }
                out[orow[h] * D + d] = to_bf16(acc / l_tot);
            }
            cluster_sync();
        }
    } else if (hist_ok && multi) {
        bool contrib;  // (uniform over the CTA) this split wrote a partial and takes part
        if constexpr (WAVES) {
            tc_fence_before();
            __syncthreads();  // the staged result, and the producer's slot and claim count
            const int claimed = lastv[3];
            const float4* st_o4 = reinterpret_cast<const float4*>(gb + L::OFF_V);
            const float2* st_ml = reinterpret_cast<const float2*>(gb + L::OFF_V + NH * D * 4);
            contrib = claimed > 0 && claimed < T;
            if (claimed == T) {
                // this split took every tile: normalise straight from the staging
                for (int p = tid; p < C * (D / 4); p += kThreads) {
                    const int h = p / (D / 4), c = p % (D / 4);
                    const float4 v4 = st_o4[h * (D / 4) + c];
                    const float inv = 1.f / st_ml[h].y;
                    *reinterpret_cast<uint2*>(out + orow[h] * D + 4 * c) =
                        make_uint2(to_bf16(v4.x * inv) | (static_cast<uint32_t>(to_bf16(v4.y * inv)) << 16),
                                   to_bf16(v4.z * inv) | (static_cast<uint32_t>(to_bf16(v4.w * inv)) << 16));
                }
            } else if (contrib) {
                const int slot = lastv[2];
                for (int p = tid; p < C * (D / 4); p += kThreads) {
                    const int h = p / (D / 4), c = p % (D / 4);
                    reinterpret_cast<float4*>(part_o + (crow[h] + slot) * D)[c] = st_o4[h * (D / 4) + c];
                }
                if (tid < C) reinterpret_cast<float2*>(part_ml)[crow[tid] + slot] = st_ml[tid];
            }
        } else {
            contrib = s < T && T > 1;  // one wave: the softmax wrote the partial at slot s
        }
        if (contrib) {
            __threadfence();  // this CTA's partials are visible before it is counted
            tc_fence_before();
            __syncthreads();
            if (tid == 0) {
                // (contributors << 32 | tiles done): the split that completes the item's T tiles
                // merges, every contributor having counted itself after writing its partial
                if constexpr (WAVES) {
                    const int claimed = lastv[3];
                    const unsigned long long old =
                        atomicAdd(done_ctr, (1ull << 32) | static_cast<unsigned>(claimed));
                    const int last = static_cast<int>(old & 0xFFFFFFFFull) + claimed == T;
                    if (last) *done_ctr = 0ull;
                    lastv[0] = last;
                    lastv[1] = static_cast<int>(old >> 32) + 1;
                } else {
                    // one wave: the min(nsplit, T) splits with tiles count themselves (in the slot
                    // counter's place); the last of them merges and resets both counters, every
                    // claimer having counted itself
                    const int last = atomicAdd(slot_ctr, 1) == min(nsplit, T) - 1;
                    if (last) {
                        *slot_ctr = 0;
                        *claim_ctr = 0;
                    }
                    lastv[0] = last;
                    lastv[1] = min(nsplit, T);
                }
            }
            __syncthreads();
            tc_fence_after();
        }
        const int n_slots = lastv[1];
        if (contrib && lastv[0]) {
            // All six warps merge in one pass over the partials: warp w takes splits w, w+6, ...,
            // lane l dimensions 4l .. 4l+3 of every column, and keeps a running (M, L, acc) per
            // column, rescaled as a larger split maximum comes in; then the six warps' results
            // meet in shared memory (the idle K ring):
            //   wml  [6 warps][16] float2 (M_w, L_w);  racc [6 warps][16][D] float acc_w.
            // Splits without keys have l = 0 and are skipped; their accumulators were never
            // written, and what is read there is discarded by a select.
            __threadfence();
            float2* wml = reinterpret_cast<float2*>(gb + L::OFF_K);
            float* racc = reinterpret_cast<float*>(gb + L::OFF_K + (kThreads / 32) * NH * 8);
            float4 acc[NHP];
            float mw[NHP], lw[NHP];
#pragma unroll
            for (int h = 0; h < NHP; ++h) {
                acc[h] = make_float4(0.f, 0.f, 0.f, 0.f);
                mw[h] = -INFINITY;
                lw[h] = 0.f;
            }
            // (Every load is issued unconditionally -- padded columns re-read column C-1 --
            // so that the loads of a split for all columns are in flight together.)
#pragma unroll 2
            for (int sp = warp; sp < n_slots; sp += kThreads / 32) {
                float4 o4[NHP];
                float2 ml[NHP];
#pragma unroll
                for (int h = 0; h < NHP; ++h) {
                    const int hh = min(h, C - 1);
                    ml[h] = __ldcg(reinterpret_cast<const float2*>(part_ml) + crow[hh] + sp);
                    o4[h] = __ldcg(reinterpret_cast<const float4*>(part_o + (crow[hh] + sp) * D) + lane);
                }
#pragma unroll
                for (int h = 0; h < NHP; ++h) {
                    const bool use = h < C && ml[h].y > 0.f;
                    const float mn = use ? fmaxf(mw[h], ml[h].x) : mw[h];
                    const float a = use ? fast_exp2(mw[h] - mn) : 1.f;  // rescale of what came before
                    const float wgt = use ? fast_exp2(ml[h].x - mn) : 0.f;
                    acc[h].x = use ? fmaf(wgt, o4[h].x, acc[h].x * a) : acc[h].x;
                    acc[h].y = use ? fmaf(wgt, o4[h].y, acc[h].y * a) : acc[h].y;
                    acc[h].z = use ? fmaf(wgt, o4[h].z, acc[h].z * a) : acc[h].z;
                    acc[h].w = use ? fmaf(wgt, o4[h].w, acc[h].w * a) : acc[h].w;
                    lw[h] = use ? fmaf(wgt, ml[h].y, lw[h] * a) : lw[h];
                    mw[h] = mn;
                }
            }
#pragma unroll
            for (int h = 0; h < NHP; ++h)
                if (h < C) {
                    reinterpret_cast<float4*>(racc + (warp * NH + h) * D)[lane] = acc[h];
                    if (lane == 0) wml[warp * NH + h] = make_float2(mw[h], lw[h]);
                }
            __syncthreads();
            for (int p = tid; p < C * (D / 4); p += kThreads) {  // (column, 4 dimensions)
                const int h = p / (D / 4), c = p % (D / 4);
                float mm = -INFINITY;
#pragma unroll
                for (int w = 0; w < kThreads / 32; ++w) mm = fmaxf(mm, wml[w * NH + h].x);
                float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
                float l_tot = 0.f;
#pragma unroll
                for (int w = 0; w < kThreads / 32; ++w) {
                    const float2 m_l = wml[w * NH + h];
                    if (m_l.y > 0.f) {  // a warp without keys has M_w = -inf and nothing to add
                        const float f = fast_exp2(m_l.x - mm);
                        const float4 v4 = reinterpret_cast<const float4*>(racc + (w * NH + h) * D)[c];
                        sum.x = fmaf(f, v4.x, sum.x);
                        sum.y = fmaf(f, v4.y, sum.y);
                        sum.z = fmaf(f, v4.z, sum.z);
                        sum.w = fmaf(f, v4.w, sum.w);
                        l_tot = fmaf(f, m_l.y, l_tot);
                    }
                }
                const float inv = 1.f / l_tot;
                const uint2 packed = make_uint2(
                    to_bf16(sum.x * inv) | (static_cast<uint32_t>(to_bf16(sum.y * inv)) << 16),
                    to_bf16(sum.z * inv) | (static_cast<uint32_t>(to_bf16(sum.w * inv)) << 16));
                *reinterpret_cast<uint2*>(out + orow[h] * D + 4 * c) = packed;
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

}  // namespace

// How many clusters of each size (2 .. 16 CTAs) of the one-wave decode fit on the device at
// once, per device, set by configure_decode_tc; 0 where the size is refused.
constexpr int kMaxDevices = 64;
constexpr int kMaxCluster = 16;
int g_cluster_fit[kMaxDevices][kMaxCluster + 1] = {};

#define DECODE_TC_MODES(NHP, MAXTOK)                                                          \
    decode_tc_kernel<NHP, MAXTOK, kModeGlobal>, decode_tc_kernel<NHP, MAXTOK, kModeCluster>, \
        decode_tc_kernel<NHP, MAXTOK, kModeWaves>

cudaError_t configure_decode_tc() {
    cudaError_t e = cudaSuccess;
    for (auto fn : {DECODE_TC_MODES(8, 1), DECODE_TC_MODES(16, 1), DECODE_TC_MODES(8, kMaxTok),
                    DECODE_TC_MODES(16, kMaxTok)})
        if (e == cudaSuccess) e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, L::ALLOC);
    for (auto fn : {decode_tc_kernel<8, 1, kModeCluster>, decode_tc_kernel<16, 1, kModeCluster>,
                    decode_tc_kernel<8, kMaxTok, kModeCluster>, decode_tc_kernel<16, kMaxTok, kModeCluster>})
        if (e == cudaSuccess) e = cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    int dev = 0;
    if (e == cudaSuccess) e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    // (the four cluster instantiations share the block size, shared memory and one block per SM)
    for (int c = 2; c <= kMaxCluster; ++c) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(static_cast<unsigned>(c), 1, 1);
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = L::ALLOC;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = static_cast<unsigned>(c);
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, decode_tc_kernel<8, 1, kModeCluster>, &cfg) != cudaSuccess) {
            n = 0;
            cudaGetLastError();  // a refused size is never used
        }
        g_cluster_fit[dev][c] = n;
    }
    return cudaSuccess;
}

namespace {
// Whether `items` clusters of nsplit CTAs all fit on the current device at once.
bool decode_tc_clusters_fit(int nsplit, long long items) {
    int dev = 0;
    if (nsplit < 2 || nsplit > kMaxCluster || cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return false;
    return items <= g_cluster_fit[dev][nsplit];
}
}  // namespace

// Split counts.  With at most half as many (sequence, kv head, column group) items as SMs,
// one wave of CTAs, min(16, floor(SMs / items)) splits per item, each starting with its own
// tile.
// With more items, kWaveSplits splits per item over several waves: split 0 of every item
// comes first and the later splits, dispatched as SMs free up, claim what their items
// still have (nothing, for an item that is done), so long sequences in a batch of mixed
// lengths get help once the short ones finish.
constexpr int kWaveSplits = 3;
// One wave: at most 16 splits per item.  The long decode (8 items) measured 29.5 us with 16
// splits, 30.4-30.8 us with 19 (one per SM), 32.5 with 12 and 42 with 8: past 16 the extra
// partials and the later last CTA cost more than the SMs add.
constexpr long kMaxWaveSplits1 = 16;

int decode_tc_column_groups(int G, int ntok) { return (G * ntok + NH - 1) / NH; }

int decode_tc_num_splits(const Shape& s, int num_sms, int ncg, int ntok) {
    const long items = static_cast<long>(s.batch) * s.n_kv_heads * ncg;
    const long max_tiles = std::max(1L, static_cast<long>((s.max_len + KT - 1) / KT));
    long ns = 2 * items > num_sms ? kWaveSplits : std::min<long>(kMaxWaveSplits1, num_sms / items);
    ns = std::min(ns, std::min(max_tiles, 256L));
    // The last split of an item merges ns partials of up to 16 columns in the global merge,
    // while a cluster spreads the merge over its CTAs.  Fewer splits whose clusters fit on the
    // device pay for their longer streams with several new tokens from 128 partial rows
    // (splits x columns) on (B1 Hq32, 8188 history tokens: 4 tokens 31.5 -> 25.3 us, 8 tokens
    // 34.2 -> 31.9 us; Hq40 over 32765, 3 tokens 44.1 -> 41.6 us; but 8 tokens there, 6 splits x
    // 16 columns, went from 68.3 to 75.8 us with 5), and with one token when the cache holds
    // at most 64 tiles (B1 Hq32 over 1024 and 4096 tokens: 11.8 -> 10.3 us and 14.1 -> 12.9 us;
    // at 32767 tokens 12 splits took 32.5 us against 29.5 us with 16).
    const long cols = std::min<long>(NH, static_cast<long>(s.n_q_heads / s.n_kv_heads) * ntok);
    if (2 * items <= num_sms && ((ntok > 1 && ns * cols >= 128) || (ntok == 1 && max_tiles <= 64)))
        while (ns > 2 && !decode_tc_clusters_fit(static_cast<int>(ns), items)) --ns;
    return static_cast<int>(std::max(1L, ns));
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
                             const uint16_t* v_new, const int32_t* d_hist, int hist_add, uint16_t* k_cache,
                             uint16_t* v_cache, const float* cos_tab, const float* sin_tab, float* part_o,
                             float* part_ml, int* counters, int nsplit, uint16_t* out, int* err, bool after_decode,
                             int ntok, cudaStream_t st, bool producer_early, uint64_t wait_ns, int num_sms) {
    const float scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(D)));
    const int G = s.n_q_heads / s.n_kv_heads;
    const int ncg = decode_tc_column_groups(G, ntok);
    // every split starts with its own tile when the grid is one wave, else only split 0
    const long long ctas = static_cast<long long>(s.n_kv_heads) * s.batch * ncg * nsplit;
    const int s0 = ctas <= num_sms ? nsplit : 1;
    const dim3 grid = s0 == nsplit ? dim3(static_cast<unsigned>(nsplit), static_cast<unsigned>(s.n_kv_heads),
                                          static_cast<unsigned>(s.batch * ncg))
                                   : dim3(static_cast<unsigned>(s.n_kv_heads), static_cast<unsigned>(s.batch * ncg),
                                          static_cast<unsigned>(nsplit));
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = L::ALLOC;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    unsigned n_attr = 0;
    // dependent launch only right after another decode step, or with producer_early
    if (after_decode || producer_early) {
        attr[n_attr].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[n_attr].val.programmaticStreamSerializationAllowed = 1;
        ++n_attr;
    }
    const bool w = s0 < nsplit;
    // one wave: the splits of an item are one cluster (their merge) when a cluster per item
    // fits on the device at once, else they merge through global memory
    const int mode = w ? kModeWaves
                       : (decode_tc_clusters_fit(nsplit, static_cast<long long>(s.n_kv_heads) * s.batch * ncg)
                              ? kModeCluster
                              : kModeGlobal);
    if (mode == kModeCluster) {
        attr[n_attr].id = cudaLaunchAttributeClusterDimension;
        attr[n_attr].val.clusterDim.x = static_cast<unsigned>(nsplit);
        attr[n_attr].val.clusterDim.y = 1;
        attr[n_attr].val.clusterDim.z = 1;
        ++n_attr;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n_attr;
    if (ntok < 1 || ntok > kMaxTok || G > NH) return cudaErrorInvalidValue;
    using Kernel = decltype(&decode_tc_kernel<8, 1, kModeGlobal>);
    static const Kernel kernels[4][3] = {{DECODE_TC_MODES(8, 1)},
                                         {DECODE_TC_MODES(16, 1)},
                                         {DECODE_TC_MODES(8, kMaxTok)},
                                         {DECODE_TC_MODES(16, kMaxTok)}};
    const Kernel kernel = kernels[ntok == 1 ? (G <= 8 ? 0 : 1) : (G * ntok <= 8 ? 2 : 3)][mode];
    return cudaLaunchKernelEx(&cfg, kernel, maps.k, maps.v, q,
                              k_new, v_new, d_hist, hist_add, ntok, k_cache, v_cache, cos_tab, sin_tab, s.n_q_heads,
                              s.n_kv_heads, s.max_len, nsplit, scale_log2, part_o, part_ml, counters, out, err,
                              producer_early ? 1 : 0, wait_ns, ncg, after_decode ? 0 : 1, s0);
}

}  // namespace attn

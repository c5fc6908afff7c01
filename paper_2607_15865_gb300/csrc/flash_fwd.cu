// flash_fwd.cu -- K2: causal flash attention for prefill and prefill_kv on sm_103a.
//
// What it computes (Sections 4.2-4.3; FAttention of Section 2.2 with the causal
// mask of Section 4.6.1): for the chunk's query rows i at positions p = hist + i
// and every query head h, out[b, i, h, :] = softmax_j(q_rot . k_j / sqrt(D)) v_j
// over cache slots j <= p of kv head h / G.  The caches already hold the chunk's
// rotated keys and values (K1 runs first), so the history and the new tokens are
// one contiguous key range [0, hist + chunk) -- the "Concat" of Listing 2 is the
// in-place layout itself.  prefill is the same kernel with hist = 0 (the paper's
// with_history template, Section 4.2).
//
// Design.  A persistent CTA per SM walks a static list of work items sorted
// longest-first, dealt out in rounds of alternating direction.  An item is two 128-row query tiles (A, B) of one head, so each
// K/V tile is brought in once for 256 queries.  384 threads, three warpgroups:
//   WG0 (warps 0-3)   softmax + epilogue of tile A (one thread per row = TMEM lane)
//   WG1 (warps 4-7)   softmax + epilogue of tile B
//   WG2 (warps 8-11)  warp 8: TMA producer (lane 0: q tiles from a 4-D map of
//                     q [B,S,Hq,D] and the K/V group ring), warp 9: tcgen05
//                     issuer, warps 10-11 idle.  WG2 gives registers to
//                     the softmax warpgroups (setmaxnreg 96 / 200 of 168 at launch).
// K and V tiles (128 keys, a 2-stage ring of K(j)/V(j-1) groups) use the 128-byte
// swizzle; rows past hist+chunk are zero-filled by the map bounds, never read.
// Per KV tile j the issuer runs PV_A(j-1), S_A(j), PV_B(j-1), S_B(j).
// TMEM (512 columns): S_A [0,128) S_B [128,256) O_A [256,256+D) O_B [256+D,256+2D).
// P is written back as bf16 over the first 64 columns of its S and fed to the PV
// MMA from TMEM, so the two warpgroups ping-pong: while one turns its scores into
// P, the tensor core runs the other tile's MMAs.  A commit covers every earlier
// MMA of the issuing thread, so "S_T(j) complete" implies "PV_T(j-1) complete":
// the softmax warpgroup may rescale O_T before it hands P over.  O is rescaled lazily
// (only when the running max grows by more than 2^8, exact in value).
// Per row: RoPE of the q row in shared memory before the first MMA (cos/sin
// gathered by position from copies of the tables laid out in groups of four pairs,
// Section 4.6.2, float arithmetic and bf16 rounding as K1),
// scores from TMEM, causal mask by index compare on diagonal tiles (no mask
// tensor), online softmax in the log2 domain, O / l -> bf16 -> out.
// Every wait is bounded; on expiry the CTA records kDevErrTimeout, lets its
// in-flight copies and MMAs finish, releases TMEM and exits.
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>
#include <vector>

#include "internal.h"
#include "sm100_ptx.cuh"

namespace attn {
namespace {

constexpr int BM = 128;  // query rows per tile (TMEM lanes)
constexpr int BN = 128;  // keys per KV tile
constexpr int kThreads = 384;
constexpr int kWarpTma = 8;
constexpr int kWarpMma = 9;
constexpr uint32_t kTmemCols = 512;
// K/V ring of "groups": group j holds K tile j and V tile j-1, the operands of KV step
// j (S(j) and PV(j-1)), so the issuer waits on one barrier and releases one slot per
// step -- each satisfied wait or extra commit of the issuing thread idles the tensor
// core for about 100 cycles.  Two 64 KB slots, and 32 KB to stage the epilogue's output
// (each warp store then writes 4 whole 128-byte rows instead of 16 bytes of 32 rows
// 10 KB apart).
constexpr int GS = 2;
// Register budgets: 168 per thread at launch (65536 / 384, rounded down to 8);
// WG2 gives back 72 per thread, the two softmax warpgroups take 32 each.  The MMA
// issuer must not spill: a local-memory reload between two MMA groups idles the
// tensor core (56 for WG2 cost 8% of the prefill_kv time against 96), and at 200 the
// softmax fits because O is rescaled after its scores have been consumed.
constexpr int kLaunchRegs = 168;
constexpr uint32_t kRegsLow = 96;
constexpr uint32_t kRegsHigh = 200;
static_assert(128 * kRegsLow + 256 * kRegsHigh <= kThreads * kLaunchRegs, "register split exceeds the launch total");

enum Bar {
    B_QFULL, B_QREADY, B_QEMPTY,
    B_GFULL0, B_GEMPTY0 = B_GFULL0 + GS,
    B_SFULL0 = B_GEMPTY0 + GS, B_SFULL1, B_PFULL0, B_PFULL1,
    B_OFULL0, B_OFULL1, B_OEMPTY0, B_OEMPTY1,
    B_DRAIN, NBAR
};

template <int D>
struct Layout {
    static constexpr int DCH = D / 64;       // 64-column (128-byte) chunks of a row
    static constexpr int CHUNK = 128 * 128;  // bytes of one 128-row x 128-byte chunk
    static constexpr int Q_TILE = DCH * CHUNK;
    static constexpr int KV_TILE = DCH * CHUNK;
    static constexpr int OFF_Q = 0;                      // q tiles A, B
    static constexpr int OFF_G = OFF_Q + 2 * Q_TILE;     // group ring: slot = K tile, V tile
    static constexpr int G_SLOT = 2 * KV_TILE;
    static constexpr int OFF_STAGE = OFF_G + GS * G_SLOT;  // epilogue staging, 4 KB per softmax warp
    static constexpr int STAGE_WARP = 32 * 128;             // 32 rows x 64 bf16 columns
    static constexpr int OFF_BAR = OFF_STAGE + 8 * STAGE_WARP;
    static constexpr int OFF_TMEM = OFF_BAR + NBAR * 8;
    static constexpr int OFF_ABORT = OFF_TMEM + 8;
    static constexpr int BYTES = OFF_ABORT + 8;
    static constexpr int ALLOC = BYTES + 1024;  // slack to align the base to 1024 bytes
    static constexpr uint32_t TM_O = 2 * BN;    // TMEM column of O_A; O_B at TM_O + D
};
static_assert(Layout<128>::ALLOC <= 232448, "shared memory budget of one CTA");

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// Byte offset of the 16-byte unit holding columns [col, col+8) of row `row` inside a
// 128-row tile stored as 128-byte-swizzled 64-column chunks (TMA SWIZZLE_128B).
__device__ __forceinline__ uint32_t sw128_offset(int row, int col) {
    const int chunk = col >> 6;
    const int unit = (col & 63) >> 3;
    return static_cast<uint32_t>(chunk * (128 * 128) + row * 128 + ((unit ^ (row & 7)) << 4));
}

// One work item: query tiles A (rows q0(0)..) and B (rows q0(1)..) of head h, sequence b.
// Scalar fields with select accessors keep every field in registers when the tile
// index is only known at run time.
struct Item {
    int h, b, g;
    int q0a, q0b;
    int rowsa, rowsb;  // valid rows of each tile (0: tile absent)
    int nkva, nkvb;    // KV tiles each tile attends to
    int n_kv;          // KV tiles loaded for the item
    __device__ __forceinline__ int q0(int t) const { return t ? q0b : q0a; }
    __device__ __forceinline__ int rows(int t) const { return t ? rowsb : rowsa; }
    __device__ __forceinline__ int nkv(int t) const { return t ? nkvb : nkva; }
};

// The launch's work list: chunk S at history H, Hq query heads, batch sequences, n_pairs
// query-tile pairs per (head, sequence); `head` items whole, the rest cut into nsplit
// pieces; with the divisors the kernels use, as fast divisions (every division of the
// schedule ran as a generic integer division before: about 1 us per decoded unit).
struct Sched {
    int S, H, Hq, G, batch, n_pairs, head, nsplit, n_units;
    int kvb;  // item order: 0 longest pairs first over all heads, else blocks of kvb kv heads
    FastDiv fd_grid, fd_hqb, fd_hq, fd_g, fd_ns, fd_pb, fd_per, fd_nb;
};

// Item order.  By default the longest query-tile pairs come first across every (head,
// sequence), so a causal launch starts its longest items first and ends with the
// shortest.  When a long history makes the items about equally long and the K/V the
// launch reads is a large part of L2, the items are grouped in blocks of kvb kv heads of
// one sequence instead -- within a block longest pairs first, the block's query heads of
// a pair together -- so the CTAs of a round walk the K/V of only those kv heads, which
// stays in L2, and each kv head's cache is read from DRAM about once instead of once per
// round.
__device__ __forceinline__ Item decode_item(int lin, const Sched& sc) {
    Item it;
    int qt;
    if (sc.kvb) {
        const int per = sc.kvb * sc.G;        // query heads of a block
        const int blk = fdiv(lin, sc.fd_pb);  // (sequence, block of kv heads)
        const int r = lin - blk * (sc.n_pairs * per);
        qt = fdiv(r, sc.fd_per);
        it.b = fdiv(blk, sc.fd_nb);
        it.h = (blk - it.b * fdiv(sc.Hq, sc.fd_per)) * per + (r - qt * per);
        it.g = fdiv(it.h, sc.fd_g);
    } else {
        qt = fdiv(lin, sc.fd_hqb);
        const int rem = lin - qt * (sc.Hq * sc.batch);
        it.b = fdiv(rem, sc.fd_hq);
        it.h = rem - it.b * sc.Hq;
        it.g = fdiv(it.h, sc.fd_g);
    }
    const int pt = sc.n_pairs - 1 - qt;
    it.q0a = pt * 2 * BM;
    it.q0b = it.q0a + BM;
    it.rowsa = max(0, min(BM, sc.S - it.q0a));
    it.rowsb = max(0, min(BM, sc.S - it.q0b));
    it.nkva = it.rowsa ? (sc.H + it.q0a + it.rowsa + BN - 1) / BN : 0;
    it.nkvb = it.rowsb ? (sc.H + it.q0b + it.rowsb + BN - 1) / BN : 0;
    it.n_kv = max(it.nkva, it.nkvb);
    return it;
}

// A work unit: a whole item, or one KV-range piece of an item from the tail of the
// list.  Items fill whole rounds of CTAs first (`head` of them); the remaining
// items are cut into `nsplit` pieces each, so every CTA ends at about the same
// time.  Pieces write unnormalised partial results that a second kernel merges.
struct Unit {
    Item it;
    int kv_lo, kv_hi;  // KV tiles [kv_lo, kv_hi) of the item
    int piece;         // index of the piece in the partial workspace, -1 for a whole item
    __device__ __forceinline__ int cnt(int t) const { return max(0, min(kv_hi, it.nkv(t)) - kv_lo); }
};

__device__ __forceinline__ Unit decode_unit(int lin, const Sched& sc) {
    Unit u;
    u.piece = -1;
    if (lin >= sc.head && sc.nsplit > 1) {
        const int v = lin - sc.head;
        const int tail = fdiv(v, sc.fd_ns);
        const int s = v - tail * sc.nsplit;
        u.piece = v;
        u.it = decode_item(sc.head + tail, sc);
        u.kv_lo = fdiv(u.it.n_kv * s, sc.fd_ns);
        u.kv_hi = fdiv(u.it.n_kv * (s + 1), sc.fd_ns);
    } else {
        u.it = decode_item(lin, sc);
        u.kv_lo = 0;
        u.kv_hi = u.it.n_kv;
    }
    return u;
}

// Unit taken by a CTA in its round r = lin / gridDim.x.  Rounds alternate direction
// (odd rounds reversed), so the CTA that took one of the longest units of a round takes
// one of the shortest of the next: with items sorted longest-first this evens out the
// CTAs' totals (causal prefill 4096, 40 heads: the slowest CTA walks 74 KV tiles instead
// of 88).  The last, partial round keeps its order.  A bijection on [0, n_units).
__device__ __forceinline__ int unit_of(int lin, const Sched& sc) {
    const int g = static_cast<int>(gridDim.x), r = fdiv(lin, sc.fd_grid);
    if ((r & 1) == 0 || (r + 1) * g > sc.n_units) return lin;
    return r * g + (g - 1 - (lin - r * g));
}

// RoPE tables of one position in registers: cos/sin of pairs j = 0 .. D/2-1.  They are
// read from copies of the tables in groups of four pairs ([D/8][max_len][4]: entry (j, p)
// at ((j / 4) * stride + p) * 4 + j % 4), so that a thread loads four pairs at once and
// the 32 threads of a warp -- 32 consecutive positions -- read 512 contiguous bytes per
// load: D/4 loads per thread instead of D with one float per pair, which took about 2 us
// per work unit (the loads in flight, not the bytes, were the limit).  They are loaded
// before the q tile lands.
template <int D>
struct RopeRow {
    float c[D / 2], s[D / 2];
};

template <int D>
__device__ __forceinline__ void rope_load(RopeRow<D>& t, int pos, const float* __restrict__ cos_t,
                                          const float* __restrict__ sin_t, int stride) {
    const float4* c4 = reinterpret_cast<const float4*>(cos_t) + pos;
    const float4* s4 = reinterpret_cast<const float4*>(sin_t) + pos;
#pragma unroll
    for (int g = 0; g < D / 8; ++g) {
        const float4 c = __ldg(c4 + static_cast<size_t>(g) * stride);
        const float4 s = __ldg(s4 + static_cast<size_t>(g) * stride);
        t.c[4 * g] = c.x;
        t.c[4 * g + 1] = c.y;
        t.c[4 * g + 2] = c.z;
        t.c[4 * g + 3] = c.w;
        t.s[4 * g] = s.x;
        t.s[4 * g + 1] = s.y;
        t.s[4 * g + 2] = s.z;
        t.s[4 * g + 3] = s.w;
    }
}

// RoPE of one q row of a tile in shared memory (pairs j, j + D/2, with the tables of
// its position; float arithmetic with each product and the difference/sum rounded
// separately, bf16 result), as K1 applies to keys.
template <int D>
__device__ __forceinline__ void rope_row_smem(uint8_t* qtile, int row, const RopeRow<D>& t) {
    constexpr int HALF = D / 2;
#pragma unroll
    for (int u = 0; u < HALF / 8; ++u) {
        const int jlo = 8 * u;
        uint4* plo = reinterpret_cast<uint4*>(qtile + sw128_offset(row, jlo));
        uint4* phi = reinterpret_cast<uint4*>(qtile + sw128_offset(row, jlo + HALF));
        const uint4 xa = *plo, xb = *phi;
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
                const float cc = t.c[jlo + 2 * e + k2], ss = t.s[jlo + 2 * e + k2];
                lo[k2] = __fsub_rn(__fmul_rn(a, cc), __fmul_rn(bb, ss));
                hi[k2] = __fadd_rn(__fmul_rn(bb, cc), __fmul_rn(a, ss));
            }
            ya[e] = pack_bf16x2(lo[0], lo[1]);
            yb[e] = pack_bf16x2(hi[0], hi[1]);
        }
        *plo = make_uint4(ya[0], ya[1], ya[2], ya[3]);
        *phi = make_uint4(yb[0], yb[1], yb[2], yb[3]);
    }
}

// Wait for an item's q tiles, rotate this thread's row, hand Q to the MMA warp.
template <int D>
__device__ __forceinline__ bool rope_item(uint32_t qfull, uint32_t qready, uint32_t parity, const volatile int* abort,
                                          uint8_t* qtile, int row, int rows, int pos0,
                                          const float* __restrict__ cos_t, const float* __restrict__ sin_t,
                                          int stride, uint64_t wait_ns) {
    RopeRow<D> tabs;
    rope_load<D>(tabs, row < rows ? pos0 + row : pos0, cos_t, sin_t, stride);
    const bool w = __all_sync(0xFFFFFFFFu, mbar_wait(qfull, parity, abort, wait_ns));
    if (w && row < rows) rope_row_smem<D>(qtile, row, tabs);
    fence_proxy_async_smem();
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(qready);
    return w;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    flash_fwd_kernel(const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_k,
                     const __grid_constant__ CUtensorMap map_v, const Sched sc, int s_stride, int Hkv,
                     float scale_log2, const float* __restrict__ cos_t,
                     const float* __restrict__ sin_t, int tab_stride, uint16_t* __restrict__ out, float* __restrict__ ws_o,
                     float* __restrict__ ws_ml, int* __restrict__ err, uint64_t wait_ns) {
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
    const int S = sc.S, H = sc.H, Hq = sc.Hq, n_units = sc.n_units;

    if (warp == kWarpTma && lane == 0) {
        // Barriers, then the first unit's q tiles right away: their copy overlaps the TMEM
        // allocation and the register hand-over (q is the caller's input, complete before
        // K1 began, so it may be read before this grid waits on K1).
        *abort_flag = 0;
        mbar_init(bar(B_QFULL), 1);
        mbar_init(bar(B_QREADY), 2 * BM / 32);
        mbar_init(bar(B_QEMPTY), 1);
        for (int st = 0; st < GS; ++st) {
            mbar_init(bar(B_GFULL0 + st), 1);
            mbar_init(bar(B_GEMPTY0 + st), 1);
        }
        for (int t = 0; t < 2; ++t) {
            mbar_init(bar(B_SFULL0 + t), 1);
            mbar_init(bar(B_PFULL0 + t), BM / 32);  // one arrive per softmax warp
            mbar_init(bar(B_OFULL0 + t), 1);
            mbar_init(bar(B_OEMPTY0 + t), BM / 32);
        }
        mbar_init(bar(B_DRAIN), 1);
        fence_mbar_init();
        tma_prefetch_desc(&map_q);
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_v);
        if (static_cast<int>(blockIdx.x) < n_units) {
            const Item it = decode_unit(unit_of(blockIdx.x, sc), sc).it;
            mbar_arrive_expect_tx(bar(B_QFULL), 2 * L::Q_TILE);
#pragma unroll
            for (int t = 0; t < 2; ++t)
#pragma unroll
                for (int c = 0; c < L::DCH; ++c)
                    tma_load_4d(base + L::OFF_Q + t * L::Q_TILE + c * L::CHUNK, &map_q, c * 64, it.h, it.q0(t),
                                it.b, bar(B_QFULL));
        }
    }
    if (warp == kWarpMma) {
        tmem_alloc(base + L::OFF_TMEM, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    griddep_launch_dependents();  // the merge kernel waits for this whole grid before reading

    if (warp >= 8) {
        warpgroup_reg_dec<kRegsLow>();
        if (warp == kWarpTma && lane == 0) {
            // ---------------------------------------------------- q tiles and the group ring
            // A unit of n KV tiles takes n + 1 groups: group j holds K(j) (j < kv_hi) and
            // V(j-1) (j > kv_lo), the last one only the V the final PV reads.
            uint32_t gc = 0;  // groups issued
            int items = 0;
            bool ok = true;
            bool kv_visible = false;  // K1's cache writes complete (dependent launch)
            for (int lin = blockIdx.x; lin < n_units && ok; lin += gridDim.x) {
                const Unit un = decode_unit(unit_of(lin, sc), sc);
                const Item& it = un.it;
                if (items > 0) {  // (the first unit's q tiles were issued in the prologue)
                    if (!mbar_wait(bar(B_QEMPTY), static_cast<uint32_t>(items - 1) & 1u, abort_flag, wait_ns)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(bar(B_QFULL), 2 * L::Q_TILE);
#pragma unroll
                    for (int t = 0; t < 2; ++t)
#pragma unroll
                        for (int c = 0; c < L::DCH; ++c)
                            tma_load_4d(base + L::OFF_Q + t * L::Q_TILE + c * L::CHUNK, &map_q, c * 64, it.h,
                                        it.q0(t), it.b, bar(B_QFULL));
                }
                ++items;
                {
                    // the next unit's q tiles into L2, so that their copy after this unit is short
                    const int nxt = lin + static_cast<int>(gridDim.x);
                    if (nxt < n_units) {
                        const Item nt = decode_unit(unit_of(nxt, sc), sc).it;
#pragma unroll
                        for (int t = 0; t < 2; ++t)
                            if (nt.rows(t) > 0)
#pragma unroll
                                for (int c = 0; c < L::DCH; ++c) tma_prefetch_l2_4d(&map_q, c * 64, nt.h, nt.q0(t), nt.b);
                    }
                }
                const int kv_row = it.b * Hkv + it.g;
                if (!kv_visible) {
                    // This grid may start while K1 still appends the chunk's k and v: the q
                    // copy and its RoPE (inputs of the caller, complete before K1 began) overlap
                    // K1's tail; the first cache read waits for K1.
                    griddep_wait();
                    kv_visible = true;
                }
                for (int j = un.kv_lo; j <= un.kv_hi; ++j, ++gc) {
                    const int st = static_cast<int>(gc % GS);
                    if (gc >= GS && !mbar_wait(bar(B_GEMPTY0 + st), (gc / GS - 1u) & 1u, abort_flag, wait_ns)) {
                        ok = false;
                        break;
                    }
                    const bool has_k = j < un.kv_hi, has_v = j > un.kv_lo;
                    const uint32_t slot = base + L::OFF_G + st * L::G_SLOT;
                    mbar_arrive_expect_tx(bar(B_GFULL0 + st), (has_k ? L::KV_TILE : 0) + (has_v ? L::KV_TILE : 0));
                    if (has_k) {
#pragma unroll
                        for (int c = 0; c < L::DCH; ++c)
                            tma_load_3d(slot + c * L::CHUNK, &map_k, c * 64, j * BN, kv_row, bar(B_GFULL0 + st));
                    }
                    if (has_v) {
#pragma unroll
                        for (int c = 0; c < L::DCH; ++c)
                            tma_load_3d(slot + L::KV_TILE + c * L::CHUNK, &map_v, c * 64, (j - 1) * BN, kv_row,
                                        bar(B_GFULL0 + st));
                    }
                }
            }
            if (!ok) {
                *abort_flag = 1;
                atomicOr(err, kDevErrTimeout);
                // every copy issued must land before the CTA may exit
                if (items > 0) mbar_wait(bar(B_QFULL), static_cast<uint32_t>(items - 1) & 1u, nullptr);
                for (uint32_t t = gc >= GS ? gc - GS : 0; t < gc; ++t)
                    mbar_wait(bar(B_GFULL0 + static_cast<int>(t % GS)), (t / GS) & 1u, nullptr);
            }
        } else if (warp == kWarpMma && lane == 0) {
            // ---------------------------------------------------- tcgen05 issuer
            constexpr uint32_t kIdS = idesc_bf16_f32(BM, BN, false, false);
            constexpr uint32_t kIdPV = idesc_bf16_f32(BM, D, false, true);
            uint32_t gc = 0;  // groups consumed
            uint32_t p_cnt[2] = {0u, 0u};  // P tiles consumed per query tile
            uint32_t o_cnt[2] = {0u, 0u};  // items whose O was handed to the epilogue
            int items = 0;
            bool ok = true;
            // The tensor core holds almost no queue of MMAs, so every cycle this thread spends
            // between two MMAs is a cycle the tensor core idles: descriptors are precomputed
            // words plus constants, and each KV step waits on as few barriers as it can (the
            // V tile once for both query tiles).
            // Descriptor low words of the operand tiles; a K step adds a constant to them.
            constexpr uint32_t kHi = desc_hi_sw128(1024);
            const uint32_t q_lo0 = desc_lo_sw128(base + L::OFF_Q, 16);
            const uint32_t k_lo0 = desc_lo_sw128(base + L::OFF_G, 16);
            const uint32_t v_lo0 = desc_lo_sw128(base + L::OFF_G + L::KV_TILE, L::CHUNK);
            auto issue_s = [&](int t, uint32_t slot) {
                const uint32_t a_lo = q_lo0 + t * (L::Q_TILE >> 4);
                const uint32_t b_lo = k_lo0 + slot * (L::G_SLOT >> 4);
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t c = ((kk >> 2) * L::CHUNK + (kk & 3) * 32) >> 4;
                    umma_ss_w(tmem + t * BN, a_lo + c, kHi, b_lo + c, kHi, kIdS, kk > 0 ? 1u : 0u);
                }
                umma_commit(bar(B_SFULL0 + t));
            };
            auto issue_pv = [&](int t, bool first, uint32_t slot) {
                const uint32_t b_lo = v_lo0 + slot * (L::G_SLOT >> 4);
#pragma unroll
                for (int kk = 0; kk < BN / 16; ++kk)
                    umma_ts_w(tmem + L::TM_O + t * D, tmem + t * BN + kk * 8, b_lo + kk * ((16 * 128) >> 4), kHi, kIdPV,
                              (!first || kk > 0) ? 1u : 0u);
            };
            // P_t of the previous KV tile in TMEM, and O_t free when it is the unit's first PV
            auto wait_p = [&](int t, bool first) -> bool {
                if (!mbar_wait(bar(B_PFULL0 + t), p_cnt[t] & 1u, abort_flag, wait_ns)) return false;
                ++p_cnt[t];
                if (first && o_cnt[t] > 0 && !mbar_wait(bar(B_OEMPTY0 + t), (o_cnt[t] - 1u) & 1u, abort_flag, wait_ns))
                    return false;
                return true;
            };
            uint32_t gslot = 0;  // gc % GS
            auto next_group = [&]() {
                ++gc;
                gslot = gslot + 1 == GS ? 0 : gslot + 1;
            };
            for (int lin = blockIdx.x; lin < n_units && ok; lin += gridDim.x) {
                const Unit un = decode_unit(unit_of(lin, sc), sc);
                const Item& it = un.it;
                if (!mbar_wait(bar(B_QREADY), static_cast<uint32_t>(items) & 1u, abort_flag, wait_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                for (int j = un.kv_lo; j < un.kv_hi && ok; ++j) {
                    // group j: K(j), and V(j-1) for the PV MMAs of the previous tile
                    if (!mbar_wait(bar(B_GFULL0 + gslot), (gc / GS) & 1u, abort_flag, wait_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const bool pv_a = j > un.kv_lo && j - 1 < it.nkv(0), pv_b = j > un.kv_lo && j - 1 < it.nkv(1);
                    const bool s_a = j < it.nkv(0), s_b = j < it.nkv(1);
                    const bool first = j - 1 == un.kv_lo;
                    if (pv_a) {
                        if (!wait_p(0, first)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        issue_pv(0, first, gslot);
                    }
                    if (s_a) issue_s(0, gslot);
                    if (pv_b) {
                        if (!wait_p(1, first)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        issue_pv(1, first, gslot);
                    }
                    if (s_b) issue_s(1, gslot);
                    umma_commit(bar(B_GEMPTY0 + gslot));
                    next_group();
                }
                if (!ok) break;
                umma_commit(bar(B_QEMPTY));  // every S MMA of the unit is issued
                // the last group: V of the final tile
                if (!mbar_wait(bar(B_GFULL0 + gslot), (gc / GS) & 1u, abort_flag, wait_ns)) ok = false;
                tc_fence_after();
#pragma unroll
                for (int t = 0; t < 2; ++t)
                    if (ok && un.kv_hi - 1 < it.nkv(t)) {
                        if (!wait_p(t, un.kv_hi - 1 == un.kv_lo)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        issue_pv(t, un.kv_hi - 1 == un.kv_lo, gslot);
                    }
                if (!ok) break;
                umma_commit(bar(B_GEMPTY0 + gslot));
                next_group();
#pragma unroll
                for (int t = 0; t < 2; ++t)
                    if (un.cnt(t) > 0) {
                        umma_commit(bar(B_OFULL0 + t));
                        ++o_cnt[t];
                    }
                ++items;
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
        // ------------------------------------------------------------ softmax / epilogue warpgroups
        warpgroup_reg_inc<kRegsHigh>();
        const int t = warp >> 2;            // query tile of this warpgroup
        const int row = threadIdx.x & 127;  // row in the tile == TMEM lane
        const uint32_t lane_base = static_cast<uint32_t>((warp & 3) * 32) << 16;
        const uint32_t s_col = tmem + lane_base + t * BN;
        const uint32_t o_col = tmem + lane_base + L::TM_O + t * D;
        uint8_t* qtile = gbase + L::OFF_Q + t * L::Q_TILE;
        uint32_t s_cnt = 0, o_cnt = 0;
        int items = 0;
        bool ok = true;

        int lin = blockIdx.x;
        Unit un;
        if (lin < n_units) {
            un = decode_unit(unit_of(lin, sc), sc);
            ok = rope_item<D>(bar(B_QFULL), bar(B_QREADY), static_cast<uint32_t>(items) & 1u, abort_flag, qtile, row,
                              un.it.rows(t), H + un.it.q0(t), cos_t, sin_t, tab_stride, wait_ns);
            ++items;
        }
        while (lin < n_units && ok) {
            const Item& it = un.it;
            float m_run = -INFINITY;  // reference max of P (log2 domain)
            float l_run = 0.f;
            const int pos_row = H + it.q0(t) + row;  // last key this row may see
            const int min_pos = H + it.q0(t);        // smallest row position of the tile
            const int n_tiles = un.cnt(t);
            for (int j = un.kv_lo; j < un.kv_lo + n_tiles; ++j) {
                ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_SFULL0 + t), s_cnt & 1u, abort_flag, wait_ns));
                if (!ok) break;
                ++s_cnt;
                tc_fence_after();
                uint32_t r[BN / 32][32];
#pragma unroll
                for (int c = 0; c < BN / 32; ++c) tmem_ld32(s_col + 32 * c, r[c]);
                tmem_wait_ld();
                const int kb = j * BN;
                if (kb + BN - 1 > min_pos) {  // the tile crosses the diagonal: mask by index
#pragma unroll
                    for (int c = 0; c < BN / 32; ++c)
#pragma unroll
                        for (int e = 0; e < 32; ++e)
                            if (kb + 32 * c + e > pos_row) r[c][e] = __float_as_uint(-INFINITY);
                }
                // row max: four independent chains, one per 32-column chunk
                float mxc[BN / 32];
#pragma unroll
                for (int c = 0; c < BN / 32; ++c) {
                    mxc[c] = __uint_as_float(r[c][0]);
#pragma unroll
                    for (int e = 1; e < 31; e += 2)
                        mxc[c] = fmax3(mxc[c], __uint_as_float(r[c][e]), __uint_as_float(r[c][e + 1]));
                    mxc[c] = fmaxf(mxc[c], __uint_as_float(r[c][31]));
                }
                const float mx = fmaxf(fmaxf(mxc[0], mxc[1]), fmaxf(mxc[2], mxc[3]));
                const float m_cand = fmaxf(m_run, mx * scale_log2);
                const bool move = m_cand > m_run + 8.f;  // always on the first tile
                const float m_new = move ? m_cand : m_run;
                const float alpha = move ? fast_exp2(m_run - m_new) : 1.f;
                // P = 2^(s*scale - m) as bf16 pairs over the first 64 columns of S (keys 2c, 2c+1
                // in column c), stored a quarter (16 columns) at a time; the scores are all in
                // registers, so overwriting S is safe.  Row sums in independent accumulators.
                // A row of a piece may have seen no visible key yet (all masked): keep its
                // reference finite so that P, O and l stay 0 (the merge skips l = 0).
                const float m_ref = m_new == -INFINITY ? 0.f : m_new;
                const float2 sc2 = make_float2(scale_log2, scale_log2);
                const float2 nm2 = make_float2(-m_ref, -m_ref);
                float2 sum2[BN / 32];
#pragma unroll
                for (int c = 0; c < BN / 32; ++c) {
                    uint32_t pw[16];
                    float2 acc2 = make_float2(0.f, 0.f);
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const float2 x =
                            ffma2(make_float2(__uint_as_float(r[c][2 * i]), __uint_as_float(r[c][2 * i + 1])), sc2, nm2);
                        const float2 pp = make_float2(fast_exp2(x.x), fast_exp2(x.y));
                        acc2 = ffma2(pp, make_float2(1.f, 1.f), acc2);
                        pw[i] = pack_bf16x2(pp.x, pp.y);
                    }
                    sum2[c] = acc2;
                    tmem_st16(s_col + 16 * c, pw);
                }
                const float2 sum2a = make_float2(sum2[0].x + sum2[1].x, sum2[0].y + sum2[1].y);
                const float2 sum2b = make_float2(sum2[2].x + sum2[3].x, sum2[2].y + sum2[3].y);
                const float2 sum2t = make_float2(sum2a.x + sum2b.x, sum2a.y + sum2b.y);
                if (j > un.kv_lo && __any_sync(0xFFFFFFFFu, move)) {
                    // O_T holds the sum through tile j-1 (PV_T(j-1) completed before S_T(j)),
                    // and PV_T(j) waits for this thread's arrive below.  Done after P, when the
                    // scores no longer hold registers.
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) {
                        uint32_t o[32];
                        tmem_ld32(o_col + 32 * c, o);
                        tmem_wait_ld();
#pragma unroll
                        for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
                        tmem_st32(o_col + 32 * c, o);
                    }
                }
                tmem_wait_st();
                l_run = l_run * alpha + (sum2t.x + sum2t.y);
                m_run = m_new;
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(B_PFULL0 + t));
            }
            if (!ok) break;
            // next unit's q rows (its loads overlap this unit's last MMAs)
            const int next = lin + static_cast<int>(gridDim.x);
            Unit nun;
            if (next < n_units) {
                nun = decode_unit(unit_of(next, sc), sc);
                ok = rope_item<D>(bar(B_QFULL), bar(B_QREADY), static_cast<uint32_t>(items) & 1u, abort_flag, qtile,
                                  row, nun.it.rows(t), H + nun.it.q0(t), cos_t, sin_t, tab_stride, wait_ns);
                ++items;
                if (!ok) break;
            }
            // epilogue: O_T / l -> bf16 -> out, or for a piece the unnormalised O_T and (m, l)
            const size_t prow = (static_cast<size_t>(un.piece) * 2 * BM + t * BM + row);
            if (n_tiles > 0) {
                ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_OFULL0 + t), o_cnt & 1u, abort_flag, wait_ns));
                if (!ok) break;
                ++o_cnt;
                tc_fence_after();
                if (un.piece < 0) {
                    // O_T / l -> bf16 through this warp's staging area, 64 columns at a time: each
                    // thread writes its row there, then the warp stores 4 rows (512 contiguous-row
                    // bytes) per instruction instead of 32 rows 10 KB apart.
                    const float inv_l = 1.f / l_run;
                    const int lane = threadIdx.x & 31, r0 = row & ~31;
                    uint8_t* stage = gbase + L::OFF_STAGE + warp * L::STAGE_WARP;
                    uint16_t* obase = out + ((static_cast<size_t>(it.b) * s_stride + it.q0(t) + r0) * Hq + it.h) * D;
#pragma unroll
                    for (int c2 = 0; c2 < D / 64; ++c2) {
                        uint32_t o[2][32];
                        tmem_ld32(o_col + 64 * c2, o[0]);
                        tmem_ld32(o_col + 64 * c2 + 32, o[1]);
                        tmem_wait_ld();
#pragma unroll
                        for (int ch = 0; ch < 8; ++ch) {  // 16-byte chunks, swizzled by the row
                            const float* f = reinterpret_cast<const float*>(o[ch >> 2]) + (ch & 3) * 8;
                            *reinterpret_cast<uint4*>(stage + lane * 128 + ((ch ^ (lane & 7)) << 4)) = make_uint4(
                                pack_bf16x2(f[0] * inv_l, f[1] * inv_l), pack_bf16x2(f[2] * inv_l, f[3] * inv_l),
                                pack_bf16x2(f[4] * inv_l, f[5] * inv_l), pack_bf16x2(f[6] * inv_l, f[7] * inv_l));
                        }
                        __syncwarp();
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const int rr = 4 * i + (lane >> 3), ch = lane & 7;
                            const uint4 u = *reinterpret_cast<const uint4*>(stage + rr * 128 + ((ch ^ (rr & 7)) << 4));
                            if (r0 + rr < it.rows(t))
                                *reinterpret_cast<uint4*>(obase + static_cast<size_t>(rr) * Hq * D + 64 * c2 + 8 * ch) = u;
                        }
                        __syncwarp();
                    }
                } else {
                    // a piece: the unnormalised O_T (float) through the same staging area, 32
                    // columns per pass, so each warp store writes 4 whole 128-byte row segments
                    const int lane = threadIdx.x & 31, r0 = row & ~31;
                    uint8_t* stage = gbase + L::OFF_STAGE + warp * L::STAGE_WARP;
                    float* pbase = ws_o + (static_cast<size_t>(un.piece) * 2 * BM + t * BM + r0) * D;
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) {
                        uint32_t o[32];
                        tmem_ld32(o_col + 32 * c, o);
                        tmem_wait_ld();
#pragma unroll
                        for (int ch = 0; ch < 8; ++ch)
                            *reinterpret_cast<uint4*>(stage + lane * 128 + ((ch ^ (lane & 7)) << 4)) =
                                make_uint4(o[4 * ch], o[4 * ch + 1], o[4 * ch + 2], o[4 * ch + 3]);
                        __syncwarp();
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const int rr = 4 * i + (lane >> 3), ch = lane & 7;
                            const uint4 u = *reinterpret_cast<const uint4*>(stage + rr * 128 + ((ch ^ (rr & 7)) << 4));
                            if (r0 + rr < it.rows(t))
                                *reinterpret_cast<uint4*>(pbase + static_cast<size_t>(rr) * D + 32 * c + 4 * ch) = u;
                        }
                        __syncwarp();
                    }
                }
                if (un.piece >= 0 && row < it.rows(t)) {
                    ws_ml[prow * 2 + 0] = m_run;
                    ws_ml[prow * 2 + 1] = l_run;
                }
                tc_fence_before();
                __syncwarp();
                if ((threadIdx.x & 31) == 0) mbar_arrive(bar(B_OEMPTY0 + t));
            } else if (un.piece >= 0 && row < it.rows(t)) {  // this piece holds no key of tile t
                ws_ml[prow * 2 + 0] = -INFINITY;
                ws_ml[prow * 2 + 1] = 0.f;
            }
            lin = next;
            un = nun;
        }
        if (!ok) {
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

// Merges the pieces of each tail item: for every row, m* = max m_s over pieces with
// l_s > 0, out = sum_s 2^(m_s - m*) O_s / sum_s 2^(m_s - m*) l_s -> bf16.
// Block (tail item, query tile, group of 8 rows); one warp per row.
template <int D>
__global__ void __launch_bounds__(256) flash_combine_kernel(const float* __restrict__ ws_o,
                                                            const float* __restrict__ ws_ml, const Sched sc,
                                                            int s_stride, uint16_t* __restrict__ out) {
    constexpr int PER_LANE = D / 32;
    asm volatile("griddepcontrol.wait;" ::: "memory");  // the pieces are complete and visible
    const int head = sc.head, nsplit = sc.nsplit, Hq = sc.Hq;
    const int item = head + static_cast<int>(blockIdx.x) / 2;
    const int t = static_cast<int>(blockIdx.x) % 2;
    const Item it = decode_item(item, sc);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int row = static_cast<int>(blockIdx.y) * 8 + warp;
    if (row < it.rows(t)) {
        const size_t v0 = static_cast<size_t>(item - head) * nsplit;
        float m = -INFINITY, l = 0.f;
        if (lane < nsplit) {
            const size_t prow = (v0 + lane) * 2 * BM + t * BM + row;
            m = ws_ml[prow * 2 + 0];
            l = ws_ml[prow * 2 + 1];
        }
        float mm = l > 0.f ? m : -INFINITY;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) mm = fmaxf(mm, __shfl_xor_sync(0xFFFFFFFFu, mm, off));
        const float w = l > 0.f ? fast_exp2(m - mm) : 0.f;
        float lw = l * w;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) lw += __shfl_xor_sync(0xFFFFFFFFu, lw, off);
        float acc[PER_LANE];
#pragma unroll
        for (int e = 0; e < PER_LANE; ++e) acc[e] = 0.f;
        for (int sp = 0; sp < nsplit; ++sp) {
            const float ws = __shfl_sync(0xFFFFFFFFu, w, sp);
            if (ws == 0.f) continue;  // a piece without keys of this tile: its O was never written
            const float* src = ws_o + ((v0 + sp) * 2 * BM + t * BM + row) * D + lane * PER_LANE;
#pragma unroll
            for (int e = 0; e < PER_LANE; ++e) acc[e] = fmaf(ws, src[e], acc[e]);
        }
        const float inv = 1.f / lw;
        uint16_t* dst = out + ((static_cast<size_t>(it.b) * s_stride + it.q0(t) + row) * Hq + it.h) * D + lane * PER_LANE;
#pragma unroll
        for (int e = 0; e < PER_LANE; e += 2)
            *reinterpret_cast<uint32_t*>(dst + e) = pack_bf16x2(acc[e] * inv, acc[e + 1] * inv);
    }
}

// Host schedule: `head` items fill whole rounds of the persistent CTAs; the tail items
// (the last, partial round) may be cut into nsplit KV pieces, at most one per CTA, that
// the merge kernel combines.  The piece count minimises a model of the slowest CTA's
// time, dealt as the kernel deals (rounds of alternating direction): per unit a fixed
// cost (its q copy and RoPE hand-over, epilogue), per KV step of the two query tiles the
// tensor-core time of four 128 x 128 x D MMAs, and for a split launch the partial writes
// and the merge kernel.
struct HostSchedule {
    int n_pairs, n_items, head, nsplit, n_units, grid, kvb;
};

// Items are grouped in blocks of kv heads when the history is at least the chunk and the
// launch's K/V exceeds kKvBlockFrom; a block's K/V stays within kKvBlockBytes (of 126 MB
// of L2).  Causal launches without such a history keep the longest-first order, whose
// balance matters more there.
constexpr double kKvBlockFrom = 42.0e6, kKvBlockBytes = 48.0e6;

constexpr int kMaxSplit = 16;

int unit_of_host(int lin, int g, int n_units) {
    const int r = lin / g;
    if ((r & 1) == 0 || (r + 1) * g > n_units) return lin;
    return r * g + (g - 1 - lin % g);
}

HostSchedule make_schedule(const Shape& s, int hist, int chunk, int num_sms) {
    HostSchedule sc;
    const int n_qtiles = (chunk + BM - 1) / BM;
    sc.n_pairs = (n_qtiles + 1) / 2;
    sc.n_items = sc.n_pairs * s.n_q_heads * s.batch;
    const int hq_b = s.n_q_heads * s.batch, G = s.n_q_heads / s.n_kv_heads;
    const double head_bytes = 4.0 * (static_cast<double>(hist) + chunk) * s.head_dim;  // K/V of one kv head
    sc.kvb = 0;
    if (hist >= chunk && head_bytes * s.batch * s.n_kv_heads > kKvBlockFrom) {
        sc.kvb = 1;
        for (int d = 1; d <= s.n_kv_heads; ++d)
            if (s.n_kv_heads % d == 0 && d * head_bytes <= kKvBlockBytes) sc.kvb = d;
    }
    auto n_kv = [&](int item) {  // KV tiles of an item (longest pairs first, in either order)
        const int qt = sc.kvb ? item % (sc.n_pairs * sc.kvb * G) / (sc.kvb * G) : item / hq_b;
        const int pt = sc.n_pairs - 1 - qt;
        return (hist + std::min(2 * BM * (pt + 1), chunk) + BN - 1) / BN;
    };
    // costs in KV steps of both query tiles (about 1.3 us each)
    const double c_unit = 1.6, c_split = 2.5, c_step = 1.0;
    const int full_rounds = sc.n_items / num_sms;
    const int tail = sc.n_items - full_rounds * num_sms;
    const int nkv_min = tail > 0 ? n_kv(sc.n_items - 1) : 1;  // the tail's shortest item
    int best_ns = 1;
    double best = 1e300;
    std::vector<double> load;
    for (int ns = 1; ns <= kMaxSplit; ++ns) {
        if (ns > 1 && (tail == 0 || tail * ns > num_sms || ns > nkv_min)) break;
        const int head = ns > 1 ? full_rounds * num_sms : sc.n_items;
        const int n_units = head + (sc.n_items - head) * ns;
        const int grid = std::min(n_units, num_sms);
        load.assign(grid, 0.0);
        for (int lin = 0; lin < n_units; ++lin) {
            const int u = unit_of_host(lin, grid, n_units);
            double cost = c_unit;
            if (u < head) {
                cost += c_step * n_kv(u);
            } else {
                const int v = u - head, nk = n_kv(head + v / ns), sp = v % ns;
                cost += c_step * (nk * (sp + 1) / ns - nk * sp / ns);
            }
            load[lin % grid] += cost;
        }
        const double mk = *std::max_element(load.begin(), load.end()) + (ns > 1 ? c_split : 0.0);
        if (mk < best - 1e-9) {
            best = mk;
            best_ns = ns;
        }
    }
    sc.nsplit = best_ns;
    sc.head = best_ns > 1 ? full_rounds * num_sms : sc.n_items;
    sc.n_units = sc.head + (sc.n_items - sc.head) * sc.nsplit;
    sc.grid = std::min(sc.n_units, num_sms);
    return sc;
}

template <int D>
cudaError_t launch_d(const Shape& s, const FlashMaps& maps, int hist, int chunk, int s_stride, const float* cos_t,
                     const float* sin_t, uint16_t* out, float* ws_o, float* ws_ml, int* err, int num_sms,
                     cudaStream_t st, int* n_launched, uint64_t wait_ns) {
    const HostSchedule hs = make_schedule(s, hist, chunk, num_sms);
    Sched sc;
    sc.S = chunk;
    sc.H = hist;
    sc.Hq = s.n_q_heads;
    sc.G = s.n_q_heads / s.n_kv_heads;
    sc.batch = s.batch;
    sc.kvb = hs.kvb;
    sc.n_pairs = hs.n_pairs;
    sc.head = hs.head;
    sc.nsplit = hs.nsplit;
    sc.n_units = hs.n_units;
    sc.fd_grid = make_fastdiv(hs.grid);
    sc.fd_hqb = make_fastdiv(s.n_q_heads * s.batch);
    sc.fd_hq = make_fastdiv(s.n_q_heads);
    sc.fd_g = make_fastdiv(s.n_q_heads / s.n_kv_heads);
    sc.fd_ns = make_fastdiv(hs.nsplit);
    const int per = std::max(hs.kvb, 1) * sc.G;
    sc.fd_pb = make_fastdiv(hs.n_pairs * per);
    sc.fd_per = make_fastdiv(per);
    sc.fd_nb = make_fastdiv(s.n_q_heads / per);
    const float scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(D)));
    // Dependent launch after K1 (programmatic stream serialization): only the producer's
    // first K/V copy waits for K1 (griddep_wait).
    cudaLaunchConfig_t kcfg = {};
    kcfg.gridDim = dim3(static_cast<unsigned>(hs.grid));
    kcfg.blockDim = dim3(kThreads);
    kcfg.dynamicSmemBytes = Layout<D>::ALLOC;
    kcfg.stream = st;
    cudaLaunchAttribute kattr[1];
    kattr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    kattr[0].val.programmaticStreamSerializationAllowed = 1;
    kcfg.attrs = kattr;
    kcfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&kcfg, flash_fwd_kernel<D>, maps.q, maps.k, maps.v, sc, s_stride,
                                       s.n_kv_heads, scale_log2, cos_t, sin_t, s.max_len, out, ws_o, ws_ml, err,
                                       wait_ns);
    *n_launched = 1;
    if (e != cudaSuccess || hs.nsplit == 1) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(2 * (hs.n_items - hs.head)), BM / 8);
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, flash_combine_kernel<D>, ws_o, ws_ml, sc, s_stride, out);
    *n_launched = 2;
    return e;
}

// The register split of the warpgroups is only safe when the kernel is launched
// with exactly kLaunchRegs registers per thread: check before any launch.
template <int D>
cudaError_t configure_d() {
    cudaFuncAttributes attr;
    cudaError_t e = cudaFuncGetAttributes(&attr, flash_fwd_kernel<D>);
    if (e != cudaSuccess) return e;
    if (attr.numRegs != kLaunchRegs || attr.maxThreadsPerBlock < kThreads) return cudaErrorInvalidConfiguration;
    return cudaFuncSetAttribute(flash_fwd_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, Layout<D>::ALLOC);
}

}  // namespace

cudaError_t configure_flash_fwd() {
    const cudaError_t e = configure_d<128>();
    return e != cudaSuccess ? e : configure_d<64>();
}

cudaError_t launch_flash_fwd(const Shape& s, const FlashMaps& maps, int hist, int chunk, int s_stride,
                             const float* cos_t, const float* sin_t, uint16_t* out, float* ws_o, float* ws_ml, int* err,
                             int num_sms, cudaStream_t st, int* n_launched, uint64_t wait_ns) {
    if (s.head_dim == 128)
        return launch_d<128>(s, maps, hist, chunk, s_stride, cos_t, sin_t, out, ws_o, ws_ml, err, num_sms, st,
                             n_launched, wait_ns);
    return launch_d<64>(s, maps, hist, chunk, s_stride, cos_t, sin_t, out, ws_o, ws_ml, err, num_sms, st, n_launched,
                        wait_ns);
}

}  // namespace attn

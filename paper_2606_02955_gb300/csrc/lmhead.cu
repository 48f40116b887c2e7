// lmhead.cu -- step a1 fused with the LM head that produces the logits.  The logits of a
// masked position are x = W h (h its final hidden state [H], W the vocabulary projection
// [V, H]); instead of writing B*L*V logits and reading them back, a tcgen05 GEMM reduces
// each 128-row x BN-column accumulator tile (BN = 256 or 208 vocabulary entries) in its
// epilogue to one (max, sum of exp, first argmax) partial per row, straight from tensor
// memory.
//
// Launch sequence on one stream (all rows of one step), chained by programmatic dependent
// launches:
//   1. compact_rows_kernel   the masked rows' indices and their count (one CTA)
//   2. gather_rows_kernel    the masked rows' hidden states, packed [R, H] (TMA-friendly)
//   3. lmhead_gemm_kernel    persistent tcgen05 GEMM: warp 0 issues TMA loads into a ring of
//                            stages, warp 1 issues tcgen05.mma into one of two TMEM
//                            accumulators, warps 2-5 reduce (or store) the other one; solo
//                            or CTA-pair (cta_group::2) variants
//      lmhead_slab_kernel    (at most 32 rows) the operands swapped, W as the M = 128 side:
//                            each CTA streams one vocabulary slab, one partial per row
//   4. combine_rows_kernel   four warps per row fold its tile (or slab) partials in a fixed
//                            order
//   5. profile_select        steps a2-a5 on the confidences (profile_select.cu)
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <cstdlib>
#include <mutex>
#include <string>

#include "fdllm.h"
#include "fdllm_internal.cuh"
#include "ptx.cuh"
#include "tcgen05.cuh"

namespace fdllm {
namespace {

constexpr int BM = 128;  // rows per tile (TMEM lanes)
constexpr int BK = 64;   // hidden elements per stage: one 128-byte swizzle row of bf16
constexpr int kABytes = BM * BK * 2;
constexpr int kThreads = 192;         // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr uint32_t kAccStride = 256;  // TMEM columns between the two accumulators
constexpr uint32_t kTmemCols = 512;
constexpr size_t kBarrierBytes = 256;
constexpr size_t kRingBudget = 220 * 1024;

// How the CTAs of a cluster share a W tile.
enum Mode {
    kSolo = 0,       // one CTA per work item; it loads the whole W tile
    kPair = 2,       // 2-CTA pair MMA (tcgen05 cta_group::2, M = 256): each CTA holds its 128
                     // rows and half of the W tile; the even CTA issues the MMAs for both
    kSlab = 3,       // at most 32 rows: W as the M = 128 operand, each CTA a vocabulary slab
                     // (lmhead_slab_kernel)
};

constexpr int PAIR_KB = 2;  // pair mode: K-blocks per stage

// Vocabulary entries per tile (the MMA's N and the fp32 accumulator's width): 256, or 208,
// which splits LLaDA's V = 126464 into 608 = 4 x 152 tiles, whole waves over 152 SMs.  The
// stage count fills the ring budget: solo 4 x 48 KB at 256, 5 x 42 KB at 208; pair 3 x 64 KB
// at 256 (each CTA holds half the W tile, and a stage two K-blocks: with the pair's two
// cross-CTA signals per stage, fewer and larger stages measured faster than 6 x 32 KB).
template <int BN_, int MODE>
struct TileCfg {
    static constexpr int BN = BN_;
    static constexpr int kBRows = MODE == kPair ? BN / 2 : BN;  // W rows held per CTA
    static constexpr int kBBytes = kBRows * BK * 2;
    static constexpr int kKB = MODE == kPair ? PAIR_KB : 1;       // K-blocks of BK per stage
    static constexpr int kStageBytes = kKB * (kABytes + kBBytes);
    static constexpr int kStages =
        (int)(kRingBudget / kStageBytes) > 8 ? 8 : (int)(kRingBudget / kStageBytes);
    static constexpr size_t kSmemBytes = 1024 + (size_t)kStages * kStageBytes + kBarrierBytes;
    static_assert(BN % 16 == 0 && BN <= (int)kAccStride, "MMA N");
    static_assert((BN / 2) % 8 == 0, "halves of whole 8-row swizzle atoms");
};

enum Epilogue { kReduce = 0, kStore = 1 };

struct GemmArgs {
    const int32_t *row_count;  // R, written by compact_rows_kernel
    const int32_t *row_ids;    // [R] global row (b * L + l) of each packed row
    int32_t V;
    int32_t n_tiles;           // partials per row: ceil(V / BN), or the slab variant's grid
    int32_t k_blocks;          // ceil(H / BK)
    int32_t slab_tiles;        // slab variant: vocabulary tiles, ceil(V / slab_h)
    int32_t slab_h;            // slab variant: W rows per tile (a multiple of 8, <= 128)
    UnitPartial *partials;     // kReduce: [R][n_tiles]
    float *logits;             // kStore: [B * L][V] fp32, written at masked rows
    uint32_t *status;          // sticky device error bits
    bool pdl;                  // host side: launch as a programmatic dependent
};

// A bounded wait that also gives up as soon as another role of the CTA has given up.
__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, uint32_t *status,
                                              volatile int *abort_flag)
{
    if (mbar_try_wait(bar, parity))
        return true;
    const uint64_t t0 = global_timer_ns();
    for (uint32_t it = 1;; ++it) {
        if (mbar_try_wait(bar, parity))
            return true;
        if ((it & 63u) == 0) {
            if (*abort_flag)
                return false;
            if (global_timer_ns() - t0 > kWaitLimitNs) {
                atomicOr(status, kDevStatTimeout);
                *abort_flag = 1;
                return false;
            }
        }
    }
}

// MODE kSolo: every CTA loads its own W tile.  kPair: the two CTAs of a cluster take row
// tiles 2j and 2j + 1 of the same vocabulary tile, which form one M = 256 MMA issued by the
// even CTA (tcgen05 cta_group::2):
// each CTA loads its 128 rows and half of the W tile into its own shared memory and
// signals the even CTA's stage barrier, so each CTA's shared memory supplies half the
// operand bytes per MMA; the accumulators live in both CTAs' tensor memory.
template <int EPI, int MODE, int BN_>
__global__ void __launch_bounds__(kThreads, 1)
    lmhead_gemm_kernel(const __grid_constant__ CUtensorMap map_h,
                       const __grid_constant__ CUtensorMap map_w, const GemmArgs a)
{
    using Cfg = TileCfg<BN_, MODE>;
    constexpr int CL = MODE == kSolo ? 1 : 2;
    constexpr bool PAIR = MODE == kPair;
    constexpr int BN = Cfg::BN, kStages = Cfg::kStages, KB = Cfg::kKB;
    constexpr int kBBytes = Cfg::kBBytes, kStageBytes = Cfg::kStageBytes;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sA = smem;                          // kStages x KB x [BM rows][128 B], swizzled
    uint8_t *sB = smem + kStages * KB * kABytes; // kStages x KB x [kBRows rows][128 B]
    uint64_t *bars = reinterpret_cast<uint64_t *>(sB + kStages * KB * kBBytes);
    uint64_t *full = bars;                  // TMA -> MMA, one per stage
    uint64_t *empty = bars + kStages;       // MMA -> TMA, one per stage
    uint64_t *tfull = bars + 2 * kStages;   // MMA -> epilogue, one per accumulator
    uint64_t *tempty = tfull + 2;           // epilogue -> MMA, one per accumulator
    uint64_t *done = tempty + 2;            // MMA thread: all its MMAs have completed
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);  // released by the MMA issuer's commit
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], PAIR ? 8 : 4);  // one arrival per epilogue warp (of the pair)
        }
        mbar_init(done, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tc::prefetch_tensormap(&map_h);
        tc::prefetch_tensormap(&map_w);
    }
    if (warp == 1) {
        if (PAIR)
            tc::tmem_alloc_pair(tmem_slot, kTmemCols);
        else
            tc::tmem_alloc(tmem_slot, kTmemCols);
    }
    tc::fence_before_sync();
    __syncthreads();
    if (CL > 1)
        tc::cluster_sync();  // the peer's barriers are initialised before any remote signal
    tc::fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;

    // A programmatic dependent of the packing kernel: everything above overlapped its tail;
    // the packed rows and their count are read only past this wait.
    pdl_wait();

    const int rank = CL > 1 ? (int)tc::cluster_ctarank() : 0;
    const int64_t first = CL > 1 ? (int64_t)tc::cluster_id_x() : (int64_t)blockIdx.x;
    const int64_t stride = CL > 1 ? (int64_t)tc::cluster_count_x() : (int64_t)gridDim.x;
    // An epilogue warp hands an accumulator back to the MMA issuer (in a pair, the even
    // CTA's barrier counts the warps of both CTAs).
    auto release_acc = [](uint64_t *bar, int rk) {
        if (PAIR && rk != 0)
            tc::mbar_arrive_remote(tc::map_to_rank(bar, 0));
        else
            mbar_arrive(bar);
    };
    const int R = *a.row_count;
    const int num_m = (R + BM - 1) / BM;
    const int num_mc = (num_m + CL - 1) / CL;  // row-tile groups, one per cluster
    const int64_t total = (int64_t)num_mc * a.n_tiles;
    // Work item t covers packed rows [m*BM, +BM) with m = (t % num_mc) * CL + rank, and
    // vocabulary [n*BN, +BN) with n = t / num_mc: row tiles fastest, so the CTAs working at
    // the same time share few W tiles (read from HBM once, then from L2).  With CL = 2 and
    // an odd number of row tiles, the last rank-1 CTA computes a tile of rows >= R (zero or
    // stale inputs) that its epilogue skips.

    if (warp == 0) {
        if (lane == 0) {
            // W tiles are marked first to evict: each is read from HBM once, and the other row
            // tiles that share it (consecutive work items) read it from L2 right away.
            const uint64_t pol = make_evict_first_policy();
            int s = 0;
            uint32_t ph = 0;
            uint32_t last_ph[kStages];
            bool used[kStages];
            for (int i = 0; i < kStages; ++i)
                used[i] = false;
            bool ok = true;
            for (int64_t t = first; ok && t < total; t += stride) {
                const int m = (int)(t % num_mc) * CL + rank, n = (int)(t / num_mc);
                for (int kb = 0; kb < a.k_blocks; kb += KB) {
                    if (!wait_or_abort(&empty[s], ph ^ 1u, a.status, abort_flag)) {
                        ok = false;
                        break;
                    }
                    if constexpr (PAIR) {
                        // Both CTAs' bytes complete on the even CTA's barrier, which it arms
                        // (K-blocks past H, in the last stage when k_blocks is odd, are
                        // zero-filled and count in full).
                        if (rank == 0)
                            mbar_arrive_expect_tx(&full[s], 2 * kStageBytes);
                        const uint32_t bar0 = tc::map_to_rank(&full[s], 0);
#pragma unroll
                        for (int q = 0; q < KB; ++q) {
                            tc::tma_load_2d_pair(sA + (s * KB + q) * kABytes, &map_h,
                                                 (kb + q) * BK, m * BM, bar0);
                            tc::tma_load_2d_pair(sB + (s * KB + q) * kBBytes, &map_w,
                                                 (kb + q) * BK, n * BN + rank * (BN / 2), bar0);
                        }
                    } else {
                        mbar_arrive_expect_tx(&full[s], kStageBytes);
#pragma unroll
                        for (int q = 0; q < KB; ++q) {
                            tc::tma_load_2d(sA + (s * KB + q) * kABytes, &map_h, (kb + q) * BK,
                                            m * BM, &full[s]);
                            tc::tma_load_2d_hint(sB + (s * KB + q) * kBBytes, &map_w,
                                                 (kb + q) * BK, n * BN, &full[s], pol);
                        }
                    }
                    used[s] = true;
                    last_ph[s] = ph;
                    if (++s == kStages) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
            }
            // No copy of this CTA may still be in flight when it exits (in a pair, the even
            // CTA's barriers count both CTAs' copies, and the odd CTA leaves only after it,
            // at the final cluster barrier).
            if (!PAIR || rank == 0)
                for (int i = 0; i < kStages; ++i)
                    if (used[i])
                        mbar_wait(&full[i], last_ph[i], a.status, kDrainLimitNs);
        }
    } else if (warp == 1) {
        if (lane == 0 && (!PAIR || rank == 0)) {
            constexpr uint32_t idesc = tc::idesc_bf16_f32(PAIR ? 2 * BM : BM, BN);
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            int i = 0;
            for (int64_t t = first; ok && t < total; t += stride, ++i) {
                const int acc = i & 1;
                const uint32_t aph = (uint32_t)(i >> 1) & 1u;
                if (!wait_or_abort(&tempty[acc], aph ^ 1u, a.status, abort_flag))
                    break;
                tc::fence_after_sync();
                const uint32_t d = tmem_base + (uint32_t)acc * kAccStride;
                for (int kb = 0; kb < a.k_blocks; kb += KB) {
                    if (!wait_or_abort(&full[s], ph, a.status, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc::fence_after_sync();
#pragma unroll
                    for (int q = 0; q < KB; ++q) {
                        const uint64_t ad = tc::sw128_kmajor_desc(sA + (s * KB + q) * kABytes);
                        const uint64_t bd = tc::sw128_kmajor_desc(sB + (s * KB + q) * kBBytes);
#pragma unroll
                        for (int k = 0; k < BK / 16; ++k) {  // K = 16 per MMA: +32 B in the row
                            if constexpr (PAIR)
                                tc::mma_bf16_pair(d, ad + 2u * k, bd + 2u * k, idesc,
                                                  (kb | q | k) != 0);
                            else
                                tc::mma_bf16(d, ad + 2u * k, bd + 2u * k, idesc,
                                             (kb | q | k) != 0);
                        }
                    }
                    // The stage is free once these MMAs have read it (in a pair, in both
                    // CTAs: each refills its own half of the pair's operands).
                    if constexpr (PAIR)
                        tc::commit_pair_multicast(&empty[s]);
                    else
                        tc::commit(&empty[s]);
                    if (++s == kStages) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
                if (ok) {
                    if constexpr (PAIR)
                        tc::commit_pair_multicast(&tfull[acc]);  // both CTAs' accumulators
                    else
                        tc::commit(&tfull[acc]);
                }
            }
            // Tensor memory is freed below only after every MMA issued here has completed.
            if constexpr (PAIR)
                tc::commit_pair_multicast(done);  // the odd CTA's copy is never waited on
            else
                tc::commit(done);
            mbar_wait(done, 0, a.status, kDrainLimitNs);
        }
        __syncwarp();
    } else {
        // Epilogue: warp w reads TMEM lanes [32 (w % 4), +32): thread = one row of the tile.
        const int quarter = warp & 3;
        const int row_in_tile = quarter * 32 + lane;
        int i = 0;
        for (int64_t t = first; t < total; t += stride, ++i) {
            const int acc = i & 1;
            const uint32_t aph = (uint32_t)(i >> 1) & 1u;
            const int m = (int)(t % num_mc) * CL + rank, n = (int)(t / num_mc);
            // Every lane waits; the warp leaves together if any lane gave up, so that the
            // warp-collective tensor-memory loads below are always executed by all lanes.
            const bool ok = wait_or_abort(&tfull[acc], aph, a.status, abort_flag);
            if (!__all_sync(0xFFFFFFFFu, ok))
                break;
            tc::fence_after_sync();
            const uint32_t taddr =
                tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)acc * kAccStride;
            const int r = m * BM + row_in_tile;
            const int col0 = n * BN;
            float v[32];
            if (EPI == kReduce) {
                // Pass 1: max and its first column; NaN is tracked apart (fmax would drop it).
                float M = -__int_as_float(0x7F800000);
                uint32_t idx = kNoIdx;
                bool nan = false;
#pragma unroll 1
                for (int c = 0; c < (BN + 31) / 32; ++c) {
                    tc::tmem_ld_32cols(taddr + c * 32, v);  // columns >= BN: not this tile
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int col = col0 + c * 32 + j;
                        if (c * 32 + j < BN && col < a.V) {
                            nan |= v[j] != v[j];
                            if (v[j] > M) {
                                M = v[j];
                                idx = (uint32_t)col;
                            }
                        }
                    }
                }
                // Pass 2: sum of exp(x - M) = 2^(x sc - M2), four partial sums, with the
                // scale sc and reference M2 of rebase_scaled (sc = 1 and M2 = M for |M| at or
                // beyond kBigRef, where only x == M contributes).
                const bool big = !(fabsf(M) < kBigRef);
                const float sc = big ? 1.0f : kLog2e;
                const float M2 = big ? M : M * kLog2e;
                float S4[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll 1
                for (int c = 0; c < (BN + 31) / 32; ++c) {
                    tc::tmem_ld_32cols(taddr + c * 32, v);
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int col = col0 + c * 32 + j;
                        if (c * 32 + j < BN && col < a.V)
                            S4[j & 3] += ex2_mufu(fmaf(v[j], sc, -M2));
                    }
                }
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0)
                    release_acc(&tempty[acc], rank);
                if (r < R) {
                    UnitPartial p;
                    p.M = nan ? __int_as_float(0x7FC00000) : M;
                    // relative to M exactly; a tile with no finite logit adds exactly 0
                    p.S = M == -INFINITY
                              ? 0.0f
                              : rebase_scaled((S4[0] + S4[1]) + (S4[2] + S4[3]), sc, M2, M);
                    p.idx = idx;
                    p.pad = 0;
                    a.partials[(int64_t)r * a.n_tiles + n] = p;
                }
            } else {
                const int64_t row = r < R ? a.row_ids[r] : -1;
#pragma unroll 1
                for (int c = 0; c < (BN + 31) / 32; ++c) {
                    tc::tmem_ld_32cols(taddr + c * 32, v);
                    if (row >= 0) {
                        float *dst = a.logits + row * a.V + col0 + c * 32;
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (c * 32 + j < BN && col0 + c * 32 + j < a.V)
                                dst[j] = v[j];
                    }
                }
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0)
                    release_acc(&tempty[acc], rank);
            }
        }
    }
    if (threadIdx.x == 0)
        pdl_launch_dependents();  // the row combination may start launching
    __syncthreads();
    if (PAIR)
        tc::cluster_sync();  // both CTAs are done with the pair's tensor memory
    if (warp == 1) {
        __syncwarp();
        tc::fence_after_sync();
        if (PAIR)
            tc::tmem_dealloc_pair(tmem_base, kTmemCols);
        else
            tc::tmem_dealloc(tmem_base, kTmemCols);
    }
    if (CL > 1)
        tc::cluster_sync();  // no CTA leaves while its peer may still write into it
}

// ----------------------------------------------------------------------------- slab variant
// For at most kSlabRows masked rows the operands swap roles: W is the MMA's A operand (M =
// 128 TMEM lanes, lane = vocabulary entry) and the packed rows are its B operand (N = 32,
// TMEM column = row).  The vocabulary is cut into tiles of h entries (one TMA box of h W
// rows, h a multiple of 8 up to 128, chosen by the host so that the busiest CTA streams as
// few W rows as possible: LLaDA's V = 126464 is 1216 tiles of 104, eight per SM on 152
// SMs); CTA c of P owns the tiles c, c + P, c + 2P, ..., so the CTAs read W in a window that
// moves through it.  The MMA always spans 128 lanes; lanes h..127 hold sums of stale shared
// memory that the epilogue skips.  The padded row tile costs 4 KB per K-block instead of
// 16 KB.  A stage holds two K-blocks (two W boxes and two row boxes), five stages in all
// (130 KB of W at h = 104 in flight per SM): per-copy overhead, not the bytes in flight,
// limits how fast W streams here, and two blocks per stage beat one, three or four.  Each
// epilogue thread keeps, for every row, a running maximum, sum of exp relative to it and
// first index over its own entry of each tile; after the last tile the 128 threads' states
// are folded per row (a transposing butterfly in each warp, then the four warps in order)
// into one partial per (row, CTA).
constexpr int kSlabRows = 32;
constexpr int kSlabABytes = BM * BK * 2;                 // 128 lanes; a tile fills h rows
constexpr int kSlabBBytes = kSlabRows * BK * 2;
constexpr int kSlabKB = 2;                               // K-blocks of BK per stage
constexpr int kSlabStages = 5;
constexpr int kSlabAccs = 4;                             // accumulators of 32 columns
constexpr uint32_t kSlabTmemCols = 128;
constexpr size_t kSlabSmemBytes =
    1024 + (size_t)kSlabStages * kSlabKB * (kSlabABytes + kSlabBBytes) + kBarrierBytes;
static_assert(kSlabSmemBytes <= 227 * 1024, "slab ring");
static_assert((2 * kSlabStages + 2 * kSlabAccs + 1) * 8 + 8 <= (int)kBarrierBytes, "barriers");

// Two (max, sum relative to it, first index) states of one row -> one.  NaN logits reach
// only S (they never raise the max), which then stays NaN.
__device__ __forceinline__ void fold_state(float &M, float &S, uint32_t &I, float M2, float S2,
                                           uint32_t I2)
{
    const float Mn = fmaxf(M, M2);
    S = rebase(S, M, Mn) + rebase(S2, M2, Mn);
    const uint32_t i1 = M == Mn ? I : kNoIdx, i2 = M2 == Mn ? I2 : kNoIdx;
    I = i1 < i2 ? i1 : i2;
    M = Mn;
}

template <int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    lmhead_slab_kernel(const __grid_constant__ CUtensorMap map_h,
                       const __grid_constant__ CUtensorMap map_w, const GemmArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ float s_M[4][kSlabRows], s_S[4][kSlabRows];
    __shared__ uint32_t s_I[4][kSlabRows];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    // kSlabStages x kSlabKB x [128 W rows][128 B], then kSlabStages x kSlabKB x [32 rows][128 B]
    uint8_t *sA = smem;
    uint8_t *sB = smem + kSlabStages * kSlabKB * kSlabABytes;
    uint64_t *bars = reinterpret_cast<uint64_t *>(sB + kSlabStages * kSlabKB * kSlabBBytes);
    uint64_t *full = bars;
    uint64_t *empty = bars + kSlabStages;
    uint64_t *tfull = bars + 2 * kSlabStages;
    uint64_t *tempty = tfull + kSlabAccs;
    uint64_t *done = tempty + kSlabAccs;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kSlabStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int i = 0; i < kSlabAccs; ++i) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], 4);
        }
        mbar_init(done, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tc::prefetch_tensormap(&map_h);
        tc::prefetch_tensormap(&map_w);
    }
    if (warp == 1)
        tc::tmem_alloc(tmem_slot, kSlabTmemCols);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;

    pdl_wait();  // the packed rows and their count are complete

    const int R = *a.row_count;  // <= kSlabRows: the host takes this variant only then
    const int64_t NT = a.slab_tiles, P = gridDim.x, c = blockIdx.x;
    const int h = a.slab_h;
    const int n_t = R > 0 && c < NT ? (int)((NT - c + P - 1) / P) : 0;  // tiles of this CTA

    if (warp == 0) {
        if (lane == 0) {
            const uint64_t pol = make_evict_first_policy();  // W is read once
            int s = 0;
            uint32_t ph = 0;
            uint32_t last_ph[kSlabStages];
            bool used[kSlabStages];
            for (int i = 0; i < kSlabStages; ++i)
                used[i] = false;
            bool ok = true;
            // a box's bytes count in full, the part beyond V zero-filled
            // (K-blocks past H, in the last stage when k_blocks is odd, are zero-filled and
            // count in full too)
            const uint32_t bytes = kSlabKB * ((uint32_t)(h * BK * 2) + kSlabBBytes);
            for (int t = 0; ok && t < n_t; ++t) {
                const int64_t T = c + (int64_t)t * P;
                for (int kb = 0; kb < a.k_blocks; kb += kSlabKB) {
                    if (!wait_or_abort(&empty[s], ph ^ 1u, a.status, abort_flag)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&full[s], bytes);
#pragma unroll
                    for (int q = 0; q < kSlabKB; ++q)
                        tc::tma_load_2d_hint(sA + (s * kSlabKB + q) * kSlabABytes, &map_w,
                                             (kb + q) * BK, (int32_t)(T * h), &full[s], pol);
#pragma unroll
                    for (int q = 0; q < kSlabKB; ++q)
                        tc::tma_load_2d(sB + (s * kSlabKB + q) * kSlabBBytes, &map_h, (kb + q) * BK,
                                        0, &full[s]);
                    used[s] = true;
                    last_ph[s] = ph;
                    if (++s == kSlabStages) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
            }
            for (int i = 0; i < kSlabStages; ++i)  // none of this CTA's copies in flight at exit
                if (used[i])
                    mbar_wait(&full[i], last_ph[i], a.status, kDrainLimitNs);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_bf16_f32(BM, kSlabRows);
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int t = 0; ok && t < n_t; ++t) {
                const int acc = t % kSlabAccs;
                const uint32_t aph = (uint32_t)(t / kSlabAccs) & 1u;
                if (!wait_or_abort(&tempty[acc], aph ^ 1u, a.status, abort_flag))
                    break;
                tc::fence_after_sync();
                const uint32_t d = tmem_base + (uint32_t)(acc * kSlabRows);
                for (int kb = 0; kb < a.k_blocks; kb += kSlabKB) {
                    if (!wait_or_abort(&full[s], ph, a.status, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc::fence_after_sync();
                    // Rows h..127 of the A stage are stale: those TMEM lanes hold
                    // meaningless sums that the epilogue skips.
#pragma unroll
                    for (int q = 0; q < kSlabKB; ++q) {
                        const uint64_t ad =
                            tc::sw128_kmajor_desc(sA + (s * kSlabKB + q) * kSlabABytes);
                        const uint64_t bd =
                            tc::sw128_kmajor_desc(sB + (s * kSlabKB + q) * kSlabBBytes);
#pragma unroll
                        for (int k = 0; k < BK / 16; ++k)
                            tc::mma_bf16(d, ad + 2u * k, bd + 2u * k, idesc, (kb | q | k) != 0);
                    }
                    tc::commit(&empty[s]);
                    if (++s == kSlabStages) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
                if (ok)
                    tc::commit(&tfull[acc]);
            }
            tc::commit(done);
            mbar_wait(done, 0, a.status, kDrainLimitNs);
        }
        __syncwarp();
    } else {
        // Epilogue: warp w reads TMEM lanes [32 (w % 4), +32): thread = one vocabulary entry
        // of the tile, its 32 columns = the rows.
        const int q = warp & 3;
        float M[kSlabRows], S[kSlabRows];
        uint32_t I[kSlabRows];
#pragma unroll
        for (int r = 0; r < kSlabRows; ++r) {
            M[r] = -__int_as_float(0x7F800000);
            S[r] = 0.0f;
            I[r] = kNoIdx;
        }
        bool aborted = false;
        for (int t = 0; t < n_t; ++t) {
            const int acc = t % kSlabAccs;
            const uint32_t aph = (uint32_t)(t / kSlabAccs) & 1u;
            const bool ok = wait_or_abort(&tfull[acc], aph, a.status, abort_flag);
            if (!__all_sync(0xFFFFFFFFu, ok)) {
                aborted = true;
                break;
            }
            tc::fence_after_sync();
            float v[32];
            tc::tmem_ld_32cols(tmem_base + ((uint32_t)(q * 32) << 16) +
                                   (uint32_t)(acc * kSlabRows),
                               v);
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0)
                mbar_arrive(&tempty[acc]);
            // lane q * 32 + lane of tile c + tP: vocabulary entry (c + tP) * h + q * 32 + lane
            const int in_tile = q * 32 + lane;
            const int64_t ent = (c + (int64_t)t * P) * h + in_tile;
            if (in_tile >= h || ent >= a.V)
                continue;
            if (EPI == kStore) {
#pragma unroll
                for (int r = 0; r < kSlabRows; ++r)
                    if (r < R)
                        a.logits[(int64_t)a.row_ids[r] * a.V + ent] = v[r];
            } else {
#pragma unroll
                for (int r = 0; r < kSlabRows; ++r) {
                    // exp(x - M) in the form (x - M) * log2e, exact at any magnitude; a
                    // larger x re-bases the sum; -inf adds nothing; NaN poisons S
                    const float x = v[r];
                    const bool up = x > M[r];
                    const float e = ex2_mufu((up ? M[r] - x : x - M[r]) * kLog2e);
                    S[r] = up ? fmaf(S[r], e, 1.0f) : (x == -INFINITY ? S[r] : S[r] + e);
                    I[r] = up ? (uint32_t)ent : I[r];
                    M[r] = up ? x : M[r];
                }
            }
        }
        if (EPI == kReduce) {
            // Transposing butterfly: at offset o each lane keeps the half of its remaining
            // row slots selected by its lane bit o and folds in the partner's values for them;
            // slot 0 ends as row `lane`, folded over the warp's 32 entries.
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) {
                const bool hi = (lane & o) != 0;
#pragma unroll
                for (int j = 0; j < o; ++j) {
                    const float sM = hi ? M[j] : M[j + o], sS = hi ? S[j] : S[j + o];
                    const uint32_t sI = hi ? I[j] : I[j + o];
                    float kM = hi ? M[j + o] : M[j], kS = hi ? S[j + o] : S[j];
                    uint32_t kI = hi ? I[j + o] : I[j];
                    const float rM = __shfl_xor_sync(0xFFFFFFFFu, sM, o);
                    const float rS = __shfl_xor_sync(0xFFFFFFFFu, sS, o);
                    const uint32_t rI = __shfl_xor_sync(0xFFFFFFFFu, sI, o);
                    fold_state(kM, kS, kI, rM, rS, rI);
                    M[j] = kM;
                    S[j] = kS;
                    I[j] = kI;
                }
            }
            s_M[q][lane] = M[0];
            s_S[q][lane] = S[0];
            s_I[q][lane] = I[0];
            // every epilogue warp arrives exactly once, aborted or not
            asm volatile("bar.sync 1, 128;" ::: "memory");
            if (q == 0 && !aborted && !*abort_flag && lane < R) {
                float fM = s_M[0][lane], fS = s_S[0][lane];
                uint32_t fI = s_I[0][lane];
                for (int w = 1; w < 4; ++w)
                    fold_state(fM, fS, fI, s_M[w][lane], s_S[w][lane], s_I[w][lane]);
                UnitPartial p;
                p.M = fS != fS ? __int_as_float(0x7FC00000) : fM;
                p.S = fS;
                p.idx = fI;
                p.pad = 0;
                a.partials[(int64_t)lane * a.n_tiles + blockIdx.x] = p;
            }
        }
    }
    if (threadIdx.x == 0)
        pdl_launch_dependents();  // the row combination may start launching
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem_base, kSlabTmemCols);
    }
}

// One CTA: the packed list of masked rows (ascending) and its length.
__global__ void __launch_bounds__(1024) compact_rows_kernel(const uint8_t *mask, int rows,
                                                            int32_t *row_ids, int32_t *row_count)
{
    __shared__ int warp_sums[32];
    pdl_wait();  // the mask's writer has completed
    if (threadIdx.x == 0)
        pdl_launch_dependents();
    const int per = (rows + blockDim.x - 1) / blockDim.x;
    const int lo = threadIdx.x * per;
    const int hi = lo + per < rows ? lo + per : rows;
    int cnt = 0;
    for (int i = lo; i < hi; ++i)
        cnt += mask[i] != 0;
    // Block exclusive scan of cnt.
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o)
            incl += y;
    }
    if (lane == 31)
        warp_sums[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        const int nw = blockDim.x >> 5;
        int w = lane < nw ? warp_sums[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, w, o);
            if (lane >= o)
                w += y;
        }
        if (lane < nw)
            warp_sums[lane] = w;  // inclusive over warps
    }
    __syncthreads();
    int pos = incl - cnt + (warp > 0 ? warp_sums[warp - 1] : 0);
    for (int i = lo; i < hi; ++i)
        if (mask[i] != 0)
            row_ids[pos++] = i;
    if (threadIdx.x == blockDim.x - 1)
        *row_count = pos;
}

// CTA k copies the hidden state of packed row k (16-byte vectors).
__global__ void gather_rows_kernel(const int4 *hidden, int64_t vec_per_row, const int32_t *row_ids,
                                   const int32_t *row_count, int4 *packed)
{
    pdl_wait();  // the row list is complete
    if (threadIdx.x == 0)
        pdl_launch_dependents();  // the GEMM may start its prologue
    const int k = blockIdx.x;
    if (k >= *row_count)
        return;
    const int4 *src = hidden + (int64_t)row_ids[k] * vec_per_row;
    int4 *dst = packed + (int64_t)k * vec_per_row;
    for (int64_t i = threadIdx.x; i < vec_per_row; i += blockDim.x)
        dst[i] = __ldg(src + i);
}

struct Part {
    float M, S;
    uint32_t idx;
    bool nan;
};

// Fold of two partials: larger max, sums re-based to it, the lowest index attaining it.
// Symmetric, so both lanes of a shuffle step obtain the same bits.
__device__ __forceinline__ Part fold(const Part &x, const Part &y)
{
    Part r;
    r.nan = x.nan || y.nan;
    r.M = fmaxf(x.M, y.M);
    r.S = rebase(x.S, x.M, r.M) + rebase(y.S, y.M, r.M);
    const uint32_t ix = x.M == r.M ? x.idx : kNoIdx;
    const uint32_t iy = y.M == r.M ? y.idx : kNoIdx;
    r.idx = ix < iy ? ix : iy;
    return r;
}

// One CTA of kCombineWarps warps per packed row: lane l of warp q folds tiles
// q * 32 + l + 128 i (i = 0, 1, ...) in order, the lanes of each warp fold in a fixed
// butterfly, and the warps' results fold in warp order.  A fixed tree, so the result does not
// depend on timing.  Writes c = min(1/S, 1) and x_hat at the row's (b, l); a row with a NaN
// logit or an infinite maximum gets c = NaN, x_hat = -1.
constexpr int kCombineWarps = 4;

__global__ void __launch_bounds__(kCombineWarps * 32)
    combine_rows_kernel(const UnitPartial *partials, int n_tiles, const int32_t *row_ids,
                        const int32_t *row_count, float *conf, int32_t *tok)
{
    __shared__ Part s_part[kCombineWarps];
    pdl_wait();  // every tile partial is written
    if (threadIdx.x == 0)
        pdl_launch_dependents();
    const int r = blockIdx.x;
    const int lane = threadIdx.x & 31, q = threadIdx.x >> 5;
    if (r >= *row_count)
        return;
    Part acc{-__int_as_float(0x7F800000), 0.0f, kNoIdx, false};
    const UnitPartial *p = partials + (int64_t)r * n_tiles;
    constexpr int kStride = kCombineWarps * 32;
    constexpr int kBatch = 8;  // loads in flight per lane before the folds
    for (int j0 = q * 32 + lane; j0 < n_tiles; j0 += kStride * kBatch) {
        int4 v[kBatch];
#pragma unroll
        for (int b = 0; b < kBatch; ++b)
            if (j0 + kStride * b < n_tiles)
                v[b] = __ldcg(reinterpret_cast<const int4 *>(p + j0 + kStride * b));
#pragma unroll
        for (int b = 0; b < kBatch; ++b)
            if (j0 + kStride * b < n_tiles) {
                Part y{__int_as_float(v[b].x), __int_as_float(v[b].y), (uint32_t)v[b].z, false};
                y.nan = y.M != y.M;
                if (y.nan)
                    y.M = -__int_as_float(0x7F800000);
                acc = fold(acc, y);
            }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        Part y;
        y.M = __shfl_xor_sync(0xFFFFFFFFu, acc.M, o);
        y.S = __shfl_xor_sync(0xFFFFFFFFu, acc.S, o);
        y.idx = __shfl_xor_sync(0xFFFFFFFFu, acc.idx, o);
        y.nan = __shfl_xor_sync(0xFFFFFFFFu, (int)acc.nan, o) != 0;
        acc = fold(acc, y);
    }
    if (lane == 0)
        s_part[q] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        acc = s_part[0];
        for (int w = 1; w < kCombineWarps; ++w)
            acc = fold(acc, s_part[w]);
        const int row = row_ids[r];
        const bool finite = fabsf(acc.M) <= 3.402823466e38f && fabsf(acc.S) <= 3.402823466e38f;
        if (acc.nan || !finite || !(acc.S > 0.0f) || acc.idx == kNoIdx) {
            conf[row] = __int_as_float(0x7FC00000);
            tok[row] = -1;
        } else {
            conf[row] = fminf(1.0f / acc.S, 1.0f);
            tok[row] = (int32_t)acc.idx;
        }
    }
}

// ----------------------------------------------------------------------------- host side
// Workspace layout (offsets from the 256-byte aligned base; header shared with
// fdllm_select's layout: status at 0, the vocab reduction's counter at 4 left untouched):
//   row_count int32 at 8
//   row_ids   int32 [rows]
//   packed    bf16 [rows][H]            (1024-byte aligned: a TMA source)
//   partials  UnitPartial [rows][n_tiles]
//   conf      fp32 [rows], tok int32 [rows]
struct LmLayout {
    size_t row_count, row_ids, packed, partials, conf, tok, total;
};

size_t up(size_t x, size_t a) { return (x + a - 1) / a * a; }

LmLayout lm_layout(int64_t rows, int64_t H, int64_t n_tiles)
{
    LmLayout l;
    l.row_count = 8;
    l.row_ids = 256;
    l.packed = up(l.row_ids + (size_t)rows * 4, 1024);
    l.partials = up(l.packed + (size_t)rows * H * 2, 256);
    l.conf = up(l.partials + (size_t)rows * n_tiles * sizeof(UnitPartial), 256);
    l.tok = up(l.conf + (size_t)rows * 4, 256);
    l.total = up(l.tok + (size_t)rows * 4, 256);
    return l;
}

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                   const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                   const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return (EncodeTiledFn) nullptr;
        return reinterpret_cast<EncodeTiledFn>(p);
    }();
    return fn;
}

// bf16 matrix [outer][inner] (row stride inner * 2 bytes), loaded as boxes of
// {BK, box_outer} with 128-byte swizzling; out-of-range elements read as zero.
bool make_map(CUtensorMap *map, const void *base, int64_t inner, int64_t outer, int box_outer)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc)
        return false;
    const cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)outer};
    const cuuint64_t strides[1] = {(cuuint64_t)inner * 2};
    const cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_outer};
    const cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

// A launch as a programmatic dependent of the previous kernel on the stream (in plain
// stream order when pdl is false).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(bool pdl, void (*kern)(KArgs...), unsigned grid, unsigned block,
                       cudaStream_t stream, Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(block);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

fdllm_status check_lmhead(const void *hidden, const void *w, int B, int L, int H, int V,
                          const uint8_t *mask)
{
    if (B < 1 || L < 1 || L > FDLLM_MAX_L || (int64_t)B * L > FDLLM_MAX_ROWS || V < 1 || H < 8)
        return FDLLM_ERR_ARG;
    if (!hidden || !w || !mask)
        return FDLLM_ERR_ARG;
    if ((reinterpret_cast<uintptr_t>(hidden) & 15u) || (reinterpret_cast<uintptr_t>(w) & 15u) ||
        H % 8 != 0)
        return FDLLM_ERR_ALIGN;
    const int64_t n_tiles = (V + 207) / 208;  // the narrowest tile
    if ((int64_t)B * L * n_tiles >= ((int64_t)1 << 31) || (int64_t)H * 2 >= ((int64_t)1 << 31))
        return FDLLM_ERR_ARG;
    return FDLLM_OK;
}

int sm_count();
int choose_bn(int64_t rows, int V, bool pair);

// The slab variant's tile height: the multiple of 8 in [96, 128] that minimises the W rows
// of the busiest CTA, ceil(ceil(V / h) / P) * h with P = min(tiles, SMs); ties go to the
// taller tile (fewer, larger copies).  Heights below 96 would put too few W bytes in each
// stage to keep the stream going.
int slab_height(int V)
{
    const int64_t sms = sm_count();
    int best = 128;
    int64_t best_rows = -1;
    for (int h = 128; h >= 96; h -= 8) {
        const int64_t tiles = ((int64_t)V + h - 1) / h;
        const int64_t P = tiles < sms ? tiles : sms;
        const int64_t rows = (tiles + P - 1) / P * h;
        if (best_rows < 0 || rows < best_rows) {
            best = h;
            best_rows = rows;
        }
    }
    return best;
}

// The slab variant's grid: one CTA per SM, or one per tile if there are fewer.
int slab_grid(int V)
{
    const int64_t h = slab_height(V);
    const int64_t tiles = ((int64_t)V + h - 1) / h;
    return (int)(tiles < sm_count() ? tiles : sm_count());
}

// Rows of W per CTA on the longest-running SM, for the slab variant (whole tiles of its
// height) against the tile variant (one row tile: whole waves of vocabulary tiles times
// their width).  The slab variant's row operand is 4 KB per K-block where a row tile's is
// 16 KB, so more of each stage is W; measured on LLaDA-sized heads, it is faster when its
// busiest CTA streams no more rows.
bool slab_preferred(int V)
{
    const int64_t sms = sm_count();
    const int64_t h = slab_height(V);
    const int64_t tiles = ((int64_t)V + h - 1) / h;
    const int64_t P = tiles < sms ? tiles : sms;
    const int64_t slab_rows = (tiles + P - 1) / P * h;
    const int bn = choose_bn(1, V, false);
    const int64_t tile_rows = ((V + bn - 1) / bn + sms - 1) / sms * bn;
    return slab_rows <= tile_rows;
}

// The GEMM variant: for at most kSlabRows rows the slab variant where slab_preferred; else
// kPair (cta_group::2) when at least 8 row tiles can share every W tile, kSolo below that
// (the pair pads to an even number of row tiles, and W streaming from HBM, not
// shared-memory bandwidth, is the limit there).  FDLLM_LMHEAD_GEMM = solo, pair or slab
// forces one (slab only where B * L <= kSlabRows).
int gemm_mode(int64_t rows, int V)
{
    if (const char *e = std::getenv("FDLLM_LMHEAD_GEMM")) {
        const std::string v(e);
        if (v == "solo")
            return kSolo;
        if (v == "pair")
            return kPair;
        if (v == "slab" && rows <= kSlabRows)
            return kSlab;
    }
    if (rows <= kSlabRows && slab_preferred(V))
        return kSlab;
    return (rows + BM - 1) / BM >= 8 ? kPair : kSolo;
}

int sm_count()
{
    static std::once_flag once[64];
    static int cache[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64)
        return 152;
    std::call_once(once[dev], [&] {
        int n = 0;
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        cache[dev] = n > 0 ? n : 152;
    });
    return cache[dev];
}

// The vocabulary tile width with the least estimated time: whole waves of tiles over the
// SMs (row tiles estimated from B * L, the most the mask can hold) times the tile width.
// Ties go to 208 for one CTA per tile (measured 1.3-1.4 % faster at 4 estimated row tiles,
// B = 14 and 16 of 32 positions) and to 256 for the CTA pair (208 is slower there at every
// size).  FDLLM_LMHEAD_BN = 256 or 208 forces one.
int choose_bn(int64_t rows, int V, bool pair)
{
    if (const char *e = std::getenv("FDLLM_LMHEAD_BN")) {
        const int f = std::atoi(e);
        if (f == 256 || f == 208)
            return f;
    }
    const int64_t m_tiles = (rows + BM - 1) / BM, sms = sm_count();
    const int order[2] = {pair ? 256 : 208, pair ? 208 : 256};  // the first wins ties
    int best = order[0];
    int64_t best_cost = -1;
    for (int bn : order) {
        const int64_t tiles = (V + bn - 1) / bn * m_tiles;
        const int64_t cost = (tiles + sms - 1) / sms * bn;
        if (best_cost < 0 || cost < best_cost) {
            best = bn;
            best_cost = cost;
        }
    }
    return best;
}

template <int EPI, int MODE, int BN>
cudaError_t launch_gemm_cfg(const CUtensorMap &mh, const CUtensorMap &mw, const GemmArgs &g,
                            cudaStream_t stream)
{
    constexpr int CL = MODE == kSolo ? 1 : 2;
    static std::once_flag once[64];
    static int grid[64];
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess)
        return err;
    if (dev < 0 || dev >= 64)
        return cudaErrorInvalidDevice;
    auto kern = lmhead_gemm_kernel<EPI, MODE, BN>;
    constexpr size_t smem = TileCfg<BN, MODE>::kSmemBytes;
    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CL;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;  // the occupancy query below sees the cluster shape only
    std::call_once(once[dev], [&] {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        const int sms = sm_count();
        int clusters = 0;
        cfg.gridDim = dim3((unsigned)(sms / CL * CL));
        if (cudaOccupancyMaxActiveClusters(&clusters, kern, &cfg) != cudaSuccess || clusters < 1)
            clusters = sms / CL;
        (void)cudaGetLastError();
        grid[dev] = clusters * CL;  // persistent: every cluster resident at once
    });
    cfg.gridDim = dim3((unsigned)grid[dev]);
    cfg.numAttrs = g.pdl ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, kern, mh, mw, g);
}

template <int EPI, int MODE>
cudaError_t launch_gemm_mode(const CUtensorMap &mh, const CUtensorMap &mw, const GemmArgs &g,
                             int bn, cudaStream_t stream)
{
    return bn == 208 ? launch_gemm_cfg<EPI, MODE, 208>(mh, mw, g, stream)
                     : launch_gemm_cfg<EPI, MODE, 256>(mh, mw, g, stream);
}

template <int EPI>
cudaError_t launch_slab(const CUtensorMap &mh, const CUtensorMap &mw, const GemmArgs &g,
                        cudaStream_t stream)
{
    static std::once_flag once[64];
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess)
        return err;
    if (dev < 0 || dev >= 64)
        return cudaErrorInvalidDevice;
    auto kern = lmhead_slab_kernel<EPI>;
    std::call_once(once[dev], [&] {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kSlabSmemBytes);
    });
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)g.n_tiles);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSlabSmemBytes;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = g.pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kern, mh, mw, g);
}

template <int EPI>
cudaError_t launch_gemm(const CUtensorMap &mh, const CUtensorMap &mw, const GemmArgs &g,
                        int mode, int bn, cudaStream_t stream)
{
    if (mode == kSlab)
        return launch_slab<EPI>(mh, mw, g, stream);
    switch (mode) {
    case kPair: return launch_gemm_mode<EPI, kPair>(mh, mw, g, bn, stream);
    default: return launch_gemm_mode<EPI, kSolo>(mh, mw, g, bn, stream);
    }
}

// Steps 1-3 (and 4 for the reduce epilogue) on the owned workspace.
fdllm_status run_lmhead(const void *hidden, const void *w, int B, int L, int H, int V,
                        const uint8_t *mask, int epi, float *out_logits, cudaStream_t s,
                        uint8_t **ws_out, LmLayout *lay_out, bool pdl = true)
{
    const int64_t rows = (int64_t)B * L;
    const int mode = gemm_mode(rows, V);
    const int bn = mode == kSlab ? slab_height(V) : choose_bn(rows, V, mode == kPair);
    // partials per row: one per vocabulary tile, or one per CTA of the slab variant
    const int n_tiles = mode == kSlab ? slab_grid(V) : (V + bn - 1) / bn;
    const LmLayout lay = lm_layout(rows, H, n_tiles);
    void *wsv = nullptr;
    fdllm_status st = owned_workspace(lay.total, s, &wsv);
    if (st != FDLLM_OK)
        return st;
    uint8_t *ws = static_cast<uint8_t *>(wsv);
    int32_t *row_count = reinterpret_cast<int32_t *>(ws + lay.row_count);
    int32_t *row_ids = reinterpret_cast<int32_t *>(ws + lay.row_ids);
    uint8_t *packed = ws + lay.packed;

    CUtensorMap mh, mw;
    if (!make_map(&mh, packed, H, rows, mode == kSlab ? kSlabRows : BM) ||
        !make_map(&mw, w, H, V, mode == kSolo || mode == kSlab ? bn : bn / 2))
        return FDLLM_ERR_CUDA;

    if (launch_pdl(pdl, compact_rows_kernel, 1, 1024, s, mask, (int)rows, row_ids, row_count) !=
            cudaSuccess ||
        launch_pdl(pdl, gather_rows_kernel, (unsigned)rows, 128, s,
                   static_cast<const int4 *>(hidden), (int64_t)(H / 8),
                   (const int32_t *)row_ids, (const int32_t *)row_count,
                   reinterpret_cast<int4 *>(packed)) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    GemmArgs g;
    g.row_count = row_count;
    g.row_ids = row_ids;
    g.V = V;
    g.n_tiles = n_tiles;
    g.k_blocks = (H + BK - 1) / BK;
    g.slab_h = mode == kSlab ? bn : 0;
    g.slab_tiles = mode == kSlab ? (V + bn - 1) / bn : 0;
    g.partials = reinterpret_cast<UnitPartial *>(ws + lay.partials);
    g.logits = out_logits;
    g.status = reinterpret_cast<uint32_t *>(ws);
    g.pdl = pdl;
    const cudaError_t e = epi == kReduce ? launch_gemm<kReduce>(mh, mw, g, mode, bn, s)
                                         : launch_gemm<kStore>(mh, mw, g, mode, bn, s);
    if (e != cudaSuccess)
        return FDLLM_ERR_CUDA;
    if (epi == kReduce) {
        if (launch_pdl(pdl, combine_rows_kernel, (unsigned)rows, kCombineWarps * 32,
                       s, (const UnitPartial *)g.partials, n_tiles, (const int32_t *)row_ids,
                       (const int32_t *)row_count, reinterpret_cast<float *>(ws + lay.conf),
                       reinterpret_cast<int32_t *>(ws + lay.tok)) != cudaSuccess)
            return FDLLM_ERR_CUDA;
    }
    *ws_out = ws;
    *lay_out = lay;
    return FDLLM_OK;
}

// Copy of the confidences and argmax of the masked rows to caller arrays.
__global__ void scatter_conf_kernel(const float *conf, const int32_t *tok, const int32_t *row_ids,
                                    const int32_t *row_count, float *out_conf, int32_t *out_tok)
{
    pdl_wait();
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= *row_count)
        return;
    const int row = row_ids[k];
    out_conf[row] = conf[row];
    out_tok[row] = tok[row];
}

}  // namespace
}  // namespace fdllm

using namespace fdllm;

namespace fdllm {

fdllm_status lmhead_select_owned(const void *hidden, const void *w_vocab, int B, int L, int H,
                                 int V, uint8_t *mask, double param, int mode,
                                 int32_t *out_tokens, uint8_t *out_commit, int32_t *out_n,
                                 cudaStream_t s, bool pdl)
{
    fdllm_status st = check_lmhead(hidden, w_vocab, B, L, H, V, mask);
    if (st != FDLLM_OK)
        return st;
    if (!out_tokens || !out_commit || !out_n || !std::isfinite(param) ||
        (mode != FDLLM_PROFILE && mode != FDLLM_FACTOR && mode != FDLLM_THRESHOLD))
        return FDLLM_ERR_ARG;
    uint8_t *ws = nullptr;
    LmLayout lay;
    st = run_lmhead(hidden, w_vocab, B, L, H, V, mask, kReduce, nullptr, s, &ws, &lay, pdl);
    if (st != FDLLM_OK)
        return st;
    ProfileSelectArgs pa;
    pa.units_per_row = 0;
    pa.partials = nullptr;
    pa.next_unit = nullptr;
    pa.conf = reinterpret_cast<const float *>(ws + lay.conf);
    pa.tok = reinterpret_cast<const int32_t *>(ws + lay.tok);
    pa.mask = mask;
    pa.B = B;
    pa.L = L;
    pa.mode = mode;
    pa.param = param;
    pa.eta = 0.0;
    pa.eta_pos = nullptr;
    pa.out_tokens = out_tokens;
    pa.out_commit = out_commit;
    pa.out_n = out_n;
    pa.status = reinterpret_cast<uint32_t *>(ws);
    pa.pdl = pdl;
    return launch_profile_select(pa, s) == cudaSuccess ? FDLLM_OK : FDLLM_ERR_CUDA;
}

}  // namespace fdllm

extern "C" {

fdllm_status fdllm_lmhead_select(const void *hidden, const void *w_vocab, int B, int L, int H,
                                 int V, uint8_t *mask, double param, int mode,
                                 int32_t *out_tokens, uint8_t *out_commit, int32_t *out_n,
                                 void *stream)
{
    return lmhead_select_owned(hidden, w_vocab, B, L, H, V, mask, param, mode, out_tokens,
                               out_commit, out_n, static_cast<cudaStream_t>(stream), true);
}

fdllm_status fdllm_lmhead_confidence(const void *hidden, const void *w_vocab, int B, int L,
                                     int H, int V, const uint8_t *mask, float *out_conf,
                                     int32_t *out_argmax, void *stream)
{
    fdllm_status st = check_lmhead(hidden, w_vocab, B, L, H, V, mask);
    if (st != FDLLM_OK)
        return st;
    if (!out_conf || !out_argmax)
        return FDLLM_ERR_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    uint8_t *ws = nullptr;
    LmLayout lay;
    st = run_lmhead(hidden, w_vocab, B, L, H, V, mask, kReduce, nullptr, s, &ws, &lay);
    if (st != FDLLM_OK)
        return st;
    const int64_t rows = (int64_t)B * L;
    return launch_pdl(true, scatter_conf_kernel, (unsigned)((rows + 255) / 256), 256, s,
                      reinterpret_cast<const float *>(ws + lay.conf),
                      reinterpret_cast<const int32_t *>(ws + lay.tok),
                      reinterpret_cast<const int32_t *>(ws + lay.row_ids),
                      reinterpret_cast<const int32_t *>(ws + lay.row_count), out_conf,
                      out_argmax) == cudaSuccess
               ? FDLLM_OK
               : FDLLM_ERR_CUDA;
}

fdllm_status fdllm_lmhead_logits(const void *hidden, const void *w_vocab, int B, int L, int H,
                                 int V, const uint8_t *mask, float *out_logits, void *stream)
{
    fdllm_status st = check_lmhead(hidden, w_vocab, B, L, H, V, mask);
    if (st != FDLLM_OK)
        return st;
    if (!out_logits)
        return FDLLM_ERR_ARG;
    uint8_t *ws = nullptr;
    LmLayout lay;
    return run_lmhead(hidden, w_vocab, B, L, H, V, mask, kStore, out_logits,
                      static_cast<cudaStream_t>(stream), &ws, &lay);
}

}  // extern "C"

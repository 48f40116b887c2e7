// vocab_reduce.cu -- step a1 of the selection: for every masked position, the argmax token
// x_hat (lowest index on ties) and the confidence c = max_v softmax(v) = exp(M - lse)
// (paper Sec. 3 "Notation"; Algorithm 1, confidence loop).
//
// Design (an HBM-bound streaming reduction; no tensor cores):
//  * Work = the masked rows only.  Every CTA compacts the mask into a bitmap plus word prefix
//    counts in shared memory and maps the r-th masked row to its global row.
//  * Each row is cut into fixed units (128 KB, or 64 KB for small steps, see plan_units);
//    the units of all masked rows form one queue served by an atomic counter, so CTAs that
//    run faster take more units and the tail is at most one unit.  A producer requests its
//    next unit before it issues the current one's copies and reads the answer after, so
//    the counter's round trip overlaps the copies.  A unit is reduced by one CTA in a fixed
//    order, so a row's result depends only on its bytes and the call's shape (identical rows
//    give identical bits, for any mask).
//  * Warp 0 (one lane) streams each unit through a kStages-deep ring of kChunkBytes buffers
//    with 1-D bulk copies (cp.async.bulk, completion on mbarriers); chunk metadata travels
//    with the stage.
//  * NW math warps read the ring with conflict-free 16-byte shared loads.  Per lane: running
//    max and the index of its first maximal logit; per warp: a lagging reference `ref` for
//    the sum of 2^(x*log2e - ref2), raised (with one rescale) only when a logit exceeds it by
//    kRebaseSlack, so a logit costs half a packed f32x2 FMA, one MUFU ex2 and half a packed
//    f32x2 add; the vector max uses packed bf16x2 / f16x2 max for 16-bit logits.  Beyond
//    |ref| = kBigRef the same FMA runs with scale 1 (see rebase_scaled).
//  * At the end of a unit each math warp reduces its lanes (redux + shuffles) and queues
//    (M, S, idx), S re-based to M exactly, for the epilogue warp, which combines the warps in
//    a fixed order and stores the unit's partial.  The consumer kernel (profile select, or
//    finalize) folds a position's units in unit order.
//  * The work counter is put back to zero by the launch's last fetch, so the kernel leaves
//    the workspace ready for the next launch by itself (the consumer kernels reset it too,
//    which also covers a launch that gave up a bounded wait).
#include <cfloat>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <mutex>
#include <type_traits>

#include "fdllm_internal.cuh"
#include "ptx.cuh"

namespace fdllm {
namespace {

// A warp raises its sum reference only when a logit exceeds it by this much (natural-log
// units); lane sums then stay below (terms per lane) * e^8, far from fp32 overflow.
constexpr float kRebaseSlack = 8.0f;
constexpr uint32_t kEndMarker = 0xFFFFFFFFu;

__device__ __forceinline__ float fmax_nan(float a, float b)
{
    float r;
    asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
    return r;
}

// Monotone map of floats onto unsigned integers (for warp max via redux).
__device__ __forceinline__ uint32_t ordered(float f)
{
    const uint32_t b = __float_as_uint(f);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

__device__ __forceinline__ float unordered(uint32_t k)
{
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

__device__ __forceinline__ uint32_t hmax2_nan(uint32_t a, uint32_t b)
{
    uint32_t d;
    asm("max.NaN.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

__device__ __forceinline__ uint32_t hmax2_nan_f16(uint32_t a, uint32_t b)
{
    uint32_t d;
    asm("max.NaN.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

// fp16 (IEEE binary16) -> fp32, exact.
__device__ __forceinline__ float f16_to_f32(uint32_t h)
{
    float f;
    asm("{\n\t.reg .b16 x;\n\tcvt.u16.u32 x, %1;\n\tcvt.f32.f16 %0, x;\n\t}"
        : "=f"(f)
        : "r"(h));
    return f;
}

// Packed fp32 pairs (Blackwell f32x2 arithmetic); element order inside a pair is irrelevant
// here because every operation is elementwise.
__device__ __forceinline__ uint64_t pack2(float lo, float hi)
{
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}

__device__ __forceinline__ void unpack2(uint64_t v, float &lo, float &hi)
{
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}

__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c)
{
    uint64_t d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}

__device__ __forceinline__ uint64_t fadd2(uint64_t a, uint64_t b)
{
    uint64_t d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}

__device__ __forceinline__ uint64_t fmul2(uint64_t a, uint64_t b)
{
    uint64_t d;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}

// Keyed by the library's dtype code (fdllm_dtype).
template <int KIND>
struct VecOps;

template <>
struct VecOps<FDLLM_BF16> {  // 8 x bf16 per 16-byte vector; widening to fp32 is exact
    static constexpr uint32_t kPadWord = 0xFF80FF80u;  // two bf16 -inf
    // max of the 8 logits; NaN if any is NaN
    __device__ __forceinline__ static float vmax(const uint4 &r)
    {
        const uint32_t m = hmax2_nan(hmax2_nan(r.x, r.y), hmax2_nan(r.z, r.w));
        return fmax_nan(__uint_as_float(m << 16), __uint_as_float(m & 0xFFFF0000u));
    }
    __device__ __forceinline__ static uint64_t pair(uint32_t w)
    {
        return pack2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
    }
    __device__ __forceinline__ static void pairs(const uint4 &r, uint64_t (&p)[4])
    {
        p[0] = pair(r.x);
        p[1] = pair(r.y);
        p[2] = pair(r.z);
        p[3] = pair(r.w);
    }
    // first element of the vector equal to M (8 if none)
    __device__ __forceinline__ static uint32_t first_index(const uint4 &r, float M)
    {
        const uint32_t w[4] = {r.x, r.y, r.z, r.w};
        uint32_t hit = 8;
#pragma unroll
        for (int e = 7; e >= 0; --e) {
            const uint32_t bits = (e & 1) ? (w[e >> 1] & 0xFFFF0000u) : (w[e >> 1] << 16);
            if (__uint_as_float(bits) == M)
                hit = e;
        }
        return hit;
    }
    static constexpr int kPairs = 4;
    static constexpr int kElems = 8;
};

template <>
struct VecOps<FDLLM_FP16> {  // 8 x fp16 per 16-byte vector; widening to fp32 is exact
    static constexpr uint32_t kPadWord = 0xFC00FC00u;  // two fp16 -inf
    // max of the 8 logits; NaN if any is NaN
    __device__ __forceinline__ static float vmax(const uint4 &r)
    {
        const uint32_t m = hmax2_nan_f16(hmax2_nan_f16(r.x, r.y), hmax2_nan_f16(r.z, r.w));
        return fmax_nan(f16_to_f32(m & 0xFFFFu), f16_to_f32(m >> 16));
    }
    __device__ __forceinline__ static uint64_t pair(uint32_t w)
    {
        return pack2(f16_to_f32(w & 0xFFFFu), f16_to_f32(w >> 16));
    }
    __device__ __forceinline__ static void pairs(const uint4 &r, uint64_t (&p)[4])
    {
        p[0] = pair(r.x);
        p[1] = pair(r.y);
        p[2] = pair(r.z);
        p[3] = pair(r.w);
    }
    // first element of the vector equal to M (8 if none)
    __device__ __forceinline__ static uint32_t first_index(const uint4 &r, float M)
    {
        const uint32_t w[4] = {r.x, r.y, r.z, r.w};
        uint32_t hit = 8;
#pragma unroll
        for (int e = 7; e >= 0; --e) {
            const uint32_t bits = (e & 1) ? (w[e >> 1] >> 16) : (w[e >> 1] & 0xFFFFu);
            if (f16_to_f32(bits) == M)
                hit = e;
        }
        return hit;
    }
    static constexpr int kPairs = 4;
    static constexpr int kElems = 8;
};

template <>
struct VecOps<FDLLM_FP32> {  // 4 x fp32 per 16-byte vector
    static constexpr uint32_t kPadWord = 0xFF800000u;  // fp32 -inf
    __device__ __forceinline__ static float vmax(const uint4 &r)
    {
        return fmax_nan(fmax_nan(__uint_as_float(r.x), __uint_as_float(r.y)),
                        fmax_nan(__uint_as_float(r.z), __uint_as_float(r.w)));
    }
    __device__ __forceinline__ static void pairs(const uint4 &r, uint64_t (&p)[2])
    {
        p[0] = ((uint64_t)r.y << 32) | r.x;
        p[1] = ((uint64_t)r.w << 32) | r.z;
    }
    __device__ __forceinline__ static uint32_t first_index(const uint4 &r, float M)
    {
        const uint32_t w[4] = {r.x, r.y, r.z, r.w};
        uint32_t hit = 4;
#pragma unroll
        for (int e = 3; e >= 0; --e)
            if (__uint_as_float(w[e]) == M)
                hit = e;
        return hit;
    }
    static constexpr int kPairs = 2;
    static constexpr int kElems = 4;
};

// Partials held by lanes [0, count) (each S relative to its own M) -> one partial, combined
// by a fixed butterfly.
__device__ __forceinline__ UnitPartial warp_combine(UnitPartial p, bool valid)
{
    if (!valid) {
        p.M = -INFINITY;
        p.S = 0.0f;
        p.idx = kNoIdx;
    }
    const float M = unordered(__reduce_max_sync(0xFFFFFFFFu, ordered(p.M)));
    float s = rebase(p.S, p.M, M);
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1)
        s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
    UnitPartial r;
    r.M = M;
    r.S = s;
    r.idx = __reduce_min_sync(0xFFFFFFFFu, p.M == M ? p.idx : kNoIdx);
    r.pad = 0;
    return r;
}

// Global row of the r-th masked row: the word holding it by binary search over the
// exclusive word prefix counts, then the bit by rank within the word.
__device__ __forceinline__ int64_t masked_row(uint32_t r, const uint32_t *bits,
                                              const uint32_t *pref, int nwords)
{
    int lo = 0, hi = nwords - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (pref[mid] <= r)
            lo = mid;
        else
            hi = mid - 1;
    }
    const int bit = (int)__fns(bits[lo], 0, (int)(r - pref[lo]) + 1);
    return (int64_t)lo * 32 + bit;
}

// Bit j of the result = byte j of x is nonzero (j = 0..3): each byte folded onto its bit 0,
// then the four bits gathered by one multiply (the partial products land on distinct bits
// below 24, so bits 24-27 carry no interference).
__device__ __forceinline__ uint32_t nonzero_bytes4(uint32_t x)
{
    uint32_t t = x | (x >> 4);
    t |= t >> 2;
    t |= t >> 1;
    t &= 0x01010101u;
    return ((t * 0x01020408u) >> 24) & 0xFu;
}

struct ChunkMeta {
    uint32_t n;         // vectors in the chunk; 0 marks the end of the CTA's work
    uint32_t vec_base;  // row-relative index of the chunk's first vector
    uint32_t last;      // nonzero: last chunk of its unit
    uint32_t pidx;      // partial slot of the unit: global row * units_per_row + unit
};

template <int NW, int STAGES>
struct Smem {
    uint64_t full[STAGES];
    uint64_t empty[STAGES];
    uint64_t seg_full[kSegQueue];
    uint64_t seg_empty[kSegQueue];
    ChunkMeta meta[STAGES];
    UnitPartial seg[kSegQueue][NW];
    uint32_t seg_pidx[kSegQueue];
    uint32_t bits[kMaskWords];
    uint32_t pref[kMaskWords + 1];
};

template <int NW, int STAGES, int CHUNK>
constexpr size_t smem_bytes()
{
    return (size_t)STAGES * CHUNK + sizeof(Smem<NW, STAGES>);
}

// KIND: the logits' dtype code; NW: math warps; STAGES x CHUNK: the shared-memory ring;
// EVICT: L2 evict-first hint on the stream.
template <int KIND, int NW, int STAGES, int CHUNK, bool EVICT>
__global__ void __launch_bounds__((NW + 2) * 32, 1) vocab_reduce_kernel(const VocabReduceArgs a)
{
    constexpr int kStages = STAGES;
    constexpr int kChunkBytes = CHUNK;
    constexpr int kChunkVecs = CHUNK / 16;
    extern __shared__ __align__(128) uint8_t smem_raw[];
    uint8_t *ring = smem_raw;
    Smem<NW, STAGES> &sm =
        *reinterpret_cast<Smem<NW, STAGES> *>(smem_raw + (size_t)kStages * kChunkBytes);
    constexpr int kWarps = NW + 2;
    using Ops = VecOps<KIND>;
    constexpr int kP = Ops::kPairs;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&sm.full[s], 1);
            mbar_init(&sm.empty[s], NW);
        }
        for (int q = 0; q < kSegQueue; ++q) {
            mbar_init(&sm.seg_full[q], NW);
            mbar_init(&sm.seg_empty[q], 1);
        }
        fence_mbar_init();
    }
    // Launched as a programmatic dependent of the previous kernel: its writes (mask, logits,
    // this workspace's counter) are visible after this wait.  The consumer kernel of this
    // grid may start launching now; it waits for this grid's results itself.
    pdl_wait();
    if (threadIdx.x == 0)
        pdl_launch_dependents();

    const uint32_t upr = (uint32_t)a.units_per_row;
    const int nwords = (int)((a.rows + 31) / 32);

    // The producer's first unit (unit blockIdx.x: masked row blockIdx.x / upr) is located by
    // the producer warp alone, with a ballot scan of the mask, and its copies are issued
    // before the CTA-wide mask compaction below: the first data is in flight while the other
    // warps build the bitmap.
    uint32_t k = 0;  // producer: chunks issued so far
    uint64_t policy = 0;
    auto issue_unit = [&](uint32_t u, int64_t grow) -> bool {
        const uint32_t j = u % upr;
        const int64_t v0 = (int64_t)j * a.unit_vecs;
        const int64_t v1 = min(v0 + (int64_t)a.unit_vecs, a.vec_per_row);
        const uint8_t *rowp = a.logits + grow * a.row_bytes;
        for (int64_t v = v0; v < v1; v += kChunkVecs) {
            const uint32_t n = (uint32_t)min((int64_t)kChunkVecs, v1 - v);
            const uint32_t s = k % kStages;
            if (k >= kStages && !mbar_wait(&sm.empty[s], ((k / kStages) - 1) & 1, a.status))
                return false;  // the math warps stopped consuming; the caller drains
            ChunkMeta cm;
            cm.n = n;
            cm.vec_base = (uint32_t)v;
            cm.last = (v + n == v1) ? 1u : 0u;
            cm.pidx = (uint32_t)(grow * upr + j);
            sm.meta[s] = cm;
            mbar_arrive_expect_tx(&sm.full[s], n * 16u);
            if (EVICT)
                bulk_copy_g2s_hint(ring + (size_t)s * kChunkBytes, rowp + v * 16, n * 16u,
                                   &sm.full[s], policy);
            else
                bulk_copy_g2s(ring + (size_t)s * kChunkBytes, rowp + v * 16, n * 16u,
                              &sm.full[s]);
            ++k;
        }
        return true;
    };
    bool first_tried = false, first_issued = false;
    uint32_t u_next = 0;
    if (warp == 0) {
        if (EVICT)
            policy = make_evict_first_policy();
        const uint32_t kth = blockIdx.x / upr;
        int64_t grow = -1;
        // A bounded scan of the first kScanRows rows in one memory round trip: lane l reads
        // rows [16 l, 16 l + 16) (one 16-byte load where the mask allows, byte loads at a
        // ragged end or an unaligned mask), then a warp scan of the per-lane counts finds the
        // kth masked row.  With fewer masked rows there, the first unit is issued after the
        // compaction instead (below), which the other warps finish in about the same time.
        constexpr int64_t kScanRows = 512;
        const int64_t scan_end = a.rows < kScanRows ? a.rows : kScanRows;
        const int64_t r0 = (int64_t)lane * 16;
        uint32_t bits16 = 0;
        if ((reinterpret_cast<uintptr_t>(a.mask) & 15u) == 0 && r0 + 16 <= scan_end) {
            const uint4 v = __ldcg(reinterpret_cast<const uint4 *>(a.mask + r0));
            bits16 = nonzero_bytes4(v.x) | (nonzero_bytes4(v.y) << 4) |
                     (nonzero_bytes4(v.z) << 8) | (nonzero_bytes4(v.w) << 12);
        } else {
            for (int j = 0; j < 16 && r0 + j < scan_end; ++j)
                bits16 |= (a.mask[r0 + j] != 0 ? 1u : 0u) << j;
        }
        const uint32_t cnt = (uint32_t)__popc(bits16);
        uint32_t incl = cnt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (lane >= o)
                incl += t;
        }
        const bool here = kth >= incl - cnt && kth < incl;
        const uint32_t who = __ballot_sync(0xFFFFFFFFu, here);
        const int64_t cand =
            here ? r0 + (int64_t)__fns(bits16, 0, (int)(kth - (incl - cnt)) + 1) : (int64_t)-1;
        if (who != 0u)
            grow = __shfl_sync(0xFFFFFFFFu, cand, __ffs(who) - 1);
        if (grow >= 0) {
            first_tried = true;
            if (lane == 0) {
                // the first unit's copies go out first; the queue request for the next unit
                // is then in flight while they stream (its value is read only later)
                first_issued = issue_unit(blockIdx.x, grow);
                u_next = gridDim.x + atomicAdd(a.next_unit, 1u);
            }
        }
    } else {
        // Mask -> bitmap (one ballot per 32 rows, four words in flight per warp) -> exclusive
        // prefix count per word, by every warp but the producer's.
        constexpr int kBuilders = kWarps - 1;
        const int bw = warp - 1;
        for (int w0 = bw; w0 < nwords; w0 += 4 * kBuilders) {
            bool m[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int w = w0 + i * kBuilders;
                const int64_t r = (int64_t)w * 32 + lane;
                m[i] = w < nwords && r < a.rows && a.mask[r] != 0;
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint32_t b = __ballot_sync(0xFFFFFFFFu, m[i]);
                if (lane == 0 && w0 + i * kBuilders < nwords)
                    sm.bits[w0 + i * kBuilders] = b;
            }
        }
        asm volatile("bar.sync 1, %0;" ::"r"(kBuilders * 32) : "memory");
        if (warp == 1) {
            const int per = (nwords + 31) / 32;
            const int w0 = lane * per;
            uint32_t local = 0;
            for (int q = 0; q < per; ++q)
                if (w0 + q < nwords)
                    local += __popc(sm.bits[w0 + q]);
            uint32_t incl = local;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
                if (lane >= o)
                    incl += t;
            }
            uint32_t run = incl - local;
            for (int q = 0; q < per; ++q)
                if (w0 + q < nwords) {
                    sm.pref[w0 + q] = run;
                    run += __popc(sm.bits[w0 + q]);
                }
            if (lane == 31)
                sm.pref[nwords] = incl;
        }
    }
    __syncthreads();

    const uint32_t total = sm.pref[nwords] * upr;  // host checks rows * upr < 2^31
    if (total == 0)
        return;

    if (warp == 0) {
        // ------------------------------------------------------------ producer (one lane)
        if (lane != 0)
            return;
        // Every CTA that has a first unit fetches from the queue until it draws a unit past
        // the last one: the launch makes exactly n_fetch fetches, and the one drawing
        // n_fetch - 1 is the last, after which the counter is put back to zero for the next
        // launch.
        const uint32_t G = gridDim.x;
        const uint32_t n_fetch = (total > G ? total - G : 0u) + (total < G ? total : G);
        auto fetched = [&](uint32_t u) {
            if (u - G == n_fetch - 1u)
                *a.next_unit = 0;
            return u;
        };
        bool alive = true;  // false once a bounded wait has given up
        if (first_tried) {
            u_next = fetched(u_next);
            alive = first_issued;
        } else if (blockIdx.x < total) {
            // the first unit was not within the producer's scan
            u_next = fetched(G + atomicAdd(a.next_unit, 1u));
            first_issued = issue_unit(blockIdx.x,
                                      masked_row(blockIdx.x / upr, sm.bits, sm.pref, nwords));
            alive = first_issued;
        }
        if (first_issued) {
            // Then the work queue, which hands out units gridDim.x, gridDim.x + 1, ...
            uint32_t u = u_next;
            while (u < total) {
                // the request for the unit after u is in flight while u's copies are issued
                const uint32_t raw = atomicAdd(a.next_unit, 1u);
                if (!issue_unit(u, masked_row(u / upr, sm.bits, sm.pref, nwords))) {
                    alive = false;
                    break;
                }
                u = fetched(G + raw);
            }
        }
        if (alive) {
            const uint32_t s = k % kStages;
            if (k < kStages || mbar_wait(&sm.empty[s], ((k / kStages) - 1) & 1, a.status)) {
                ChunkMeta end;
                end.n = 0;
                end.vec_base = 0;
                end.last = 1;
                end.pidx = kEndMarker;
                sm.meta[s] = end;
                mbar_arrive(&sm.full[s]);
            } else {
                alive = false;
            }
        }
        if (!alive) {
            // A bounded wait gave up.  Copies already issued still write this CTA's shared
            // memory, so before the producer lets the CTA exit it waits (bounded again) for
            // the last chunk issued into each stage; every earlier chunk of a stage completed
            // before the stage was reused.
            for (uint32_t c = k > (uint32_t)kStages ? k - (uint32_t)kStages : 0u; c < k; ++c)
                mbar_wait(&sm.full[c % kStages], (c / kStages) & 1u, a.status, kDrainLimitNs);
        }
    } else if (warp <= NW) {
        // ------------------------------------------------------------ math warps
        const int mw = warp - 1;
        const int ct = threadIdx.x - 32;
        constexpr int kPer = kChunkVecs / (NW * 32);
        static_assert(kChunkVecs % (NW * 32) == 0, "chunk must split evenly over math warps");
        float m = -INFINITY;     // lane max (the first logit attaining it wins ties)
        float mnan = -INFINITY;  // lane max propagating NaN (NaN detection, rebase trigger)
        uint32_t idx = kNoIdx;   // row-relative index of that first logit
        uint64_t acc[kP];
        // Warp-uniform reference ref, its fp32 form ref2 and the scale sc of rebase_scaled
        // (sc = log2e, or 1 for |ref| >= kBigRef).  Before the first finite logit ref = -inf,
        // so that logit always rebases, and the sums stay 0.
        float ref = -INFINITY, ref2 = -FLT_MAX, sc = kLog2e;
        uint64_t sc2 = pack2(kLog2e, kLog2e);
#pragma unroll
        for (int q = 0; q < kP; ++q)
            acc[q] = 0;

        // One chunk: vector maxima and the first maximal logit, the reference update, then
        // 2^(x*sc - ref2) accumulated.  FULL: every vector of the chunk exists.
        auto process_chunk = [&](auto full_tag, const uint4 *buf, const ChunkMeta &cm) {
            constexpr bool FULL = decltype(full_tag)::value;
            const uint4 pad = make_uint4(Ops::kPadWord, Ops::kPadWord, Ops::kPadWord,
                                         Ops::kPadWord);
            uint4 raw[kPer];
#pragma unroll
            for (int it = 0; it < kPer; ++it) {
                const int v = ct + it * NW * 32;
                raw[it] = (FULL || v < (int)cm.n) ? buf[v] : pad;
            }
            float vm[kPer];
            int vi[kPer];
#pragma unroll
            for (int it = 0; it < kPer; ++it) {
                vm[it] = Ops::vmax(raw[it]);
                vi[it] = it;
                mnan = fmax_nan(mnan, vm[it]);
            }
#pragma unroll
            for (int w = 1; w < kPer; w *= 2)
#pragma unroll
                for (int it = 0; it + w < kPer; it += 2 * w)
                    if (vm[it + w] > vm[it]) {
                        vm[it] = vm[it + w];
                        vi[it] = vi[it + w];
                    }
            if (vm[0] > m) {  // rare after a unit's first chunk
                // the winning vector is still in the ring (the stage is not released yet)
                const int v = ct + vi[0] * NW * 32;
                m = vm[0];
                idx = (cm.vec_base + (uint32_t)v) * Ops::kElems + Ops::first_index(buf[v], m);
            }
            if (__any_sync(0xFFFFFFFFu, mnan > ref + kRebaseSlack)) {
                const float wmax = unordered(__reduce_max_sync(0xFFFFFFFFu, ordered(mnan)));
                const bool big = !(fabsf(wmax) < kBigRef);
                const float r2 = big ? wmax : wmax * kLog2e;
                // Old sums -> the new reference: 2^(ref2 - r2) between two fp32 references.
                // Where either reference has magnitude >= kBigRef every old logit lies at
                // least 56 below the new maximum and the old terms are dropped (under e^-56
                // each); the first sums are 0.
                const float f = (big || sc != kLog2e) ? 0.0f : ex2_mufu(ref2 - r2);
                const uint64_t f2 = pack2(f, f);
#pragma unroll
                for (int q = 0; q < kP; ++q)
                    acc[q] = fmul2(acc[q], f2);
                ref = wmax;
                ref2 = r2;
                sc = big ? 1.0f : kLog2e;
                sc2 = pack2(sc, sc);
            }
            const uint64_t nref2 = pack2(-ref2, -ref2);
#pragma unroll
            for (int it = 0; it < kPer; ++it) {
                uint64_t p[kP];
                Ops::pairs(raw[it], p);
#pragma unroll
                for (int q = 0; q < kP; ++q) {
                    float t0, t1;
                    unpack2(ffma2(p[q], sc2, nref2), t0, t1);
                    acc[q] = fadd2(acc[q], pack2(ex2_mufu(t0), ex2_mufu(t1)));
                }
            }
        };
        uint32_t seg = 0;
        for (uint32_t k = 0;; ++k) {
            const uint32_t st = k % kStages;
            if (!mbar_wait(&sm.full[st], (k / kStages) & 1, a.status))
                return;
            const ChunkMeta cm = sm.meta[st];
            if (cm.n != 0) {
                const uint4 *buf =
                    reinterpret_cast<const uint4 *>(ring + (size_t)st * kChunkBytes);
                if (cm.n == (uint32_t)kChunkVecs)
                    process_chunk(std::true_type{}, buf, cm);
                else
                    process_chunk(std::false_type{}, buf, cm);
            }
            __syncwarp();
            if (cm.n != 0 && lane == 0)
                mbar_arrive(&sm.empty[st]);
            if (!cm.last)
                continue;
            // end of a unit (or of the CTA's work): hand the warp's result to the epilogue
            const uint32_t q = seg % kSegQueue;
            if (seg >= kSegQueue &&
                !mbar_wait(&sm.seg_empty[q], ((seg / kSegQueue) - 1) & 1, a.status))
                return;
            float S = 0.0f;
#pragma unroll
            for (int j = 0; j < kP; ++j) {
                float lo, hi;
                unpack2(acc[j], lo, hi);
                S += lo + hi;
            }
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1)
                S += __shfl_xor_sync(0xFFFFFFFFu, S, o);
            UnitPartial p;
            p.M = unordered(__reduce_max_sync(0xFFFFFFFFu, ordered(m)));
            // NaN anywhere poisons the sum; a warp that saw no finite logit adds exactly 0.
            const bool bad = __any_sync(0xFFFFFFFFu, mnan != mnan);
            p.S = bad ? __int_as_float(0x7FC00000)
                      : (p.M == -INFINITY ? 0.0f : rebase_scaled(S, sc, ref2, p.M));
            p.idx = __reduce_min_sync(0xFFFFFFFFu, m == p.M ? idx : kNoIdx);
            p.pad = 0;
            if (lane == 0) {
                sm.seg[q][mw] = p;
                if (mw == 0)
                    sm.seg_pidx[q] = cm.pidx;
                mbar_arrive(&sm.seg_full[q]);
            }
            if (cm.n == 0)
                return;
            ++seg;
            m = -INFINITY;
            mnan = -INFINITY;
            idx = kNoIdx;
            ref = -INFINITY;
            ref2 = -FLT_MAX;
            sc = kLog2e;
            sc2 = pack2(kLog2e, kLog2e);
#pragma unroll
            for (int j = 0; j < kP; ++j)
                acc[j] = 0;
        }
    } else {
        // ------------------------------------------------------------ epilogue warp
        for (uint32_t seg = 0;; ++seg) {
            const uint32_t q = seg % kSegQueue;
            if (!mbar_wait(&sm.seg_full[q], (seg / kSegQueue) & 1, a.status))
                return;
            const uint32_t pidx = sm.seg_pidx[q];
            UnitPartial p = {-INFINITY, 0.0f, kNoIdx, 0};
            if (lane < NW)
                p = sm.seg[q][lane];
            __syncwarp();
            if (lane == 0)
                mbar_arrive(&sm.seg_empty[q]);
            if (pidx == kEndMarker)
                return;
            p = warp_combine(p, lane < NW);
            if (lane == 0)
                a.partials[pidx] = p;
        }
    }
}

__global__ void finalize_kernel(const FinalizeArgs a)
{
    pdl_wait();  // the vocab reduction's partials are complete and visible
    if (threadIdx.x == 0)
        pdl_launch_dependents();  // a following vocab reduction may start its prologue
    if (blockIdx.x == 0 && threadIdx.x == 0)
        *a.next_unit = 0;
    const int64_t row = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (row >= a.rows)
        return;
    // The mask byte and the partials are loaded together; an unmasked row's partials are
    // in-bounds leftovers and are discarded.
    const bool masked = a.mask[row] != 0;
    float c;
    int32_t tok;
    combine_position(a.partials + row * a.units_per_row, a.units_per_row, c, tok);
    if (!masked)
        return;
    a.out_conf[row] = c;
    a.out_tok[row] = tok;
}

template <int KIND, int NW, int STAGES, int CHUNK, bool EVICT>
cudaError_t launch_variant(const VocabReduceArgs &a, cudaStream_t stream)
{
    // Per device, once (host threads may make their first calls concurrently): the shared
    // memory attribute and the grid of every CTA resident at once.
    static std::once_flag once[64];
    static cudaError_t setup_err[64];
    static int grid_cache[64];
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess)
        return err;
    if (dev < 0 || dev >= 64)
        return cudaErrorInvalidDevice;
    constexpr size_t smem = smem_bytes<NW, STAGES, CHUNK>();
    static_assert(smem <= 227 * 1024, "ring does not fit in shared memory");
    auto *kern = vocab_reduce_kernel<KIND, NW, STAGES, CHUNK, EVICT>;
    std::call_once(once[dev], [&] {
        setup_err[dev] =
            cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        int sms = 0, per_sm = 0;
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, (NW + 2) * 32, smem);
        (void)cudaGetLastError();
        const int g = (sms > 0 ? sms : 1) * (per_sm > 0 ? per_sm : 1);
        grid_cache[dev] = g < kMaxGrid ? g : kMaxGrid;
    });
    if (setup_err[dev] != cudaSuccess)
        return setup_err[dev];
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid_cache[dev]);
    cfg.blockDim = dim3((NW + 2) * 32);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = a.pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

// Tuning table (math warps, ring stages x chunk bytes, L2 hint).  Entry 0 is the
// configuration in use; FDLLM_K1_VARIANT=<index> selects another for measurements.
template <int KIND>
cudaError_t launch_kind(const VocabReduceArgs &a, cudaStream_t stream, int which)
{
    switch (which) {
    case 1: return launch_variant<KIND, 16, 3, 65536, false>(a, stream);
    case 2: return launch_variant<KIND, 8, 3, 65536, true>(a, stream);
    case 3: return launch_variant<KIND, 16, 6, 32768, true>(a, stream);
    default: return launch_variant<KIND, 16, 3, 65536, true>(a, stream);
    }
}

int variant_index()
{
    static const int v = [] {
        const char *e = std::getenv("FDLLM_K1_VARIANT");
        return e ? std::atoi(e) : 0;
    }();
    return v;
}

// Health check of the bounded waits: one thread waits on an mbarrier that nobody arrives
// at, so the wait must run out after limit_ns, record kDevStatTimeout and return.
__global__ void bounded_wait_probe_kernel(uint32_t *status, uint64_t limit_ns)
{
    __shared__ uint64_t bar;
    mbar_init(&bar, 1);
    fence_mbar_init();
    mbar_wait(&bar, 0, status, limit_ns);
}

}  // namespace

cudaError_t launch_bounded_wait_probe(uint32_t *status, uint64_t limit_ns, cudaStream_t stream)
{
    bounded_wait_probe_kernel<<<1, 1, 0, stream>>>(status, limit_ns);
    return cudaGetLastError();
}

cudaError_t launch_vocab_reduce(const VocabReduceArgs &a, int dtype, cudaStream_t stream)
{
    const int which = variant_index();
    switch (dtype) {
    case FDLLM_BF16: return launch_kind<FDLLM_BF16>(a, stream, which);
    case FDLLM_FP16: return launch_kind<FDLLM_FP16>(a, stream, which);
    default: return launch_kind<FDLLM_FP32>(a, stream, which);
    }
}

cudaError_t launch_finalize(const FinalizeArgs &a, cudaStream_t stream)
{
    const int threads = 256;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((a.rows + threads - 1) / threads));
    cfg.blockDim = dim3(threads);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, finalize_kernel, a);
}

}  // namespace fdllm

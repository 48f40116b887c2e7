// fdllm_internal.cuh -- what the kernels and the C interface share: argument blocks,
// workspace pieces, launch entry points and the per-row combination of unit results.
#pragma once

#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "fdllm.h"

namespace fdllm {

// ------------------------------------------------------------------ vocab reduction (a1)
// Each row of logits is cut into units_per_row units of unit_vecs 16-byte vectors (the last
// unit may be shorter), with units_per_row = ceil(row_bytes / target).  A unit is reduced by
// one CTA in a fixed order, so a row's result depends only on its bytes and the call's
// shape (B * L, V, dtype), which fixes the plan.  The CTA streams a unit through a ring of
// shared-memory chunk buffers.  The target is 128 KB; a step whose logits, all B * L rows
// counted, fit in about one wave of such units over the SMs (kSmallStepBytes) takes 64 KB
// units instead, so that twice as many SMs share its reduction: there the per-SM exp
// throughput and the first copy's latency, not HBM, set the time.  Smaller units pay for
// themselves nowhere: a unit must fill the ring (192 KB in flight per SM) to stream at
// full bandwidth.
constexpr int kSegQueue = 8;  // unit results queued from math warps to the epilogue warp
constexpr int64_t kUnitTargetBytes = 131072;
constexpr int64_t kSmallUnitTargetBytes = 65536;
constexpr int64_t kSmallStepBytes = 20ll << 20;
constexpr int kMaxGrid = 1024;
constexpr int kMaxRows = 65536;
constexpr int kMaskWords = kMaxRows / 32;

constexpr float kLog2e = 1.4426950408889634f;
constexpr uint32_t kNoIdx = 0xFFFFFFFFu;

// Reduction of one unit (or one vocabulary tile or slab of the LM head): max logit M,
// S = sum of exp(x - M) over it, relative to M exactly (see rebase_scaled), and the
// row-relative index of the first logit equal to M.
struct UnitPartial {
    float M;
    float S;
    uint32_t idx;
    uint32_t pad;
};

struct VocabReduceArgs {
    const uint8_t *logits;   // [rows, V] element size esize
    const uint8_t *mask;     // [rows]
    int64_t rows;            // B * L
    int64_t row_bytes;       // V * esize
    int64_t vec_per_row;     // row_bytes / 16
    int32_t units_per_row;
    int32_t unit_vecs;
    UnitPartial *partials;   // [rows][units_per_row]; written for masked rows
    uint32_t *next_unit;     // work queue past the first gridDim.x units: zero on entry,
                             // zero again after the launch's last fetch
    uint32_t *status;        // sticky device error bits
    bool pdl = true;         // launch as a programmatic dependent of the previous kernel
};

struct UnitPlan {
    int32_t units_per_row;
    int32_t unit_vecs;
};

// Unit lengths are rounded up to a multiple of kUnitAlignVecs vectors (8 KB), so that every
// unit but a row's last one fills whole chunks; the unit count is then recomputed so that
// no unit is empty.
constexpr int64_t kUnitAlignVecs = 512;

inline UnitPlan plan_units(int64_t row_bytes, int64_t rows)
{
    const int64_t vpr = row_bytes / 16;
    const int64_t target =
        rows * row_bytes <= kSmallStepBytes ? kSmallUnitTargetBytes : kUnitTargetBytes;
    int64_t upr = (row_bytes + target - 1) / target;
    if (upr < 1)
        upr = 1;
    int64_t uv = (vpr + upr - 1) / upr;
    uv = (uv + kUnitAlignVecs - 1) / kUnitAlignVecs * kUnitAlignVecs;
    upr = (vpr + uv - 1) / uv;
    if (upr < 1)
        upr = 1;
    return UnitPlan{(int32_t)upr, (int32_t)uv};
}

// Enqueue the vocab reduction on all SMs, as a programmatic dependent of the previous
// kernel on the stream.
cudaError_t launch_vocab_reduce(const VocabReduceArgs &a, int dtype, cudaStream_t stream);

// One thread waits, bounded by limit_ns, on an mbarrier that never completes.
cudaError_t launch_bounded_wait_probe(uint32_t *status, uint64_t limit_ns, cudaStream_t stream);

// Per masked position: combine its unit partials, write (c, x_hat); resets next_unit.
// Launched as a programmatic dependent of the vocab reduction.
struct FinalizeArgs {
    const uint8_t *mask;
    int64_t rows;
    int32_t units_per_row;
    const UnitPartial *partials;
    float *out_conf;
    int32_t *out_tok;
    uint32_t *next_unit;
};

cudaError_t launch_finalize(const FinalizeArgs &a, cudaStream_t stream);

// ------------------------------------------------------------------ profile select (a2-a5)
// The profile rule on calibration-robust lower confidences max{0, c - eta} (App. C).
constexpr int kModeRobust = 3;

struct ProfileSelectArgs {
    // Source of (c, x_hat): unit partials (from the vocab reduction, which this kernel then
    // follows as a programmatic dependent launch) when `partials` is non-null, otherwise the
    // given conf/tok arrays.
    int32_t units_per_row;
    const UnitPartial *partials;
    uint32_t *next_unit;     // reset to zero when partials are consumed
    const float *conf;       // [B, L]
    const int32_t *tok;      // [B, L]
    uint8_t *mask;           // [B, L], updated in place
    int B;
    int L;
    int mode;                // 0 profile, 1 factor, 2 threshold, kModeRobust
    double param;
    double eta;              // kModeRobust: uniform calibration allowance
    const float *eta_pos;    // kModeRobust: [B, L] per-position allowances, or null
    int32_t *out_tokens;     // [B, L]
    uint8_t *out_commit;     // [B, L]
    int32_t *out_n;          // [B]
    uint32_t *status;        // nullable: the timeout bit set -> every row reports a device
                             // error; a non-finite row sets the non-finite bit
    bool pdl = true;         // with partials: launch as a programmatic dependent
};

cudaError_t launch_profile_select(const ProfileSelectArgs &a, cudaStream_t stream);

// fdllm_lmhead_select on the library-owned workspace, with programmatic dependent launches
// switched on or off (as select_owned).
fdllm_status lmhead_select_owned(const void *hidden, const void *w_vocab, int B, int L, int H,
                                 int V, uint8_t *mask, double param, int mode,
                                 int32_t *out_tokens, uint8_t *out_commit, int32_t *out_n,
                                 cudaStream_t stream, bool pdl);

// The library-owned workspace of the current device, grown on demand and zero-filled when
// allocated.  Every user shares its 256-byte header: the sticky status word at offset 0 and
// the vocab reduction's work counter at 4 (zero between calls); the LM-head path keeps its
// compact row count at 8.
fdllm_status owned_workspace(size_t need, cudaStream_t stream, void **out);

// fdllm_select's argument checks (shape, pointers, mode, param, logits alignment and the
// unit plan's index range), done before anything is enqueued.
fdllm_status check_select_args(const void *logits, int dtype, int B, int L, int V,
                               const uint8_t *mask, double param, int mode,
                               const int32_t *out_tokens, const uint8_t *out_commit,
                               const int32_t *out_n);

// Frees fdllm_select_host's device staging buffer of device `dev` (the caller synchronises).
void release_host_staging(int dev);

// fdllm_select on the library-owned workspace, with programmatic dependent launches
// switched on or off (the decode loop's graph body falls back to plain stream order where
// the driver does not accept programmatic edges inside a conditional node).
fdllm_status select_owned(const void *logits, int dtype, int B, int L, int V, uint8_t *mask,
                          double param, int mode, int32_t *out_tokens, uint8_t *out_commit,
                          int32_t *out_n, cudaStream_t stream, bool pdl);

struct ProfileTermsArgs {
    const float *conf;       // [B, L]
    const uint8_t *mask;     // [B, L]
    int B;
    int L;
    double *out_G;           // [B, L] by rank, nullable
    double *out_F;           // [B, L] by rank, nullable
    double *out_B;           // [B, L] by rank, nullable
    double delta;            // the profile rule's margin, for out_feff
    double *out_feff;        // [B, L] by rank: 1 - delta + B_n, nullable
    int32_t *out_order;      // [B, L] position at each rank, nullable
};

cudaError_t launch_profile_terms(const ProfileTermsArgs &a, cudaStream_t stream);

// ------------------------------------------------------------------ device helpers
#ifdef __CUDACC__
__device__ __forceinline__ float ex2_mufu(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Every partial (M, S) holds S = sum exp(x - M) relative to its own maximum M exactly.
//
// Sums are accumulated as 2^(x * s - r2) with a scale s and an fp32 reference r2.
//  * |ref| < kBigRef: s = log2e, r2 = round(ref * log2e).  The FMA forms x * log2e exactly;
//    the rounding residual r = ref * log2e - r2 is at most half an ulp of a value below 2^31,
//    so |r| <= 64, and it scales every term by the same 2^r, which rebase_scaled removes.
//  * |ref| >= kBigRef: s = 1, r2 = ref.  Distinct fp32 values there are at least 64 apart, so
//    every term but those equal to ref is below 2^-64 of them (under e^-64 in exp as well):
//    the sum counts the maxima, and the terms it drops weigh under 2^-40 for V < 2^24.
constexpr float kBigRef = 0x1p30f;

// S accumulated against (s, r2) -> relative to M: S * 2^(r2 - M s).  M s - r2 is formed in
// one FMA from the exact product, so the rounding of r2 cancels instead of scaling S.
__device__ __forceinline__ float rebase_scaled(float S, float s, float r2, float M)
{
    return S != 0.0f ? S * ex2_mufu(-fmaf(M, s, -r2)) : 0.0f;  // keeps NaN, avoids 0 * inf
}

// S relative to the maximum a -> relative to b >= a: S * exp(a - b).  a - b is exact when the
// two are within a factor of two and carries a relative 2^-24 otherwise, where the factor is
// below exp(-|b| / 2).  Infinite or NaN maxima give NaN, reported by the caller.
__device__ __forceinline__ float rebase(float S, float a, float b)
{
    return S != 0.0f ? S * ex2_mufu((a - b) * kLog2e) : 0.0f;
}

// Position result from its units, folded in unit order (a fixed order, so identical rows
// give identical bits): c = min(1/S, 1) (the max term alone is 1) and x_hat = the first
// index attaining the max; c = NaN, x_hat = -1 when the row holds a NaN or its maximum is
// +inf or -inf.
__device__ __forceinline__ void combine_position(const UnitPartial *p, int upr, float &c,
                                                 int32_t &tok)
{
    float Mj[8], Sj[8];
    uint32_t Ij[8];
    float M = -__int_as_float(0x7F800000);
    float S = 0.0f;
    uint32_t idx = kNoIdx;
    for (int j0 = 0; j0 < upr; j0 += 8) {
        const int cnt = upr - j0 < 8 ? upr - j0 : 8;
#pragma unroll
        for (int j = 0; j < 8; ++j)
            if (j < cnt) {
                const int4 r = __ldcg(reinterpret_cast<const int4 *>(p + j0 + j));
                Mj[j] = __int_as_float(r.x);
                Sj[j] = __int_as_float(r.y);
                Ij[j] = (uint32_t)r.z;
            }
        float Mb = M;
#pragma unroll
        for (int j = 0; j < 8; ++j)
            if (j < cnt)
                Mb = fmaxf(Mb, Mj[j]);
        float Sb = rebase(S, M, Mb);
        uint32_t ib = (M == Mb) ? idx : kNoIdx;
#pragma unroll
        for (int j = 0; j < 8; ++j)
            if (j < cnt) {
                Sb += rebase(Sj[j], Mj[j], Mb);
                if (Mj[j] == Mb && ib == kNoIdx)
                    ib = Ij[j];
            }
        M = Mb;
        S = Sb;
        idx = ib;
    }
    c = __int_as_float(0x7FC00000);
    tok = -1;
    const bool finite = fabsf(M) <= 3.402823466e38f && fabsf(S) <= 3.402823466e38f;
    if (!finite || !(S > 0.0f) || idx == kNoIdx)
        return;
    tok = (int32_t)idx;
    c = fminf(1.0f / S, 1.0f);
}

// Programmatic dependent launch: the dependent grid's wait for the primary grid's results,
// and the primary's permission for the dependent grid to start launching.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents()
{
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
#endif

}  // namespace fdllm

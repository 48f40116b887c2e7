// profile_select.cu -- steps a2-a5 of the selection for one batch row per CTA (paper
// Algorithm 1: sort, scan, select, reveal):
//   a2  sort the masked (c, position) pairs by c descending, position ascending: one 64-bit
//       key per thread; rows of at most 32 positions (one warp) by rank counting (each key's
//       rank is the number of smaller keys, 32 independent shuffles), longer rows by a
//       bitonic network (warp shuffles for partner distance < 32, shared memory above);
//   a3  prefix sums over the sorted order in 64-bit fixed point (units of 2^-52, exact and
//       independent of the summation order; warp shuffles, then across warps):
//       P_n = sum_{j<=n} (1 - c_(j)), so L_n = max{0, 1 - P_n} (= sum c - (n-1), Sec. 3),
//       U_n = 1 - c_(n), G_n = L_n - U_n; factor: (n+1)(1 - c_(n)) < f; threshold: c_(n) >= tau;
//   a4  n* = max{n : rule accepts n} (a block max, the literal definition), 1 if none;
//   a5  reveal the first n* sorted positions: token, commit flag, mask cleared.
// The row has L <= 1024 positions, so this is latency-bound work on a few KB: the kernel's
// time after its launch wait is the selection's share of a decode step.  No fp64
// arithmetic: GB300's fp64 pipe is slow enough (on the order of a hundred cycles per
// dependent operation) that an fp64 scan and rule cost more than the sort.
#include <cmath>
#include <cstdint>

#include "fdllm_internal.cuh"
#include "ptx.cuh"

namespace fdllm {
namespace {

constexpr uint64_t kPadKey = ~0ull;  // sorts after every real key

// Fixed point of the scan: 1 - c in units of 2^-52.  c is an fp32 value in [0, 1], so
// c * 2^52 is exact in fp32 and an integer for every c >= 2^-29; smaller c round to the
// nearest unit (an absolute error of at most 2^-53 per term).  A prefix of up to 1024 terms
// stays below 2^63, and integer addition makes the sums exact and order-independent.
constexpr int64_t kFixOne = (int64_t)1 << 52;

__device__ __forceinline__ int64_t one_minus_fixed(float c)
{
    return kFixOne - __float2ll_rn(c * 0x1p52f);
}

// Masked: (bits(1) - bits(c)) << 32 | pos — for c in [0, 1] larger c gives a smaller key
// (0 for c = 1, bits(1) for c = 0), and equal c falls back to the position.  Unmasked:
// 0xFFFFFFFF << 32 | pos, after every masked key.
constexpr uint32_t kOneBits = 0x3F800000u;

__device__ __forceinline__ uint64_t make_key(bool masked, float c, int pos)
{
    const uint32_t hi = masked ? kOneBits - __float_as_uint(c) : 0xFFFFFFFFu;
    return ((uint64_t)hi << 32) | (uint32_t)pos;
}

__device__ __forceinline__ float key_conf(uint64_t key)
{
    return __uint_as_float(kOneBits - (uint32_t)(key >> 32));
}

template <int T>
__device__ __forceinline__ uint64_t bitonic_sort(uint64_t key, uint64_t *sk)
{
    const int t = threadIdx.x;
#pragma unroll 1
    for (int k = 2; k <= T; k <<= 1) {
#pragma unroll 1
        for (int j = k >> 1; j > 0; j >>= 1) {
            uint64_t other;
            if (j >= 32) {
                sk[t] = key;
                __syncthreads();
                other = sk[t ^ j];
                __syncthreads();
            } else {
                other = __shfl_xor_sync(0xFFFFFFFFu, key, j);
            }
            const bool ascending = (t & k) == 0;
            const bool lower = (t & j) == 0;
            const uint64_t lo = key < other ? key : other;
            const uint64_t hi = key < other ? other : key;
            key = (lower == ascending) ? lo : hi;
        }
    }
    return key;
}

template <int T, typename V>
__device__ __forceinline__ V block_inclusive_scan(V v, V *warp_tot)
{
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const V u = __shfl_up_sync(0xFFFFFFFFu, v, o);
        if (lane >= o)
            v += u;
    }
    if constexpr (T > 32) {
        if (lane == 31)
            warp_tot[w] = v;
        __syncthreads();
        if (w == 0) {
            V x = lane < T / 32 ? warp_tot[lane] : V(0);
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const V u = __shfl_up_sync(0xFFFFFFFFu, x, o);
                if (lane >= o)
                    x += u;
            }
            if (lane < T / 32)
                warp_tot[lane] = x;  // inclusive over warps
        }
        __syncthreads();
        if (w > 0)
            v += warp_tot[w - 1];
    }
    return v;
}

// The rule's acceptance of prefix size n, from c_(n) (fp32), v = 1 - c_(n) and the prefix
// P_n = sum_{j<=n} (1 - c_(j)) in fixed point.  `bound`: for the profile (and robust) rule
// delta = 1 - f in fixed point, for the factor rule f; `tau_f`: the smallest fp32 value
// >= tau, so that c >= tau_f in fp32 decides c >= tau exactly.
__device__ __forceinline__ bool rule_accepts(int mode, int n, float cn, int64_t v, int64_t P,
                                             int64_t bound, float tau_f)
{
    if (mode == 0 || mode == kModeRobust) {  // profile: G_n = L_n - U_n > delta
        const int64_t Ln = kFixOne - P > 0 ? kFixOne - P : 0;
        return Ln - v > bound;
    }
    if (mode == 1)  // factor: (n+1)(1 - c_(n)) < f
        return (int64_t)(n + 1) * v < bound;
    return cn >= tau_f;  // threshold: c_(n) >= tau
}

template <int T>
__device__ __forceinline__ int block_max(int v, int *warp_red)
{
    v = __reduce_max_sync(0xFFFFFFFFu, v);
    if constexpr (T > 32) {
        const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
        __syncthreads();  // warp_red may still be read from an earlier use
        if (lane == 0)
            warp_red[w] = v;
        __syncthreads();
        int x = lane < T / 32 ? warp_red[lane] : 0;
        v = __reduce_max_sync(0xFFFFFFFFu, x);
    }
    return v;
}

template <int T>
__global__ void __launch_bounds__(T) profile_select_kernel(const ProfileSelectArgs a,
                                                            int64_t bound, float tau_f)
{
    __shared__ uint64_t sk[T > 32 ? T : 1];
    __shared__ int32_t s_tok[T];
    __shared__ int64_t warp_tot[32];
    __shared__ int warp_red[32];

    const int t = threadIdx.x;
    const int L = a.L;
    const int64_t base = (int64_t)blockIdx.x * L;

    // (c, x_hat) of this thread's position: folded from the vocab reduction's unit
    // partials, or read from the given arrays.  Launched as a programmatic dependent: the
    // producer of the partials or confidences has completed past the launch wait.  As in the
    // warp kernel, after the vocab reduction the mask byte and the allowance are loaded
    // before that wait (their writers completed before the reduction passed its own wait,
    // and the reduction writes neither); the partials or confidences and the status word
    // after it, all issued before any is used.
    const bool in_row = t < L;
    const bool early = a.partials != nullptr;
    uint8_t mask_byte = 0;
    float eta = (float)a.eta;
    auto load_row_inputs = [&]() {
        mask_byte = in_row ? __ldcg(a.mask + base + t) : (uint8_t)0;
        if (a.mode == kModeRobust && a.eta_pos != nullptr && in_row)
            eta = fmaxf(__ldcg(a.eta_pos + base + t), 0.0f);  // negative or NaN: 0
    };
    if (threadIdx.x == 0)
        pdl_launch_dependents();  // a following vocab reduction may start its prologue
    if (early)
        load_row_inputs();
    pdl_wait();
    if (!early)
        load_row_inputs();
    const bool dev_err = a.status != nullptr && (__ldcg(a.status) & kDevStatTimeout) != 0;
    const bool masked = mask_byte != 0;
    float c = 0.0f;
    int32_t tok = -1;
    if (in_row) {
        if (a.partials != nullptr) {
            combine_position(a.partials + (base + t) * a.units_per_row, a.units_per_row, c,
                             tok);
        } else {
            c = __ldcg(a.conf + base + t);
            tok = __ldcg(a.tok + base + t);
        }
    }
    if (!masked) {
        c = 0.0f;
        tok = -1;
    }
    s_tok[t] = tok;
    if (a.partials != nullptr && a.next_unit != nullptr && blockIdx.x == 0 && t == 0)
        *a.next_unit = 0;  // the vocab reduction before this kernel has finished
    const bool bad = masked && !(c > 0.0f && c <= 1.0f);  // NaN fails both
    // The robust rule ranks and scans lower confidences max{0, c - eta} (App. C).
    float c_rank = c;
    if (a.mode == kModeRobust && masked && !bad)
        c_rank = fmaxf(0.0f, c - eta);
    uint64_t key = t < L ? make_key(masked, c_rank, t) : kPadKey;

    const int m = __syncthreads_count(masked);
    const int any_bad = __syncthreads_or(bad);

    key = bitonic_sort<T>(key, sk);

    // Thread t now holds the (t+1)-th most confident masked position when t < m.
    const int n = t + 1;
    const bool live = t < m;
    const float cn = live ? key_conf(key) : 1.0f;
    const int64_t v = live ? one_minus_fixed(cn) : 0;
    const int64_t P = block_inclusive_scan<T>(v, warp_tot);
    const bool ok = live && rule_accepts(a.mode, n, cn, v, P, bound, tau_f);
    int nstar = block_max<T>(ok ? n : 0, warp_red);
    if (m > 0 && nstar == 0)
        nstar = 1;  // progress convention
    if (any_bad) {
        nstar = -1;
        if (t == 0 && a.status != nullptr)
            atomicOr(a.status, kDevStatNonfinite);
    }
    if (dev_err)
        nstar = -2;

    if (t < L) {
        const int pos = (int)(key & 0xFFFFFFFFu);
        const bool commit = t < nstar;  // nstar <= m, so only masked keys qualify
        a.out_commit[base + pos] = commit ? 1 : 0;
        if (commit) {
            a.out_tokens[base + pos] = s_tok[pos];
            a.mask[base + pos] = 0;
        }
    }
    if (t == 0)
        a.out_n[blockIdx.x] = nstar;
}

// The same steps for rows of at most 32 positions, one warp per row: no block barriers, the
// sort by rank counting (the keys are distinct: the position is in their low bits, pads
// included), the scan by warp shuffles alone.
__global__ void __launch_bounds__(32) profile_select_warp_kernel(const ProfileSelectArgs a,
                                                                  int64_t bound, float tau_f)
{
    __shared__ uint64_t sk[32];
    __shared__ int32_t s_tok[32];
    constexpr unsigned kFull = 0xFFFFFFFFu;
    const int t = threadIdx.x;
    const int L = a.L;
    const int64_t base = (int64_t)blockIdx.x * L;

    // After the vocab reduction (partials given), the mask byte and the allowance are loaded
    // before the launch wait: this kernel starts only once the reduction has passed its own
    // launch wait, so whatever wrote them has completed, and the reduction writes neither.
    // The unit partials and the status word are the reduction's output: loaded after it.
    // Otherwise (confidences given) everything is loaded after the wait.
    const bool in_row = t < L;
    const bool early = a.partials != nullptr;
    uint8_t mask_byte = 0;
    float eta = (float)a.eta;
    auto load_row_inputs = [&]() {
        mask_byte = in_row ? __ldcg(a.mask + base + t) : (uint8_t)0;
        if (a.mode == kModeRobust && a.eta_pos != nullptr && in_row)
            eta = fmaxf(__ldcg(a.eta_pos + base + t), 0.0f);  // negative or NaN: 0
    };
    if (t == 0)
        pdl_launch_dependents();  // a following vocab reduction may start its prologue
    if (early)
        load_row_inputs();
    pdl_wait();  // the producer of the partials or confidences has completed
    if (!early)
        load_row_inputs();
    // The rest of the row's loads are issued here, before any of them is used (one memory
    // round trip): status word and the position's unit partials or (c, x_hat).
    const uint32_t status = a.status != nullptr ? __ldcg(a.status) : 0u;
    const bool masked = mask_byte != 0;
    float c = 0.0f;
    int32_t tok = -1;
    if (in_row) {
        if (a.partials != nullptr) {
            combine_position(a.partials + (base + t) * a.units_per_row, a.units_per_row, c,
                             tok);
        } else {
            c = __ldcg(a.conf + base + t);
            tok = __ldcg(a.tok + base + t);
        }
    }
    if (!masked) {
        c = 0.0f;
        tok = -1;
    }
    s_tok[t] = tok;
    if (a.partials != nullptr && a.next_unit != nullptr && blockIdx.x == 0 && t == 0)
        *a.next_unit = 0;  // the vocab reduction before this kernel has finished
    const bool bad = masked && !(c > 0.0f && c <= 1.0f);  // NaN fails both
    float c_rank = c;
    if (a.mode == kModeRobust && masked && !bad)
        c_rank = fmaxf(0.0f, c - eta);  // App. C: lower confidences max{0, c - eta}
    uint64_t key = make_key(masked, c_rank, t);
    const int m = __popc(__ballot_sync(kFull, masked));
    const bool any_bad = __any_sync(kFull, bad);

    int rank = 0;
#pragma unroll
    for (int j = 0; j < 32; ++j)
        rank += __shfl_sync(kFull, key, j) < key ? 1 : 0;
    sk[rank] = key;
    __syncwarp();
    key = sk[t];

    // Lane t now holds the (t+1)-th most confident masked position when t < m.
    const int n = t + 1;
    const bool live = t < m;
    const float cn = live ? key_conf(key) : 1.0f;
    const int64_t v = live ? one_minus_fixed(cn) : 0;
    int64_t P = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int64_t u = __shfl_up_sync(kFull, P, o);
        if (t >= o)
            P += u;
    }
    const bool ok = live && rule_accepts(a.mode, n, cn, v, P, bound, tau_f);
    int nstar = __reduce_max_sync(kFull, ok ? n : 0);
    if (m > 0 && nstar == 0)
        nstar = 1;  // progress convention
    if (any_bad) {
        nstar = -1;
        if (t == 0 && a.status != nullptr)
            atomicOr(a.status, kDevStatNonfinite);
    }
    if ((status & kDevStatTimeout) != 0)
        nstar = -2;

    if (t < L) {
        const int pos = (int)(key & 0xFFFFFFFFu);  // < L: the L row keys precede the pads
        const bool commit = t < nstar;
        a.out_commit[base + pos] = commit ? 1 : 0;
        if (commit) {
            a.out_tokens[base + pos] = s_tok[pos];
            a.mask[base + pos] = 0;
        }
    }
    if (t == 0)
        a.out_n[blockIdx.x] = nstar;
}

// Heterogeneity-bonus diagnostics of one batch row per CTA (Prop. heterogeneity-bonus,
// Eq. heterogeneity_decomp): the masked confidences sorted as in the selection, an fp64
// inclusive scan S_n = sum_{j<=n} c_(j), and at rank n: G_n = max{0, S_n - (n-1)} - (1 - c_(n)),
// F_n = (n+1) c_(n) - n and B_n = S_n - n c_(n) (= sum_{j<n} (c_(j) - c_(n))); and the
// effective factor f_eff(n) = 1 - delta + B_n of Remark adaptive-factor.
template <int T>
__global__ void __launch_bounds__(T) profile_terms_kernel(const ProfileTermsArgs a)
{
    __shared__ uint64_t sk[T > 32 ? T : 1];
    __shared__ double warp_tot[32];
    const int t = threadIdx.x;
    const int L = a.L;
    const int64_t base = (int64_t)blockIdx.x * L;
    const bool masked = t < L && a.mask[base + t] != 0;
    const float c = masked ? a.conf[base + t] : 0.0f;
    uint64_t key = t < L ? make_key(masked, c, t) : kPadKey;
    const int m = __syncthreads_count(masked);
    key = bitonic_sort<T>(key, sk);
    const bool live = t < m;
    const double cn = live ? (double)key_conf(key) : 0.0;
    const double S = block_inclusive_scan<T>(cn, warp_tot);
    if (t >= L)
        return;
    const double n = (double)(t + 1);
    const double nan = __longlong_as_double(0x7FF8000000000000ll);
    if (a.out_G != nullptr)
        a.out_G[base + t] = live ? fmax(0.0, S - (n - 1.0)) - (1.0 - cn) : nan;
    if (a.out_F != nullptr)
        a.out_F[base + t] = live ? (n + 1.0) * cn - n : nan;
    if (a.out_B != nullptr)
        a.out_B[base + t] = live ? S - n * cn : nan;
    if (a.out_feff != nullptr)
        a.out_feff[base + t] = live ? 1.0 - a.delta + (S - n * cn) : nan;
    if (a.out_order != nullptr)
        a.out_order[base + t] = live ? (int32_t)(key & 0xFFFFFFFFu) : -1;
}

template <int T>
cudaError_t launch_terms_t(const ProfileTermsArgs &a, cudaStream_t stream)
{
    profile_terms_kernel<T><<<a.B, T, 0, stream>>>(a);
    return cudaGetLastError();
}

template <typename Kernel>
cudaError_t launch_select(Kernel kern, int threads, const ProfileSelectArgs &a,
                          int64_t bound, float tau_f, cudaStream_t stream)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)a.B);
    cfg.blockDim = dim3(threads);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = a.pdl ? 1 : 0;  // a programmatic dependent of the previous kernel
    return cudaLaunchKernelEx(&cfg, kern, a, bound, tau_f);
}

}  // namespace

cudaError_t launch_profile_select(const ProfileSelectArgs &a, cudaStream_t stream)
{
    // The rule's parameter in the kernels' arithmetic.  f in fixed point (clamped to
    // [-1500, 1500]: beyond, (n+1)(1 - c) <= 1025 decides every n the same way), and the
    // profile margin delta = 1 - f from the same integer, so that delta + f = 1 exactly and
    // the equal-confidence reduction to the factor rule holds bit for bit.
    const double f = a.param < -1500.0 ? -1500.0 : (a.param > 1500.0 ? 1500.0 : a.param);
    const int64_t f_fix = std::llround(f * 0x1p52);
    const int64_t bound = a.mode == 1 ? f_fix : kFixOne - f_fix;
    float tau_f = (float)a.param;  // the smallest fp32 value >= tau
    if ((double)tau_f < a.param)
        tau_f = std::nextafter(tau_f, INFINITY);
    if (a.L <= 32)
        return launch_select(profile_select_warp_kernel, 32, a, bound, tau_f, stream);
    if (a.L <= 64)
        return launch_select(profile_select_kernel<64>, 64, a, bound, tau_f, stream);
    if (a.L <= 128)
        return launch_select(profile_select_kernel<128>, 128, a, bound, tau_f, stream);
    if (a.L <= 256)
        return launch_select(profile_select_kernel<256>, 256, a, bound, tau_f, stream);
    if (a.L <= 512)
        return launch_select(profile_select_kernel<512>, 512, a, bound, tau_f, stream);
    return launch_select(profile_select_kernel<1024>, 1024, a, bound, tau_f, stream);
}

cudaError_t launch_profile_terms(const ProfileTermsArgs &a, cudaStream_t stream)
{
    if (a.L <= 32)
        return launch_terms_t<32>(a, stream);
    if (a.L <= 64)
        return launch_terms_t<64>(a, stream);
    if (a.L <= 128)
        return launch_terms_t<128>(a, stream);
    if (a.L <= 256)
        return launch_terms_t<256>(a, stream);
    if (a.L <= 512)
        return launch_terms_t<512>(a, stream);
    return launch_terms_t<1024>(a, stream);
}

}  // namespace fdllm

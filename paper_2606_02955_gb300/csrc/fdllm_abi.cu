// fdllm_abi.cu -- the C interface declared in include/fdllm.h: argument checks on the host,
// the workspace (library-owned per device, or caller-provided) and the kernel launches.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <mutex>

#include "fdllm.h"
#include "fdllm_internal.cuh"
#include "ptx.cuh"

namespace fdllm {
namespace {

constexpr size_t kAlign = 256;

size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Workspace layout (offsets from a kAlign-aligned base).  The header block sits at a fixed
// offset, so a workspace can be reused across shapes:
//   header   status (uint32, sticky device error bits) at 0, next_unit (uint32, the vocab
//            reduction's work counter, zero between calls) at 4
//   partials UnitPartial [rows][units_per_row]
struct Layout {
    size_t status, next_unit, partials, total;
    UnitPlan plan;
};

Layout layout_for(int64_t rows, int64_t row_bytes)
{
    Layout l;
    l.plan = plan_units(row_bytes, rows);
    l.status = 0;
    l.next_unit = 4;
    l.partials = kAlign;
    l.total = align_up(l.partials + (size_t)rows * l.plan.units_per_row * sizeof(UnitPartial));
    return l;
}

bool valid_dtype(int d) { return d == FDLLM_BF16 || d == FDLLM_FP32 || d == FDLLM_FP16; }
bool valid_mode(int m) { return m == FDLLM_PROFILE || m == FDLLM_FACTOR || m == FDLLM_THRESHOLD; }
int esize_of(int d) { return d == FDLLM_FP32 ? 4 : 2; }

fdllm_status check_shape(int B, int L, int V)
{
    if (B < 1 || L < 1 || L > FDLLM_MAX_L || V < 1)
        return FDLLM_ERR_ARG;
    if ((int64_t)B * L > FDLLM_MAX_ROWS)
        return FDLLM_ERR_ARG;
    return FDLLM_OK;
}

// Unit partial slots are indexed with 32 bits.
bool plan_fits(int64_t rows, int64_t row_bytes)
{
    return rows * (int64_t)plan_units(row_bytes, rows).units_per_row < ((int64_t)1 << 31);
}

fdllm_status check_logits(const void *logits, int dtype, int V)
{
    if (!logits || !valid_dtype(dtype))
        return FDLLM_ERR_ARG;
    if ((reinterpret_cast<uintptr_t>(logits) & 15u) != 0)
        return FDLLM_ERR_ALIGN;
    if (((int64_t)V * esize_of(dtype)) % 16 != 0)
        return FDLLM_ERR_ALIGN;
    return FDLLM_OK;
}

// Library-owned workspace, one per device, grown on demand and zero-filled when allocated.
struct OwnedWorkspace {
    void *ptr = nullptr;
    size_t bytes = 0;
};
constexpr int kMaxDevices = 64;
OwnedWorkspace g_ws[kMaxDevices];
std::mutex g_ws_mutex;

}  // namespace

fdllm_status owned_workspace(size_t need, cudaStream_t stream, void **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return FDLLM_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_ws_mutex);
    OwnedWorkspace &w = g_ws[dev];
    if (w.bytes < need) {
        if (w.ptr) {
            if (cudaDeviceSynchronize() != cudaSuccess)
                return FDLLM_ERR_CUDA;
            cudaFree(w.ptr);
            w.ptr = nullptr;
            w.bytes = 0;
        }
        void *p = nullptr;
        if (cudaMalloc(&p, need) != cudaSuccess)
            return FDLLM_ERR_CUDA;
        if (cudaMemsetAsync(p, 0, need, stream) != cudaSuccess) {
            cudaFree(p);
            return FDLLM_ERR_CUDA;
        }
        w.ptr = p;
        w.bytes = need;
    }
    *out = w.ptr;
    return FDLLM_OK;
}

namespace {

VocabReduceArgs reduce_args(const void *logits, int dtype, int B, int L, int V,
                            const uint8_t *mask, uint8_t *ws, const Layout &lay)
{
    VocabReduceArgs a;
    a.logits = static_cast<const uint8_t *>(logits);
    a.mask = mask;
    a.rows = (int64_t)B * L;
    a.row_bytes = (int64_t)V * esize_of(dtype);
    a.vec_per_row = a.row_bytes / 16;
    a.units_per_row = lay.plan.units_per_row;
    a.unit_vecs = lay.plan.unit_vecs;
    a.partials = reinterpret_cast<UnitPartial *>(ws + lay.partials);
    a.next_unit = reinterpret_cast<uint32_t *>(ws + lay.next_unit);
    a.status = reinterpret_cast<uint32_t *>(ws + lay.status);
    return a;
}

fdllm_status run_select(const void *logits, int dtype, int B, int L, int V, uint8_t *mask,
                        double param, int mode, int32_t *out_tokens, uint8_t *out_commit,
                        int32_t *out_n, uint8_t *ws, const Layout &lay, cudaStream_t stream,
                        double eta = 0.0, const float *eta_pos = nullptr, bool pdl = true)
{
    VocabReduceArgs ra = reduce_args(logits, dtype, B, L, V, mask, ws, lay);
    ra.pdl = pdl;
    if (launch_vocab_reduce(ra, dtype, stream) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    ProfileSelectArgs pa;
    pa.units_per_row = ra.units_per_row;
    pa.partials = ra.partials;
    pa.next_unit = ra.next_unit;
    pa.conf = nullptr;
    pa.tok = nullptr;
    pa.mask = mask;
    pa.B = B;
    pa.L = L;
    pa.mode = mode;
    pa.param = param;
    pa.eta = eta;
    pa.eta_pos = eta_pos;
    pa.out_tokens = out_tokens;
    pa.out_commit = out_commit;
    pa.out_n = out_n;
    pa.status = ra.status;
    pa.pdl = pdl;
    if (launch_profile_select(pa, stream) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    return FDLLM_OK;
}

}  // namespace

fdllm_status check_select_args(const void *logits, int dtype, int B, int L, int V,
                               const uint8_t *mask, double param, int mode,
                               const int32_t *out_tokens, const uint8_t *out_commit,
                               const int32_t *out_n)
{
    fdllm_status st = check_shape(B, L, V);
    if (st != FDLLM_OK)
        return st;
    if (!mask || !out_tokens || !out_commit || !out_n || !valid_mode(mode) ||
        !std::isfinite(param))
        return FDLLM_ERR_ARG;
    st = check_logits(logits, dtype, V);
    if (st != FDLLM_OK)
        return st;
    return plan_fits((int64_t)B * L, (int64_t)V * esize_of(dtype)) ? FDLLM_OK : FDLLM_ERR_ARG;
}

namespace {

// Reads the sticky status word and, when it is set, zeroes `clear_bytes` from it: for a
// workspace header the status word and the vocab reduction's work counter, which a launch
// that gave up a wait may leave mid-queue (it stops fetching before its last unit).  A
// gave-up wait outranks a non-finite row.
fdllm_status read_and_clear_status(uint32_t *status, cudaStream_t stream,
                                   size_t clear_bytes = sizeof(uint32_t))
{
    uint32_t host = 0;
    if (cudaMemcpyAsync(&host, status, sizeof host, cudaMemcpyDeviceToHost, stream) !=
        cudaSuccess)
        return FDLLM_ERR_CUDA;
    if (cudaStreamSynchronize(stream) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    if (host == 0)
        return FDLLM_OK;
    if (cudaMemsetAsync(status, 0, clear_bytes, stream) != cudaSuccess ||
        cudaStreamSynchronize(stream) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    return (host & kDevStatTimeout) != 0 ? FDLLM_ERR_DEVICE : FDLLM_ERR_NONFINITE;
}

// Status word and work counter at the head of every workspace.
constexpr size_t kHeaderClearBytes = 2 * sizeof(uint32_t);

// Scratch for fdllm_select_static: a fixed array in device memory that every GPU loading
// this library holds until the process exits, so that a selection step needs no
// allocation at call time.  Host code only ever sees a host-side stand-in for the symbol;
// the device address comes from cudaGetSymbolAddress, looked up once per device.
static __device__ __align__(256) uint8_t g_static_scratch[FDLLM_STATIC_SCRATCH_BYTES];

// Status word of fdllm_check_bounded_wait (kept apart from every workspace).
static __device__ uint32_t g_probe_status;

void *g_static_scratch_addr[kMaxDevices] = {nullptr};
std::mutex g_static_mutex;

fdllm_status static_scratch_address(void **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return FDLLM_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_static_mutex);
    if (g_static_scratch_addr[dev] == nullptr) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || p == nullptr)
            return FDLLM_ERR_CUDA;
        g_static_scratch_addr[dev] = p;
    }
    *out = g_static_scratch_addr[dev];
    return FDLLM_OK;
}

}  // namespace

fdllm_status select_owned(const void *logits, int dtype, int B, int L, int V, uint8_t *mask,
                          double param, int mode, int32_t *out_tokens, uint8_t *out_commit,
                          int32_t *out_n, cudaStream_t stream, bool pdl)
{
    fdllm_status st = check_select_args(logits, dtype, B, L, V, mask, param, mode, out_tokens,
                                        out_commit, out_n);
    if (st != FDLLM_OK)
        return st;
    const Layout lay = layout_for((int64_t)B * L, (int64_t)V * esize_of(dtype));
    void *ws = nullptr;
    st = owned_workspace(lay.total, stream, &ws);
    if (st != FDLLM_OK)
        return st;
    return run_select(logits, dtype, B, L, V, mask, param, mode, out_tokens, out_commit, out_n,
                      static_cast<uint8_t *>(ws), lay, stream, 0.0, nullptr, pdl);
}

}  // namespace fdllm

using namespace fdllm;

extern "C" {

size_t fdllm_workspace_bytes(int B, int L, int V, int dtype)
{
    if (B < 1 || L < 1 || V < 1 || !valid_dtype(dtype))
        return 0;
    return layout_for((int64_t)B * L, (int64_t)V * esize_of(dtype)).total;
}

fdllm_status fdllm_select_ws(const void *logits, int dtype, int B, int L, int V, uint8_t *mask,
                             double param, int mode, int32_t *out_tokens, uint8_t *out_commit,
                             int32_t *out_n, void *workspace, size_t workspace_bytes,
                             void *stream)
{
    fdllm_status st = check_select_args(logits, dtype, B, L, V, mask, param, mode, out_tokens,
                                        out_commit, out_n);
    if (st != FDLLM_OK)
        return st;
    const Layout lay = layout_for((int64_t)B * L, (int64_t)V * esize_of(dtype));
    if (!workspace || (reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0 ||
        workspace_bytes < lay.total)
        return FDLLM_ERR_WORKSPACE;
    return run_select(logits, dtype, B, L, V, mask, param, mode, out_tokens, out_commit, out_n,
                      static_cast<uint8_t *>(workspace), lay,
                      static_cast<cudaStream_t>(stream));
}

fdllm_status fdllm_select(const void *logits, int dtype, int B, int L, int V, uint8_t *mask,
                          double param, int mode, int32_t *out_tokens, uint8_t *out_commit,
                          int32_t *out_n, void *stream)
{
    return select_owned(logits, dtype, B, L, V, mask, param, mode, out_tokens, out_commit,
                        out_n, static_cast<cudaStream_t>(stream), true);
}

fdllm_status fdllm_select_robust(const void *logits, int dtype, int B, int L, int V,
                                 uint8_t *mask, double param, double eta,
                                 const float *eta_per_position, int32_t *out_tokens,
                                 uint8_t *out_commit, int32_t *out_n, void *stream)
{
    fdllm_status st = check_select_args(logits, dtype, B, L, V, mask, param, FDLLM_PROFILE,
                                        out_tokens, out_commit, out_n);
    if (st != FDLLM_OK)
        return st;
    if (!std::isfinite(eta) || eta < 0.0)
        return FDLLM_ERR_ARG;
    const Layout lay = layout_for((int64_t)B * L, (int64_t)V * esize_of(dtype));
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    void *ws = nullptr;
    st = owned_workspace(lay.total, s, &ws);
    if (st != FDLLM_OK)
        return st;
    return run_select(logits, dtype, B, L, V, mask, param, kModeRobust, out_tokens, out_commit,
                      out_n, static_cast<uint8_t *>(ws), lay, s, eta, eta_per_position);
}

fdllm_status fdllm_select_static(const void *logits, int dtype, int B, int L, int V,
                                 uint8_t *mask, double param, int mode, int32_t *out_tokens,
                                 uint8_t *out_commit, int32_t *out_n, void *stream)
{
    fdllm_status st = check_select_args(logits, dtype, B, L, V, mask, param, mode, out_tokens,
                                        out_commit, out_n);
    if (st != FDLLM_OK)
        return st;
    const Layout lay = layout_for((int64_t)B * L, (int64_t)V * esize_of(dtype));
    if (lay.total > (size_t)FDLLM_STATIC_SCRATCH_BYTES)
        return FDLLM_ERR_WORKSPACE;  // shape needs more scratch than the fixed array holds
    void *ws = nullptr;
    st = static_scratch_address(&ws);
    if (st != FDLLM_OK)
        return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // The array keeps the previous call's contents: zero the status word and the work
    // counter (the header block) before the kernels read them.
    if (cudaMemsetAsync(ws, 0, kAlign, s) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    return run_select(logits, dtype, B, L, V, mask, param, mode, out_tokens, out_commit, out_n,
                      static_cast<uint8_t *>(ws), lay, s);
}

fdllm_status fdllm_confidence(const void *logits, int dtype, int B, int L, int V,
                              const uint8_t *mask, float *out_conf, int32_t *out_argmax,
                              void *stream)
{
    fdllm_status st = check_shape(B, L, V);
    if (st != FDLLM_OK)
        return st;
    if (!mask || !out_conf || !out_argmax)
        return FDLLM_ERR_ARG;
    st = check_logits(logits, dtype, V);
    if (st != FDLLM_OK)
        return st;
    if (!plan_fits((int64_t)B * L, (int64_t)V * esize_of(dtype)))
        return FDLLM_ERR_ARG;
    const Layout lay = layout_for((int64_t)B * L, (int64_t)V * esize_of(dtype));
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    void *ws = nullptr;
    st = owned_workspace(lay.total, s, &ws);
    if (st != FDLLM_OK)
        return st;
    VocabReduceArgs ra = reduce_args(logits, dtype, B, L, V, mask, static_cast<uint8_t *>(ws),
                                     lay);
    if (launch_vocab_reduce(ra, dtype, s) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    FinalizeArgs fa;
    fa.mask = mask;
    fa.rows = ra.rows;
    fa.units_per_row = ra.units_per_row;
    fa.partials = ra.partials;
    fa.out_conf = out_conf;
    fa.out_tok = out_argmax;
    fa.next_unit = ra.next_unit;
    if (launch_finalize(fa, s) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    return FDLLM_OK;
}

fdllm_status fdllm_vocab_reduce(const void *logits, int dtype, int B, int L, int V,
                                const uint8_t *mask, void *stream)
{
    fdllm_status st = check_shape(B, L, V);
    if (st != FDLLM_OK)
        return st;
    if (!mask)
        return FDLLM_ERR_ARG;
    st = check_logits(logits, dtype, V);
    if (st != FDLLM_OK)
        return st;
    if (!plan_fits((int64_t)B * L, (int64_t)V * esize_of(dtype)))
        return FDLLM_ERR_ARG;
    const Layout lay = layout_for((int64_t)B * L, (int64_t)V * esize_of(dtype));
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    void *ws = nullptr;
    st = owned_workspace(lay.total, s, &ws);
    if (st != FDLLM_OK)
        return st;
    VocabReduceArgs ra = reduce_args(logits, dtype, B, L, V, mask, static_cast<uint8_t *>(ws),
                                     lay);
    // The reduction leaves its work counter at zero itself (its last fetch resets it).
    return launch_vocab_reduce(ra, dtype, s) == cudaSuccess ? FDLLM_OK : FDLLM_ERR_CUDA;
}

fdllm_status fdllm_select_from_conf(const float *conf, const int32_t *argmax, int B, int L,
                                    uint8_t *mask, double param, int mode,
                                    int32_t *out_tokens, uint8_t *out_commit, int32_t *out_n,
                                    void *stream)
{
    if (B < 1 || L < 1 || L > FDLLM_MAX_L || (int64_t)B * L > FDLLM_MAX_ROWS)
        return FDLLM_ERR_ARG;
    if (!conf || !argmax || !mask || !out_tokens || !out_commit || !out_n || !valid_mode(mode) ||
        !std::isfinite(param))
        return FDLLM_ERR_ARG;
    ProfileSelectArgs pa;
    pa.units_per_row = 0;
    pa.partials = nullptr;
    pa.next_unit = nullptr;
    pa.conf = conf;
    pa.tok = argmax;
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
    pa.status = nullptr;
    if (launch_profile_select(pa, static_cast<cudaStream_t>(stream)) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    return FDLLM_OK;
}

fdllm_status fdllm_profile_terms(const float *conf, const uint8_t *mask, int B, int L,
                                 double delta, double *out_G, double *out_F, double *out_B,
                                 double *out_feff, int32_t *out_order, void *stream)
{
    if (B < 1 || L < 1 || L > FDLLM_MAX_L || (int64_t)B * L > FDLLM_MAX_ROWS)
        return FDLLM_ERR_ARG;
    if (!conf || !mask || !std::isfinite(delta))
        return FDLLM_ERR_ARG;
    ProfileTermsArgs a;
    a.conf = conf;
    a.mask = mask;
    a.B = B;
    a.L = L;
    a.out_G = out_G;
    a.out_F = out_F;
    a.out_B = out_B;
    a.delta = delta;
    a.out_feff = out_feff;
    a.out_order = out_order;
    return launch_profile_terms(a, static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? FDLLM_OK
               : FDLLM_ERR_CUDA;
}

fdllm_status fdllm_check_bounded_wait(double seconds, void *stream)
{
    if (!(seconds > 0.0) || seconds > 10.0)
        return FDLLM_ERR_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    uint32_t *status = nullptr;
    if (cudaGetSymbolAddress(reinterpret_cast<void **>(&status), g_probe_status) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    if (cudaMemsetAsync(status, 0, sizeof(uint32_t), s) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    if (launch_bounded_wait_probe(status, (uint64_t)(seconds * 1e9), s) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    return read_and_clear_status(status, s);
}

fdllm_status fdllm_device_status(void *stream)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return FDLLM_ERR_CUDA;
    void *ptr = nullptr;
    {
        std::lock_guard<std::mutex> lock(g_ws_mutex);
        ptr = g_ws[dev].ptr;
    }
    if (!ptr)
        return FDLLM_OK;
    return read_and_clear_status(static_cast<uint32_t *>(ptr), static_cast<cudaStream_t>(stream),
                                 kHeaderClearBytes);
}

fdllm_status fdllm_workspace_status(void *workspace, void *stream)
{
    if (!workspace || (reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0)
        return FDLLM_ERR_WORKSPACE;
    return read_and_clear_status(static_cast<uint32_t *>(workspace),
                                 static_cast<cudaStream_t>(stream), kHeaderClearBytes);
}

fdllm_status fdllm_static_status(void *stream)
{
    void *ws = nullptr;
    fdllm_status st = static_scratch_address(&ws);
    if (st != FDLLM_OK)
        return st;
    return read_and_clear_status(static_cast<uint32_t *>(ws), static_cast<cudaStream_t>(stream),
                                 kHeaderClearBytes);
}

void fdllm_release_workspace(void)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return;
    std::lock_guard<std::mutex> lock(g_ws_mutex);
    if (g_ws[dev].ptr) {
        cudaDeviceSynchronize();
        cudaFree(g_ws[dev].ptr);
        g_ws[dev].ptr = nullptr;
        g_ws[dev].bytes = 0;
    }
    release_host_staging(dev);
}

const char *fdllm_status_string(int status)
{
    switch (status) {
    case FDLLM_OK:
        return "ok";
    case FDLLM_ERR_ARG:
        return "invalid argument (null pointer, size out of range, unknown enum or non-finite param)";
    case FDLLM_ERR_ALIGN:
        return "logits base not 16-byte aligned or V*sizeof(dtype) not a multiple of 16";
    case FDLLM_ERR_NONFINITE:
        return "non-finite logits in a masked row";
    case FDLLM_ERR_CUDA:
        return "CUDA runtime error";
    case FDLLM_ERR_WORKSPACE:
        return "workspace missing, misaligned or too small";
    case FDLLM_ERR_DEVICE:
        return "a kernel gave up a bounded wait";
    default:
        return "unknown status";
    }
}

int fdllm_version(void) { return 100; }

}  // extern "C"

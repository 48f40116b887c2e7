// host_io.cu -- the end-to-end path on host buffers: the rows of masked positions are read
// by the GPU straight from page-locked host memory (over the host link) into a device buffer,
// so that only the logits the selection needs cross the link; fdllm_select_host wraps that,
// the step and the copies of its results back to the host in one call.
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "fdllm.h"
#include "fdllm_internal.cuh"

namespace fdllm {
namespace {

// One CTA per (b, l) row: copies the row's 16-byte vectors when the position is masked.
__global__ void __launch_bounds__(256) gather_masked_rows_kernel(const int4 *src, int4 *dst,
                                                                 const uint8_t *mask,
                                                                 int64_t vec_per_row)
{
    pdl_wait();  // the mask's writer has completed
    if (threadIdx.x == 0)
        pdl_launch_dependents();  // the vocab reduction may start its prologue
    const int64_t row = blockIdx.x;
    if (mask[row] == 0)
        return;
    const int4 *s = src + row * vec_per_row;
    int4 *d = dst + row * vec_per_row;
    int64_t i = threadIdx.x;
    // Four loads in flight per thread: each crosses the host link with its full latency.
    for (; i + 3 * 256 < vec_per_row; i += 4 * 256) {
        const int4 a = s[i], b = s[i + 256], c = s[i + 512], e = s[i + 768];
        d[i] = a;
        d[i + 256] = b;
        d[i + 512] = c;
        d[i + 768] = e;
    }
    for (; i < vec_per_row; i += 256)
        d[i] = s[i];
}

// Where the GPU reads `src`: device memory as it is, page-locked host memory through its
// mapping; nullptr for pageable host memory (or an address CUDA does not know).
const void *device_view(const void *src)
{
    cudaPointerAttributes attr;
    if (cudaPointerGetAttributes(&attr, src) != cudaSuccess) {
        (void)cudaGetLastError();
        return nullptr;
    }
    if (attr.type == cudaMemoryTypeDevice || attr.type == cudaMemoryTypeManaged)
        return src;
    if (attr.type == cudaMemoryTypeHost)
        return attr.devicePointer;
    return nullptr;
}

cudaError_t launch_gather(const void *dsrc, void *dst, const uint8_t *mask, int64_t rows,
                          int64_t row_bytes, cudaStream_t stream)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)rows);
    cfg.blockDim = dim3(256);
    cfg.stream = stream;
    cudaLaunchAttribute a[1];
    a[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    a[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = a;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, gather_masked_rows_kernel, static_cast<const int4 *>(dsrc),
                              static_cast<int4 *>(dst), mask, row_bytes / 16);
}

// fdllm_select_host's device staging, one buffer per device, grown on demand (allocated
// outside the step's kernels, like the library workspace).
struct Staging {
    void *ptr = nullptr;
    size_t bytes = 0;
};
constexpr int kStageDevices = 64;
Staging g_stage[kStageDevices];
std::mutex g_stage_mutex;

size_t up256(size_t x) { return (x + 255) / 256 * 256; }

fdllm_status staging_buffer(size_t need, void **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kStageDevices)
        return FDLLM_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_stage_mutex);
    Staging &s = g_stage[dev];
    if (s.bytes < need) {
        if (s.ptr) {
            if (cudaDeviceSynchronize() != cudaSuccess)
                return FDLLM_ERR_CUDA;
            cudaFree(s.ptr);
            s.ptr = nullptr;
            s.bytes = 0;
        }
        void *p = nullptr;
        if (cudaMalloc(&p, need) != cudaSuccess)
            return FDLLM_ERR_CUDA;
        s.ptr = p;
        s.bytes = need;
    }
    *out = s.ptr;
    return FDLLM_OK;
}

}  // namespace

void release_host_staging(int dev)
{
    if (dev < 0 || dev >= kStageDevices)
        return;
    std::lock_guard<std::mutex> lock(g_stage_mutex);
    if (g_stage[dev].ptr) {
        cudaDeviceSynchronize();
        cudaFree(g_stage[dev].ptr);
        g_stage[dev].ptr = nullptr;
        g_stage[dev].bytes = 0;
    }
}

}  // namespace fdllm

using namespace fdllm;

extern "C" fdllm_status fdllm_gather_masked_rows(const void *src, void *dst, int dtype, int B,
                                                 int L, int V, const uint8_t *mask, void *stream)
{
    if (!src || !dst || !mask || B < 1 || L < 1 || L > FDLLM_MAX_L || V < 1 ||
        (int64_t)B * L > FDLLM_MAX_ROWS ||
        (dtype != FDLLM_BF16 && dtype != FDLLM_FP32 && dtype != FDLLM_FP16))
        return FDLLM_ERR_ARG;
    const int64_t row_bytes = (int64_t)V * (dtype == FDLLM_FP32 ? 4 : 2);
    if (row_bytes % 16 != 0 || (reinterpret_cast<uintptr_t>(src) & 15u) ||
        (reinterpret_cast<uintptr_t>(dst) & 15u))
        return FDLLM_ERR_ALIGN;
    // The device-side address of src: page-locked host memory is read through its mapping.
    const void *dsrc = device_view(src);
    if (!dsrc || (reinterpret_cast<uintptr_t>(dsrc) & 15u))
        return FDLLM_ERR_ARG;  // pageable host memory: not readable by the GPU here
    return launch_gather(dsrc, dst, mask, (int64_t)B * L, row_bytes,
                         static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? FDLLM_OK
               : FDLLM_ERR_CUDA;
}

extern "C" fdllm_status fdllm_select_host(const void *logits, int dtype, int B, int L, int V,
                                          uint8_t *mask, double param, int mode,
                                          int32_t *out_tokens, uint8_t *out_commit,
                                          int32_t *out_n, void *stream)
{
    fdllm_status st = check_select_args(logits, dtype, B, L, V, mask, param, mode, out_tokens,
                                        out_commit, out_n);
    if (st != FDLLM_OK)
        return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int64_t rows = (int64_t)B * L;
    const int64_t row_bytes = (int64_t)V * (dtype == FDLLM_FP32 ? 4 : 2);
    // Logits already in device memory are read in place; page-locked host logits are read
    // by the GPU at the masked rows only; pageable host logits are copied whole.
    cudaPointerAttributes attr;
    const bool known = cudaPointerGetAttributes(&attr, logits) == cudaSuccess;
    if (!known)
        (void)cudaGetLastError();
    const bool on_device =
        known && (attr.type == cudaMemoryTypeDevice || attr.type == cudaMemoryTypeManaged);
    const void *mapped = known && attr.type == cudaMemoryTypeHost ? attr.devicePointer : nullptr;
    const size_t logits_bytes = on_device ? 0 : up256((size_t)(rows * row_bytes));
    const size_t off_mask = logits_bytes;
    const size_t off_tok = off_mask + up256((size_t)rows);
    const size_t off_commit = off_tok + up256((size_t)rows * 4);
    const size_t off_n = off_commit + up256((size_t)rows);
    const size_t total = off_n + up256((size_t)B * 4);
    void *stage = nullptr;
    st = staging_buffer(total, &stage);
    if (st != FDLLM_OK)
        return st;
    uint8_t *base = static_cast<uint8_t *>(stage);
    uint8_t *d_mask = base + off_mask;
    int32_t *d_tok = reinterpret_cast<int32_t *>(base + off_tok);
    uint8_t *d_commit = base + off_commit;
    int32_t *d_n = reinterpret_cast<int32_t *>(base + off_n);
    const void *d_logits = on_device ? logits : base;

    // Inputs: the mask, the caller's token array (the step writes only committed positions,
    // the others keep the caller's values), then the logits the step reads.
    if (cudaMemcpyAsync(d_mask, mask, (size_t)rows, cudaMemcpyDefault, s) != cudaSuccess ||
        cudaMemcpyAsync(d_tok, out_tokens, (size_t)rows * 4, cudaMemcpyDefault, s) !=
            cudaSuccess)
        return FDLLM_ERR_CUDA;
    if (!on_device) {
        if (mapped && (reinterpret_cast<uintptr_t>(mapped) & 15u) == 0) {
            if (launch_gather(mapped, base, d_mask, rows, row_bytes, s) != cudaSuccess)
                return FDLLM_ERR_CUDA;
        } else if (cudaMemcpyAsync(base, logits, (size_t)(rows * row_bytes), cudaMemcpyDefault,
                                   s) != cudaSuccess) {
            return FDLLM_ERR_CUDA;
        }
    }
    st = select_owned(d_logits, dtype, B, L, V, d_mask, param, mode, d_tok, d_commit, d_n, s,
                      true);
    if (st != FDLLM_OK)
        return st;
    if (cudaMemcpyAsync(out_tokens, d_tok, (size_t)rows * 4, cudaMemcpyDefault, s) !=
            cudaSuccess ||
        cudaMemcpyAsync(out_commit, d_commit, (size_t)rows, cudaMemcpyDefault, s) !=
            cudaSuccess ||
        cudaMemcpyAsync(out_n, d_n, (size_t)B * 4, cudaMemcpyDefault, s) != cudaSuccess ||
        cudaMemcpyAsync(mask, d_mask, (size_t)rows, cudaMemcpyDefault, s) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    return cudaStreamSynchronize(s) == cudaSuccess ? FDLLM_OK : FDLLM_ERR_CUDA;
}

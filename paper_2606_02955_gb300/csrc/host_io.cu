// host_io.cu -- the end-to-end path's input movement: the rows of masked positions are read
// by the GPU straight from page-locked host memory (over the host link) into a device buffer,
// so that only the logits the selection needs cross the link.
#include <cuda_runtime.h>

#include <cstdint>

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

}  // namespace
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
    cudaPointerAttributes attr;
    if (cudaPointerGetAttributes(&attr, src) != cudaSuccess) {
        (void)cudaGetLastError();
        return FDLLM_ERR_ARG;
    }
    const void *dsrc = nullptr;
    if (attr.type == cudaMemoryTypeDevice || attr.type == cudaMemoryTypeManaged)
        dsrc = src;
    else if (attr.type == cudaMemoryTypeHost)
        dsrc = attr.devicePointer;
    if (!dsrc || (reinterpret_cast<uintptr_t>(dsrc) & 15u))
        return FDLLM_ERR_ARG;  // pageable host memory: not readable by the GPU here
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((int64_t)B * L));
    cfg.blockDim = dim3(256);
    cfg.stream = static_cast<cudaStream_t>(stream);
    cudaLaunchAttribute a[1];
    a[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    a[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = a;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, gather_masked_rows_kernel, static_cast<const int4 *>(dsrc),
                              static_cast<int4 *>(dst), mask, row_bytes / 16) == cudaSuccess
               ? FDLLM_OK
               : FDLLM_ERR_CUDA;
}

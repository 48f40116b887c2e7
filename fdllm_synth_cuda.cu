// fdllm_synth_cuda.cu -- counter-based synthetic logits on the GPU: a stand-in for the
// model forward pass in decode-loop tests and benchmarks.  An input generator only (no
// selection arithmetic); the CPU oracle implements the same published generator itself.
//
// Definition (for seed s, step t, batch row b, block position l, vocabulary index v):
//   mix(z)     = SplitMix64 finaliser (Steele, Lea, Flood 2014):
//                z ^= z >> 30; z *= 0xBF58476D1CE4E5B9; z ^= z >> 27;
//                z *= 0x94D049BB133111EB; z ^= z >> 31
//   G          = 0x9E3779B97F4A7C15
//   row key  k = mix(s ^ mix(t * G ^ mix(((uint64)b << 32) | l)))
//   noise      h = mix(k + (v + 1) * G); u_j = (h >> 16 j) & 0xFFFF, j = 0..3;
//              x = float(sum_j (2 u_j + 1) - 262144) * fl32(sqrt(3) / 131072)
//              (Irwin-Hall sum of four uniforms, unit variance, one fp32 rounding)
//   peak       p = mix(k ^ 0xD1B54A32D192ED03); index p % V;
//              height = float(p >> 40) * fl32(peak_max / 2^24); x[index] += height (fp32)
//   bf16 output: round to nearest even.
#include <cstdint>

#include <cuda_bf16.h>
#include <cuda_runtime.h>

namespace {

__device__ __forceinline__ uint64_t mix64(uint64_t z)
{
    z ^= z >> 30;
    z *= 0xBF58476D1CE4E5B9ull;
    z ^= z >> 27;
    z *= 0x94D049BB133111EBull;
    z ^= z >> 31;
    return z;
}

constexpr uint64_t kGolden = 0x9E3779B97F4A7C15ull;

__device__ __forceinline__ uint64_t row_key(uint64_t seed, uint64_t step, uint32_t b, uint32_t l)
{
    return mix64(seed ^ mix64(step * kGolden ^ mix64(((uint64_t)b << 32) | l)));
}

// One CTA per (b, l) row of the block; rows whose mask byte is 0 are skipped.
__global__ void synth_block_logits(__nv_bfloat16 *out, const uint8_t *mask, int B, int L, int V,
                                   uint64_t seed, const int32_t *step_ptr, int64_t step_const,
                                   float noise_scale, float peak_scale)
{
    const int row = blockIdx.x;
    if (row >= B * L || (mask != nullptr && mask[row] == 0))
        return;
    const int b = row / L, l = row % L;
    const uint64_t step = step_ptr != nullptr ? (uint64_t)step_ptr[0] : (uint64_t)step_const;
    const uint64_t k = row_key(seed, step, (uint32_t)b, (uint32_t)l);
    const uint64_t p = mix64(k ^ 0xD1B54A32D192ED03ull);
    const int pidx = (int)(p % (uint64_t)V);
    const float height = (float)(p >> 40) * peak_scale;
    __nv_bfloat16 *o = out + (int64_t)row * V;
    for (int v = threadIdx.x; v < V; v += blockDim.x) {
        const uint64_t h = mix64(k + (uint64_t)(v + 1) * kGolden);
        const int32_t s = (int32_t)(2 * (h & 0xFFFF) + 2 * ((h >> 16) & 0xFFFF) +
                                    2 * ((h >> 32) & 0xFFFF) + 2 * ((h >> 48) & 0xFFFF) + 4) -
                          262144;
        float x = (float)s * noise_scale;
        if (v == pidx)
            x = __fadd_rn(x, height);
        o[v] = __float2bfloat16_rn(x);
    }
}

// Hidden states with a planted target (the LM-head counterpart of synth_block_logits).
// For row (b, l): k as above, p = mix(k ^ 0xD1B54A32D192ED03), target t = p % V, height
// beta = float(p >> 40) * fl32(beta_max / 2^24); noise z_j as the logits noise at index j;
// n2 = |w_t|^2 in fp32, lane i of 32 summing w_tj^2 for j = i, i + 32, ... in order, then an
// xor butterfly over offsets 16, 8, 4, 2, 1; scale = beta / n2 (IEEE division);
// h_j = z_j + scale * w_tj (each operation rounded to fp32), stored as bf16 (nearest even).
// Then w_t . h ~ beta + N(0, 1): a planted peak at t in the logits x = W h.
__global__ void synth_block_hidden(__nv_bfloat16 *out, const uint8_t *mask, int B, int L, int H,
                                   int V, const __nv_bfloat16 *w, uint64_t seed,
                                   const int32_t *step_ptr, int64_t step_const,
                                   float noise_scale, float beta_scale)
{
    __shared__ float s_scale;
    const int row = blockIdx.x;
    if (row >= B * L || (mask != nullptr && mask[row] == 0))
        return;
    const int b = row / L, l = row % L;
    const uint64_t step = step_ptr != nullptr ? (uint64_t)step_ptr[0] : (uint64_t)step_const;
    const uint64_t k = row_key(seed, step, (uint32_t)b, (uint32_t)l);
    const uint64_t p = mix64(k ^ 0xD1B54A32D192ED03ull);
    const int64_t t = (int64_t)(p % (uint64_t)V);
    const float beta = __fmul_rn((float)(p >> 40), beta_scale);
    const __nv_bfloat16 *wt = w + t * H;
    if (threadIdx.x < 32) {
        float acc = 0.0f;
        for (int j = threadIdx.x; j < H; j += 32) {
            const float x = __bfloat162float(wt[j]);
            acc = __fadd_rn(acc, __fmul_rn(x, x));
        }
        for (int o = 16; o > 0; o >>= 1)
            acc = __fadd_rn(acc, __shfl_xor_sync(0xFFFFFFFFu, acc, o));
        if (threadIdx.x == 0)
            s_scale = __fdiv_rn(beta, acc);
    }
    __syncthreads();
    const float scale = s_scale;
    __nv_bfloat16 *o = out + (int64_t)row * H;
    for (int j = threadIdx.x; j < H; j += blockDim.x) {
        const uint64_t h = mix64(k + (uint64_t)(j + 1) * kGolden);
        const int32_t sv = (int32_t)(2 * (h & 0xFFFF) + 2 * ((h >> 16) & 0xFFFF) +
                                     2 * ((h >> 32) & 0xFFFF) + 2 * ((h >> 48) & 0xFFFF) + 4) -
                           262144;
        const float z = __fmul_rn((float)sv, noise_scale);
        o[j] = __float2bfloat16_rn(__fadd_rn(z, __fmul_rn(scale, __bfloat162float(wt[j]))));
    }
}

}  // namespace

extern "C" {

// Enqueue synthetic bf16 hidden states [B, L, H] for the masked rows against the bf16 head
// w [V, H]; the step as for fdllm_synth_block_logits.
int fdllm_synth_block_hidden(void *out, const uint8_t *mask, int B, int L, int H, int V,
                             const void *w, unsigned long long seed, const int32_t *step_ptr,
                             long long step_const, double beta_max, void *stream)
{
    const float noise_scale = (float)(1.7320508075688772 / 131072.0);
    const float beta_scale = (float)(beta_max / 16777216.0);
    synth_block_hidden<<<B * L, 128, 0, static_cast<cudaStream_t>(stream)>>>(
        static_cast<__nv_bfloat16 *>(out), mask, B, L, H, V,
        static_cast<const __nv_bfloat16 *>(w), seed, step_ptr, step_const, noise_scale,
        beta_scale);
    return (int)cudaGetLastError();
}


// Enqueue synthetic bf16 logits [B, L, V] for the masked rows (mask may be NULL: all rows).
// The step comes from device memory (step_ptr, read when the kernel runs, so a captured
// graph draws fresh logits every iteration) or, when step_ptr is NULL, from step_const.
int fdllm_synth_block_logits(void *out, const uint8_t *mask, int B, int L, int V,
                             unsigned long long seed, const int32_t *step_ptr,
                             long long step_const, double peak_max, void *stream)
{
    const float noise_scale = (float)(1.7320508075688772 / 131072.0);
    const float peak_scale = (float)(peak_max / 16777216.0);
    synth_block_logits<<<B * L, 256, 0, static_cast<cudaStream_t>(stream)>>>(
        static_cast<__nv_bfloat16 *>(out), mask, B, L, V, seed, step_ptr, step_const,
        noise_scale, peak_scale);
    return (int)cudaGetLastError();
}

}  // extern "C"

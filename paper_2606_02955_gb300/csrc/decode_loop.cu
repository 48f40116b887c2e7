// decode_loop.cu -- Algorithm 1's outer loop resident on the GPU: for every block of the
// generation, repeat {forward pass; selection; reveal} while the block has masked positions,
// then move to the next block.  The loop is one CUDA graph whose body sits in a conditional
// WHILE node; a controller kernel at the end of each iteration reveals the committed tokens
// into the sequence, counts the steps (NFE) of the block, advances to the next block and
// clears the loop condition after the last one.  No host round trip per step.
#include <cuda_runtime.h>

#include <cstdint>

#include "fdllm.h"
#include "fdllm_internal.cuh"

namespace fdllm {
namespace {

// Why the loop stopped before the generation finished (LoopState::stop_reason).
constexpr int32_t kStopNone = 0;
constexpr int32_t kStopMaxSteps = 1;   // max_steps reached
constexpr int32_t kStopNonfinite = 2;  // a row's logits were unusable (FDLLM_ROW_NONFINITE)
constexpr int32_t kStopDevice = 3;     // a kernel gave up a bounded wait (FDLLM_ROW_DEVICE_ERROR)

struct LoopState {
    int32_t step;         // global step (forward passes so far)
    int32_t block;        // current block
    int32_t block_steps;  // steps spent in the current block
    int32_t stop_reason;  // kStop*: nonzero when the loop ended early
};

__global__ void loop_init_kernel(LoopState *st, uint8_t *block_mask, int64_t block_rows,
                                 int32_t *seq, int64_t seq_len, int32_t *nfe, int nblocks)
{
    const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    if (tid == 0) {
        st->step = 0;
        st->block = 0;
        st->block_steps = 0;
        st->stop_reason = kStopNone;
    }
    for (int64_t i = tid; i < block_rows; i += stride)
        block_mask[i] = 1;
    for (int64_t i = tid; i < seq_len; i += stride)
        seq[i] = -1;
    for (int64_t i = tid; i < nblocks; i += stride)
        nfe[i] = 0;
}

// One CTA.  Runs after the step's selection: reveal (Alg. 1) into the sequence, count the
// step, and at the end of a block move on (re-mask the block buffer) or stop the loop.  A
// step whose selection reported a row as unusable or failed ends the loop: such a row
// commits nothing, so the block would never finish.
__global__ void loop_control_kernel(LoopState *st, uint8_t *block_mask, const uint8_t *commit,
                                    const int32_t *block_tokens, const int32_t *block_n,
                                    int32_t *seq, int32_t *nfe, int B, int Lb, int gen_len,
                                    int nblocks, int max_steps, cudaGraphConditionalHandle cond)
{
    __shared__ int any_masked;
    __shared__ int advance;
    __shared__ int worst_n;
    if (threadIdx.x == 0) {
        any_masked = 0;
        advance = 0;
        worst_n = 0;
    }
    __syncthreads();
    const int blk = st->block;
    for (int i = threadIdx.x; i < B * Lb; i += blockDim.x) {
        if (commit[i]) {
            const int b = i / Lb, l = i % Lb;
            seq[(int64_t)b * gen_len + (int64_t)blk * Lb + l] = block_tokens[i];
        }
        if (block_mask[i])
            any_masked = 1;
    }
    for (int b = threadIdx.x; b < B; b += blockDim.x)
        if (block_n[b] < 0)
            atomicMin(&worst_n, block_n[b]);
    __syncthreads();
    if (threadIdx.x == 0) {
        st->step += 1;
        st->block_steps += 1;
        bool stop = false;
        if (worst_n < 0) {
            st->stop_reason = worst_n == FDLLM_ROW_DEVICE_ERROR ? kStopDevice : kStopNonfinite;
            nfe[blk] = st->block_steps;
            stop = true;
        } else if (!any_masked) {
            nfe[blk] = st->block_steps;
            st->block = blk + 1;
            st->block_steps = 0;
            stop = blk + 1 >= nblocks;
            advance = !stop;
        }
        if (!stop && st->step >= max_steps) {
            st->stop_reason = kStopMaxSteps;
            nfe[blk] = st->block_steps;
            stop = true;
            advance = 0;
        }
        if (stop)
            cudaGraphSetConditional(cond, 0);
    }
    __syncthreads();
    if (advance)
        for (int i = threadIdx.x; i < B * Lb; i += blockDim.x)
            block_mask[i] = 1;
}

// The loop's graph: a conditional WHILE node whose body is {forward; selection;
// controller}, captured from `cs`.  The condition starts at 1 on every launch.
struct LoopGraph {
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    ~LoopGraph()
    {
        if (exec)
            cudaGraphExecDestroy(exec);
        if (graph)
            cudaGraphDestroy(graph);
    }
};

struct LoopArgs {
    int B, Lb, V, dtype, mode, gen_len, nblocks, max_steps;
    double param;
    fdllm_forward_fn forward;
    void *user;
    void *logits;           // what the forward pass writes: logits, or hidden states with w_vocab
    const void *w_vocab;    // non-null: the selection runs on the LM head (hidden size H)
    int H;
    int32_t *seq;
    int32_t *nfe;
    LoopState *st;
    uint8_t *block_mask, *commit;
    int32_t *block_tokens, *block_n;
};

// One step's selection on the block buffer: from logits, or from hidden states through the
// LM head.
fdllm_status run_step_select(const LoopArgs &a, cudaStream_t s, bool pdl)
{
    if (a.w_vocab)
        return lmhead_select_owned(a.logits, a.w_vocab, a.B, a.Lb, a.H, a.V, a.block_mask,
                                   a.param, a.mode, a.block_tokens, a.commit, a.block_n, s, pdl);
    return select_owned(a.logits, a.dtype, a.B, a.Lb, a.V, a.block_mask, a.param, a.mode,
                        a.block_tokens, a.commit, a.block_n, s, pdl);
}

fdllm_status build_loop_graph(const LoopArgs &a, cudaStream_t cs, bool pdl, LoopGraph &g)
{
    cudaGraphConditionalHandle cond;
    if (cudaGraphCreate(&g.graph, 0) != cudaSuccess ||
        cudaGraphConditionalHandleCreate(&cond, g.graph, 1, cudaGraphCondAssignDefault) !=
            cudaSuccess)
        return FDLLM_ERR_CUDA;
    cudaGraphNodeParams cp = {};
    cp.type = cudaGraphNodeTypeConditional;
    cp.conditional.handle = cond;
    cp.conditional.type = cudaGraphCondTypeWhile;
    cp.conditional.size = 1;
    cudaGraphNode_t loop_node;
    if (cudaGraphAddNode(&loop_node, g.graph, nullptr, nullptr, 0, &cp) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    cudaGraph_t body = cp.conditional.phGraph_out[0];
    if (cudaStreamBeginCaptureToGraph(cs, body, nullptr, nullptr, 0,
                                      cudaStreamCaptureModeRelaxed) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    fdllm_status st = FDLLM_OK;
    if (a.forward(a.user, &a.st->step, a.block_mask, a.logits, cs) != 0)
        st = FDLLM_ERR_ARG;
    if (st == FDLLM_OK)
        st = run_step_select(a, cs, pdl);
    if (st == FDLLM_OK) {
        loop_control_kernel<<<1, 256, 0, cs>>>(a.st, a.block_mask, a.commit, a.block_tokens,
                                               a.block_n, a.seq, a.nfe, a.B, a.Lb, a.gen_len,
                                               a.nblocks, a.max_steps, cond);
        if (cudaGetLastError() != cudaSuccess)
            st = FDLLM_ERR_CUDA;
    }
    cudaGraph_t captured = nullptr;
    if (cudaStreamEndCapture(cs, &captured) != cudaSuccess && st == FDLLM_OK)
        st = FDLLM_ERR_CUDA;
    if (st != FDLLM_OK)
        return st;
    if (cudaGraphInstantiate(&g.exec, g.graph, 0) != cudaSuccess)
        return FDLLM_ERR_CUDA;
    return FDLLM_OK;
}

}  // namespace
}  // namespace fdllm

using namespace fdllm;

namespace fdllm {
namespace {

fdllm_status run_decode_loop(LoopArgs a, int *out_steps, cudaStream_t s)
{
    if (a.B < 1 || a.Lb < 1 || a.Lb > FDLLM_MAX_L || a.gen_len < a.Lb ||
        a.gen_len % a.Lb != 0 || (int64_t)a.B * a.Lb > FDLLM_MAX_ROWS || a.max_steps < 1 ||
        !a.forward || !a.logits || !a.seq || !a.nfe || !out_steps)
        return FDLLM_ERR_ARG;
    if (a.mode != FDLLM_PROFILE && a.mode != FDLLM_FACTOR && a.mode != FDLLM_THRESHOLD)
        return FDLLM_ERR_ARG;
    *out_steps = 0;
    const int B = a.B, Lb = a.Lb, gen_len = a.gen_len;
    a.nblocks = gen_len / Lb;
    const int64_t rows = (int64_t)B * Lb;
    cudaStream_t cs = nullptr;
    fdllm_status result = FDLLM_ERR_CUDA;

    do {
        if (cudaMalloc(&a.st, sizeof(LoopState)) != cudaSuccess ||
            cudaMalloc(&a.block_mask, rows) != cudaSuccess ||
            cudaMalloc(&a.commit, rows) != cudaSuccess ||
            cudaMalloc(&a.block_tokens, rows * sizeof(int32_t)) != cudaSuccess ||
            cudaMalloc(&a.block_n, (size_t)B * sizeof(int32_t)) != cudaSuccess)
            break;
        // One selection on an all-unmasked block, outside the graph, checks the arguments
        // and sizes the library workspace (nothing may be allocated inside the captured body).
        if (cudaMemsetAsync(a.block_mask, 0, rows, s) != cudaSuccess)
            break;
        fdllm_status pre = run_step_select(a, s, true);
        if (pre != FDLLM_OK) {
            result = pre;
            break;
        }
        if (cudaStreamSynchronize(s) != cudaSuccess ||
            cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) != cudaSuccess)
            break;
        LoopGraph with_pdl, plain;
        LoopGraph *g = &with_pdl;
        fdllm_status built = build_loop_graph(a, cs, true, with_pdl);
        if (built == FDLLM_ERR_CUDA) {
            // Programmatic edges inside the conditional body were not accepted: capture
            // the same body in plain stream order.
            (void)cudaGetLastError();
            g = &plain;
            built = build_loop_graph(a, cs, false, plain);
        }
        if (built != FDLLM_OK) {
            result = built;
            break;
        }
        const int64_t total = rows > (int64_t)B * gen_len ? rows : (int64_t)B * gen_len;
        const int threads = 256;
        const int blocks = (int)((total + threads - 1) / threads);
        loop_init_kernel<<<blocks, threads, 0, s>>>(a.st, a.block_mask, rows, a.seq,
                                                     (int64_t)B * gen_len, a.nfe, a.nblocks);
        if (cudaGetLastError() != cudaSuccess || cudaGraphLaunch(g->exec, s) != cudaSuccess)
            break;
        LoopState host;
        if (cudaMemcpyAsync(&host, a.st, sizeof host, cudaMemcpyDeviceToHost, s) !=
                cudaSuccess ||
            cudaStreamSynchronize(s) != cudaSuccess)
            break;
        *out_steps = host.step;
        result = host.stop_reason == kStopNone        ? FDLLM_OK
                 : host.stop_reason == kStopNonfinite ? FDLLM_ERR_NONFINITE
                                                      : FDLLM_ERR_DEVICE;
    } while (false);

    if (cs)
        cudaStreamDestroy(cs);
    cudaStreamSynchronize(s);
    cudaFree(a.st);
    cudaFree(a.block_mask);
    cudaFree(a.commit);
    cudaFree(a.block_tokens);
    cudaFree(a.block_n);
    return result;
}

}  // namespace
}  // namespace fdllm

extern "C" fdllm_status fdllm_decode_loop(int B, int gen_len, int block_len, int V, int dtype,
                                          double param, int mode, fdllm_forward_fn forward,
                                          void *user, void *logits, int32_t *seq_tokens,
                                          int32_t *nfe_per_block, int max_steps, int *out_steps,
                                          void *stream)
{
    LoopArgs a = {};
    a.B = B;
    a.Lb = block_len;
    a.V = V;
    a.dtype = dtype;
    a.mode = mode;
    a.gen_len = gen_len;
    a.max_steps = max_steps;
    a.param = param;
    a.forward = forward;
    a.user = user;
    a.logits = logits;
    a.seq = seq_tokens;
    a.nfe = nfe_per_block;
    return run_decode_loop(a, out_steps, static_cast<cudaStream_t>(stream));
}

extern "C" fdllm_status fdllm_decode_loop_lmhead(int B, int gen_len, int block_len, int H, int V,
                                                 const void *w_vocab, double param, int mode,
                                                 fdllm_forward_fn forward, void *user,
                                                 void *hidden, int32_t *seq_tokens,
                                                 int32_t *nfe_per_block, int max_steps,
                                                 int *out_steps, void *stream)
{
    if (!w_vocab)
        return FDLLM_ERR_ARG;
    LoopArgs a = {};
    a.B = B;
    a.Lb = block_len;
    a.V = V;
    a.dtype = FDLLM_BF16;
    a.mode = mode;
    a.gen_len = gen_len;
    a.max_steps = max_steps;
    a.param = param;
    a.forward = forward;
    a.user = user;
    a.logits = hidden;
    a.w_vocab = w_vocab;
    a.H = H;
    a.seq = seq_tokens;
    a.nfe = nfe_per_block;
    return run_decode_loop(a, out_steps, static_cast<cudaStream_t>(stream));
}

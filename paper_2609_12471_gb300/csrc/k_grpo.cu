// GRPO token loss and its batch mean (Sec. "GRPO Optimization", Eq. advantage and
// Eq. ppo).  One CTA per row forms (or, after the scoring epilogue formed them,
// reads) the row's token losses and sums mask * loss and the mask in a fixed order;
// one CTA then adds the rows in row order.  Both passes are deterministic.
#include "qk_internal.cuh"

namespace qk {

namespace {

constexpr int kThreads = 256;

// Sum over the block in a fixed order (warp shuffles, then the warps in order).
__device__ float2 block_sum2(float2 v, float2* red) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        v.x += __shfl_xor_sync(0xffffffffu, v.x, o);
        v.y += __shfl_xor_sync(0xffffffffu, v.y, o);
    }
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    if (l == 0) red[w] = v;
    __syncthreads();
    float2 t = make_float2(0.f, 0.f);
    if (threadIdx.x == 0)
        for (int i = 0; i < (int)(blockDim.x >> 5); ++i) t.x += red[i].x, t.y += red[i].y;
    return t;  // valid in thread 0
}

__global__ void __launch_bounds__(kThreads)
    grpo_rows_kernel(const float* __restrict__ lp, int T, GrpoArgs g, bool compute,
                     float2* __restrict__ rows) {
    __shared__ float2 red[kThreads / 32];
    pdl_wait();
    pdl_trigger();
    const int b = blockIdx.x;
    const size_t r0 = (size_t)b * g.ld;
    const float A = compute ? grpo_advantage(g.rewards, b, g.group) : 0.f;
    float2 acc = make_float2(0.f, 0.f);
    for (int t = threadIdx.x; t < T; t += blockDim.x) {
        float L;
        if (compute) {
            const float l = lp[r0 + t];
            L = grpo_token(l, g.lp_old[r0 + t], g.lp_ref ? g.lp_ref[r0 + t] : l, A, g);
            g.loss_tok[r0 + t] = L;
        } else {
            L = g.loss_tok[r0 + t];
        }
        const float m = g.mask ? (float)g.mask[r0 + t] : 1.f;
        acc.x += m * L;
        acc.y += m;
    }
    const float2 tot = block_sum2(acc, red);
    if (threadIdx.x == 0) rows[b] = tot;
}

__global__ void __launch_bounds__(kThreads)
    grpo_mean_kernel(const float2* __restrict__ rows, int B, float* __restrict__ loss_mean) {
    __shared__ float2 red[kThreads / 32];
    pdl_wait();
    pdl_trigger();
    float2 acc = make_float2(0.f, 0.f);
    for (int b = threadIdx.x; b < B; b += blockDim.x) acc.x += rows[b].x, acc.y += rows[b].y;
    const float2 tot = block_sum2(acc, red);
    if (threadIdx.x == 0) *loss_mean = tot.y > 0.f ? tot.x / tot.y : 0.f;
}

// d L_t / d lp_t of Eq. ppo: rho A where the unclipped term is the minimum (its
// derivative; rho = exp(lp - lp_old) has d rho / d lp = rho), 0 where the clipped term
// is smaller (clip(rho) is then constant), plus beta (1 - e^x), x = lp_ref - lp, the
// derivative of k3.  coef = -mask * dL / n with n the batch's mask count (so that the
// gradient of sum coef * (-lp) is the gradient of the masked token mean).
__global__ void __launch_bounds__(kThreads)
    grpo_coef_kernel(const float* __restrict__ lp, int T, GrpoArgs g, const float2* __restrict__ rows,
                     int B, float* __restrict__ coef) {
    __shared__ float2 red[kThreads / 32];
    __shared__ float n_sh;
    pdl_wait();
    float2 acc = make_float2(0.f, 0.f);
    for (int b = threadIdx.x; b < B; b += blockDim.x) acc.y += rows[b].y;
    const float2 tot = block_sum2(acc, red);
    if (threadIdx.x == 0) n_sh = tot.y;
    __syncthreads();
    const float n = n_sh;
    const int b = blockIdx.x;
    const size_t r0 = (size_t)b * g.ld;
    const float A = grpo_advantage(g.rewards, b, g.group);
    for (int t = threadIdx.x; t < T; t += blockDim.x) {
        const float l = lp[r0 + t];
        const float rho = expf(l - g.lp_old[r0 + t]);
        const float clipped = fminf(fmaxf(rho, 1.f - g.eps_low), 1.f + g.eps_high);
        float dL = rho * A <= clipped * A ? -rho * A : 0.f;
        if (g.beta != 0.f) dL += g.beta * (1.f - expf(g.lp_ref[r0 + t] - l));
        const float m = g.mask ? (float)g.mask[r0 + t] : 1.f;
        coef[r0 + t] = n > 0.f ? -m * dL / n : 0.f;
    }
}

}  // namespace

void launch_grpo_coef(const float* lp, int B, int T, const GrpoArgs& g, const void* scratch, float* coef,
                      cudaStream_t s) {
    launch_k(grpo_coef_kernel, dim3(B), dim3(kThreads), 0, s, lp, T, g, (const float2*)scratch, B, coef);
    note_launch();
}

size_t grpo_scratch_bytes(int B) { return (((size_t)B * sizeof(float2)) + 255) & ~(size_t)255; }

void launch_grpo_loss(const float* lp, int B, int T, const GrpoArgs& g, bool compute,
                      void* scratch, float* loss_mean, cudaStream_t s) {
    float2* rows = (float2*)scratch;
    launch_k(grpo_rows_kernel, dim3(B), dim3(kThreads), 0, s, lp, T, g, compute, rows);
    note_launch();
    if (loss_mean) {
        launch_k(grpo_mean_kernel, dim3(1), dim3(kThreads), 0, s, (const float2*)rows, B, loss_mean);
        note_launch();
    }
}

}  // namespace qk

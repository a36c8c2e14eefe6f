// Forward of the multi-level training objective of Sec. 2.3 (Eq. 3-6) on a draft's logits
// and hidden states (NEXT to the drafting path: it reads the full-vocabulary logits that
// fe_draft_forward writes to its dbg_logits buffer):
//   ce_i   = -sum_k p_k log q_k,  q = softmax(logits_i)  (Eq. 4)  = lse_i * sum_k p_k - sum_k p_k logits_k
//   feat_i = sum_j SmoothL1(h_ij - f_ij)                    (Eq. 5, 6)
//   total  = sum_i w_i (alpha ce_i + beta feat_i), w_i = decay^(N - i), i = 1..N   (Eq. 3)
// loss_row_kernel: one CTA per (depth i, sequence b), two passes over the row (max, then
// sum of exp, sum of p and of p * logit); loss_total_kernel: one thread per sequence.
#include "fe_kernels.h"
#include "fe_common.cuh"

namespace fe {

namespace {

constexpr int kLossThreads = 256;

__device__ __forceinline__ float block_reduce(float v, float* red, bool is_max) {
    v = is_max ? warp_max(v) : warp_sum(v);
    const int w = threadIdx.x >> 5;
    __syncthreads();  // red may still be read from the previous reduction
    if ((threadIdx.x & 31) == 0) red[w] = v;
    __syncthreads();
    float r = red[0];
    for (int i = 1; i < kLossThreads / 32; ++i) r = is_max ? fmaxf(r, red[i]) : r + red[i];
    return r;
}

__device__ __forceinline__ float smooth_l1(float x) {
    const float a = fabsf(x);
    return a < 1.f ? 0.5f * x * x : a - 0.5f;
}

__global__ void __launch_bounds__(kLossThreads) loss_row_kernel(int N, int B, int V, int d, const float* logits,
                                                                 const float* teacher, const float* hidden,
                                                                 const float* feat, float* ce, float* fl) {
    __shared__ float red[kLossThreads / 32];
    const int i = blockIdx.x, b = blockIdx.y, t = threadIdx.x;
    const size_t row = (size_t)b * N + i;
    const float* lg = logits + row * V;
    const float* p = teacher + row * V;
    float m = -INFINITY;
    for (int k = t; k < V; k += kLossThreads) m = fmaxf(m, lg[k]);
    const float M = block_reduce(m, red, true);
    float s = 0.f, sp = 0.f, spl = 0.f;
    for (int k = t; k < V; k += kLossThreads) {
        const float x = lg[k], pk = p[k];
        s += expf(x - M);
        sp += pk;
        spl = fmaf(pk, x, spl);
    }
    const float S = block_reduce(s, red, false);
    const float SP = block_reduce(sp, red, false);
    const float SPL = block_reduce(spl, red, false);
    const float* h = hidden + ((size_t)i * B + b) * d;
    const float* f = feat + ((size_t)i * B + b) * d;
    float a = 0.f;
    for (int j = t; j < d; j += kLossThreads) a += smooth_l1(h[j] - f[j]);
    const float A = block_reduce(a, red, false);
    if (t == 0) {
        ce[row] = (M + logf(S)) * SP - SPL;
        fl[row] = A;
    }
}

__global__ void loss_total_kernel(int N, int B, const float* ce, const float* fl, float alpha, float beta, float decay,
                                  float* total) {
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= B) return;
    float acc = 0.f;
    for (int i = 0; i < N; ++i) {
        const float w = powf(decay, (float)(N - 1 - i));
        acc = fmaf(w, alpha * ce[(size_t)b * N + i] + beta * fl[(size_t)b * N + i], acc);
    }
    total[b] = acc;
}

}  // namespace

cudaError_t launch_loss(int N, int B, int V, int d, const float* logits, const float* teacher, const float* hidden,
                        const float* feat, float alpha, float beta, float decay, float* ce, float* fl, float* total,
                        cudaStream_t st) {
    loss_row_kernel<<<dim3(N, B), kLossThreads, 0, st>>>(N, B, V, d, logits, teacher, hidden, feat, ce, fl);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    loss_total_kernel<<<(B + 127) / 128, 128, 0, st>>>(N, B, ce, fl, alpha, beta, decay, total);
    return cudaGetLastError();
}

}  // namespace fe

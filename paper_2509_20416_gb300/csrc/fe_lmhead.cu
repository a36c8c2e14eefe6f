// The frozen LM head applied to every cascade output h_i (Sec. 2.1), fused with the
// softmax statistics and the top-k selection of Sec. 2.2, so the [N*B, V] logits never
// reach global memory.
//
// Kernel 1 (lmhead_kernel): one weight-streaming CTA per vocabulary slab (a contiguous
// range of LM-head rows). The hidden rows z_r = RMSNorm(h_r; gamma_out) of all N*B rows
// are staged once in shared memory, so the LM head is read from HBM once for all N
// depths. Per row r the CTA keeps a running top-k (by logit, ties to the smaller id)
// and the running (max, sum of exp) of logit / T, and writes them as the slab's partial.
// Kernel 2 (topk_merge_kernel): one CTA per row merges the slabs' partials: k rounds of
// a block arg-max over n_slabs * k candidates, lse = M + log sum_j s_j e^(m_j - M), and
// prob = exp(logit / T - lse).
#include <float.h>

#include "fe_kernels.h"
#include "fe_stream.cuh"

namespace fe {

constexpr int kMaxTopK = 32;

__device__ __forceinline__ bool better(float va, int ia, float vb, int ib) {
    return va > vb || (va == vb && ia < ib);
}

struct TopkState {
    int id[8][kMaxTopK];
    float val[8][kMaxTopK];
    int cnt[8];
    float m[8], s[8];
};

template <int BT>
struct LmEpi {
    const LmHeadArgs* a;
    TopkState* st;
    int b0, nb;
    __device__ __forceinline__ void operator()(int g, const float* red) const {
        const int t = threadIdx.x;
        if (t >= nb) return;
        const int zr = b0 + t;
        const int k = a->top_k;
        int* ids = st->id[t];
        float* vals = st->val[t];
        int cnt = st->cnt[t];
        float m = st->m[t], s = st->s[t];
        for (int r = 0; r < kGroupRows; ++r) {
            const int v = g * kGroupRows + r;
            if (v >= a->V) break;
            const float lg = group_sum<BT>(red, r, t);
            if (a->dbg_logits) {
                const int i = zr / a->B, b = zr % a->B;
                a->dbg_logits[((size_t)b * a->N + i) * a->V + v] = lg;
            }
            const float lt = lg * a->inv_temp;
            if (lt > m) {
                s = s * expf(m - lt) + 1.0f;
                m = lt;
            } else {
                s += expf(lt - m);
            }
            int pos;
            if (cnt < k) {
                pos = cnt++;
            } else if (better(lg, v, vals[k - 1], ids[k - 1])) {
                pos = k - 1;
            } else {
                continue;
            }
            while (pos > 0 && better(lg, v, vals[pos - 1], ids[pos - 1])) {
                vals[pos] = vals[pos - 1];
                ids[pos] = ids[pos - 1];
                --pos;
            }
            vals[pos] = lg;
            ids[pos] = v;
        }
        st->cnt[t] = cnt;
        st->m[t] = m;
        st->s[t] = s;
    }
};

template <typename WT, int BT>
__global__ void __launch_bounds__(kStreamThreads, 1) lmhead_kernel(const LmHeadArgs a, int ns) {
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ TopkState st;
    const int K = a.d;
    const int Kpad = (K + 3) & ~3;
    const int b0 = blockIdx.y * BT;
    const int nb = min(BT, a.R - b0);
    StreamSmem s = carve_stream_smem(smem, ns, min(BT, a.R), Kpad, BT);
    if (threadIdx.x < 8) {
        st.cnt[threadIdx.x] = 0;
        st.m[threadIdx.x] = -INFINITY;
        st.s[threadIdx.x] = 0.f;
    }
    stream_init_barriers(s, ns);

    const int GM = (a.V + kGroupRows - 1) / kGroupRows;
    const int slab = blockIdx.x;
    const int g0 = (int)(((int64_t)slab * GM) / gridDim.x);
    const int g1 = (int)(((int64_t)(slab + 1) * GM) / gridDim.x);

    if (threadIdx.x >= kConsumers) {
        if (threadIdx.x == kConsumers) stream_produce<WT>((const unsigned char*)a.W, a.V, K, g0, g1, s, ns, a.status);
        return;
    }
    ProParams pp{PRO_RMSNORM, a.hid, a.d, a.gamma, a.eps, nullptr, nullptr, 0, 0};
    stage_activations<WT>(pp, K, s.X, Kpad, b0, nb, a.status, s.red);
    named_sync(1, kConsumers);
    LmEpi<BT> ep{&a, &st, b0, nb};
    stream_consume<WT, BT>(K, g0, g1, s, ns, Kpad, nb, a.status, ep);

    // partials of this slab (entries past cnt are padding that loses every comparison)
    const int t = threadIdx.x;
    if (t < nb) {
        const int zr = b0 + t;
        const size_t base = ((size_t)zr * a.n_slabs + slab);
        for (int j = 0; j < a.top_k; ++j) {
            const bool ok = j < st.cnt[t];
            a.part_id[base * a.top_k + j] = ok ? st.id[t][j] : INT_MAX;
            a.part_val[base * a.top_k + j] = ok ? st.val[t][j] : -INFINITY;
        }
        a.part_ms[base * 2 + 0] = st.m[t];
        a.part_ms[base * 2 + 1] = st.s[t];
    }
}

__global__ void __launch_bounds__(256) topk_merge_kernel(const MergeArgs a) {
    extern __shared__ __align__(16) unsigned char smem[];
    const int zr = blockIdx.x;
    const int n = a.n_slabs * a.top_k;
    float* vals = (float*)smem;
    int* ids = (int*)(vals + n);
    __shared__ float rv[8];
    __shared__ int ri[8], rp[8];
    __shared__ float s_lse;
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    for (int j = t; j < n; j += 256) {
        vals[j] = a.part_val[(size_t)zr * n + j];
        ids[j] = a.part_id[(size_t)zr * n + j];
    }
    // lse of logit / T from the slabs' (max, sum) pairs
    float M = -INFINITY;
    for (int j = t; j < a.n_slabs; j += 256) M = fmaxf(M, a.part_ms[((size_t)zr * a.n_slabs + j) * 2]);
    M = warp_max(M);
    if (lane == 0) rv[warp] = M;
    __syncthreads();
    M = rv[0];
    for (int w = 1; w < 8; ++w) M = fmaxf(M, rv[w]);
    __syncthreads();
    float S = 0.f;
    for (int j = t; j < a.n_slabs; j += 256) {
        const float mj = a.part_ms[((size_t)zr * a.n_slabs + j) * 2];
        const float sj = a.part_ms[((size_t)zr * a.n_slabs + j) * 2 + 1];
        if (sj > 0.f) S += sj * expf(mj - M);
    }
    S = warp_sum(S);
    if (lane == 0) rv[warp] = S;
    __syncthreads();
    if (t == 0) {
        float tot = 0.f;
        for (int w = 0; w < 8; ++w) tot += rv[w];
        s_lse = M + logf(tot);
    }
    __syncthreads();
    const float lse = s_lse;
    const int i = zr / a.B, b = zr % a.B;
    const size_t ob = ((size_t)b * a.N + i) * a.top_k;
    for (int r = 0; r < a.top_k; ++r) {
        float bv = -INFINITY;
        int bi = INT_MAX, bp = -1;
        for (int j = t; j < n; j += 256) {
            if (bp < 0 || better(vals[j], ids[j], bv, bi)) {
                bv = vals[j];
                bi = ids[j];
                bp = j;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
            const int op = __shfl_xor_sync(0xffffffffu, bp, o);
            if (op >= 0 && (bp < 0 || better(ov, oi, bv, bi))) { bv = ov; bi = oi; bp = op; }
        }
        if (lane == 0) { rv[warp] = bv; ri[warp] = bi; rp[warp] = bp; }
        __syncthreads();
        if (t == 0) {
            for (int w = 1; w < 8; ++w)
                if (rp[w] >= 0 && (rp[0] < 0 || better(rv[w], ri[w], rv[0], ri[0]))) {
                    rv[0] = rv[w]; ri[0] = ri[w]; rp[0] = rp[w];
                }
            a.topk_id[ob + r] = ri[0];
            a.topk_logit[ob + r] = rv[0];
            a.topk_prob[ob + r] = expf(rv[0] * a.inv_temp - lse);
            if (rp[0] >= 0) { vals[rp[0]] = -INFINITY; ids[rp[0]] = INT_MAX; }
        }
        __syncthreads();
    }
    if (t == 0) a.lse[(size_t)b * a.N + i] = lse;
}

// ---- host side ----------------------------------------------------------------------------
namespace {
constexpr size_t kXBudget = 128 * 1024;
constexpr size_t kStaticReserve = sizeof(TopkState) + 256;

int pick_bt(int R, int K) {
    const size_t row = (size_t)((K + 3) & ~3) * sizeof(float);
    int bt = 8;
    while (bt > 1 && ((size_t)(bt < R ? bt : R) * row > kXBudget || bt / 2 >= R)) bt >>= 1;
    return bt;
}

template <typename WT, int BT>
cudaError_t set_attr(const DeviceInfo& dev) {
    return cudaFuncSetAttribute(lmhead_kernel<WT, BT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                dev.max_smem_optin - (int)kStaticReserve);
}

template <typename WT, int BT>
cudaError_t launch_bt(const LmHeadArgs& a, const DeviceInfo& dev, cudaStream_t st) {
    const int Kpad = (a.d + 3) & ~3;
    const int xrows = BT < a.R ? BT : a.R;
    const size_t budget = (size_t)dev.max_smem_optin - kStaticReserve;
    const size_t fixed = stream_smem_bytes(0, xrows, Kpad, BT);
    int ns = (int)((budget - fixed) / (kStageBytes + 16));
    ns = ns > kMaxStages ? kMaxStages : ns;
    if (ns < 2) return cudaErrorInvalidValue;
    dim3 grid(a.n_slabs, (a.R + BT - 1) / BT);
    lmhead_kernel<WT, BT><<<grid, kStreamThreads, stream_smem_bytes(ns, xrows, Kpad, BT), st>>>(a, ns);
    return cudaGetLastError();
}

template <typename WT>
cudaError_t launch_t(const LmHeadArgs& a, const DeviceInfo& dev, cudaStream_t st) {
    switch (pick_bt(a.R, a.d)) {
        case 1: return launch_bt<WT, 1>(a, dev, st);
        case 2: return launch_bt<WT, 2>(a, dev, st);
        case 4: return launch_bt<WT, 4>(a, dev, st);
        default: return launch_bt<WT, 8>(a, dev, st);
    }
}
}  // namespace

cudaError_t lmhead_prepare(const DeviceInfo& dev) {
    cudaError_t e;
    if ((e = set_attr<float, 1>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<float, 2>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<float, 4>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<float, 8>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<bf16_t, 1>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<bf16_t, 2>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<bf16_t, 4>(dev)) != cudaSuccess) return e;
    return set_attr<bf16_t, 8>(dev);
}

int lmhead_slabs(int V, const DeviceInfo& dev) {
    const int GM = (V + kGroupRows - 1) / kGroupRows;
    return GM < dev.num_sms ? GM : dev.num_sms;
}

int lmhead_launches(int, int, const DeviceInfo&) { return 2; }

cudaError_t launch_lmhead(fe_dtype dt, const LmHeadArgs& a, const DeviceInfo& dev, cudaStream_t st) {
    return dt == FE_F32 ? launch_t<float>(a, dev, st) : launch_t<bf16_t>(a, dev, st);
}

cudaError_t launch_topk_merge(const MergeArgs& a, cudaStream_t st) {
    const size_t smem = (size_t)a.n_slabs * a.top_k * (sizeof(float) + sizeof(int));
    topk_merge_kernel<<<a.R, 256, smem, st>>>(a);
    return cudaGetLastError();
}

}  // namespace fe

// The frozen LM head applied to every cascade output h_i (Sec. 2.1), fused with the
// softmax statistics and the top-k selection of Sec. 2.2, in one kernel: the [N*B, V]
// logits never reach global memory (unless the caller asks for them for a parity check).
//
// Grid: (n_slabs, ceil(R / BT)). Each CTA streams one vocabulary slab (a contiguous range
// of LM-head row groups) through the weight-streaming core (fe_stream.cuh) against the
// RMSNorm'd hidden rows z_r = RMSNorm(h_r; gamma_out) of its tile of BT rows, staged once
// in shared memory, so the LM head is read from HBM once for all N depths.
//  - Per chunk of row groups, the CTA writes the chunk's logits into a small shared-memory
//    buffer; warp b then folds row b's new logits into per-lane running (max, sum of exp)
//    of logit / T, tests them against the row's current k-th best (ties to the smaller
//    id) and inserts the few that pass into the row's sorted top-k list, one lane at a time.
//  - At the end of the slab, warp b reduces row b's per-lane statistics and writes the
//    slab's partial (top-k list and statistics).
//  - The last CTA to finish a row tile (an atomic counter per tile) merges all slabs'
//    partials: lse = M + log sum_j s_j e^(m_j - M); the global top-k is taken from the
//    candidates not below tau = max over slabs of the slab's k-th value (a slab holds k
//    candidates >= tau, so nothing below tau can be among the k best); probabilities are
//    exp(logit / T - lse).
#include <float.h>

#include "fe_kernels.h"
#include "fe_stream.cuh"

namespace fe {

constexpr int kMaxTopK = 32;
constexpr int kLmTile = 8;           // rows of z per tile (BT <= 8)
constexpr int kMergeCap = 256;       // survivors per row kept in shared memory for the merge

__device__ __forceinline__ bool better(float va, int ia, float vb, int ib) {
    return va > vb || (va == vb && ia < ib);
}

struct TopkState {
    int id[kLmTile][kMaxTopK];
    float val[kLmTile][kMaxTopK];
    int cnt[kLmTile];
    int last;
};

__device__ __forceinline__ void topk_insert(TopkState* st, int b, int k, float lg, int v) {
    const int c = st->cnt[b];
    int pos;
    if (c < k) {
        pos = c;
        st->cnt[b] = c + 1;
    } else if (better(lg, v, st->val[b][k - 1], st->id[b][k - 1])) {
        pos = k - 1;
    } else {
        return;
    }
    while (pos > 0 && better(lg, v, st->val[b][pos - 1], st->id[b][pos - 1])) {
        st->val[b][pos] = st->val[b][pos - 1];
        st->id[b][pos] = st->id[b][pos - 1];
        --pos;
    }
    st->val[b][pos] = lg;
    st->id[b][pos] = v;
}

template <int BT>
struct LmEpi {
    const LmHeadArgs* a;
    TopkState* st;
    float* cbuf;  // [BT][chunk_groups(BT) * 4] logits of the current chunk
    int b0, nb;
    float m = -INFINITY, sum = 0.f;  // this lane's running statistics of its warp's row
    __device__ void chunk(int cg0, int cg1, const float* red) {
        constexpr int CW = chunk_groups(BT) * kGroupRows;
        const int ng = cg1 - cg0;
        // 1. the chunk's logits, into the chunk buffer (and the optional full-logit dump)
        for (int q = threadIdx.x; q < ng * kGroupRows * BT; q += kStreamThreads) {
            const int gl = q / (kGroupRows * BT), r = (q / BT) % kGroupRows, b = q % BT;
            const int v = (cg0 + gl) * kGroupRows + r;
            if (b < nb && v < a->V) {
                const float lg = chunk_value<BT>(red, gl, r, b);
                cbuf[b * CW + gl * kGroupRows + r] = lg;
                if (a->dbg_logits) {
                    const int zr = b0 + b;
                    const int i = zr / a->B, sb = zr % a->B;
                    a->dbg_logits[((size_t)sb * a->N + i) * a->V + v] = lg;
                }
            }
        }
        __syncthreads();
        // 2. warp b folds row b's candidates into its statistics and top-k, in vocabulary order
        const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
        if (warp < nb) {
            const int k = a->top_k;
            const int n = min(ng * kGroupRows, a->V - cg0 * kGroupRows);
            const float* sb = cbuf + warp * CW;
            for (int base = 0; base < n; base += 32) {
                const int idx = base + lane;
                const bool valid = idx < n;
                const float lg = valid ? sb[idx] : -INFINITY;
                if (valid) {
                    const float lt = lg * a->inv_temp;
                    if (lt > m) {
                        sum = sum * expf(m - lt) + 1.0f;
                        m = lt;
                    } else {
                        sum += expf(lt - m);
                    }
                }
                const int v = cg0 * kGroupRows + idx;
                const bool pass =
                    valid && (st->cnt[warp] < k || better(lg, v, st->val[warp][k - 1], st->id[warp][k - 1]));
                unsigned mask = __ballot_sync(0xffffffffu, pass);
                while (mask) {
                    const int j = __ffs(mask) - 1;
                    mask &= mask - 1;
                    if (lane == j) topk_insert(st, warp, k, lg, v);
                    __syncwarp();
                }
            }
        }
    }
};

// Merge of all slabs' partials for one row zr, by one warp.
__device__ void merge_row(const LmHeadArgs& a, int zr, float* sv, int* si, int* scount, unsigned* taken) {
    const int lane = threadIdx.x & 31;
    const int k = a.top_k, ns = a.n_slabs;
    const float* pv = a.part_val + (size_t)zr * ns * k;
    const int* pi = a.part_id + (size_t)zr * ns * k;
    const float* pm = a.part_ms + (size_t)zr * ns * 2;
    // log-sum-exp of logit / T over the whole vocabulary
    float M = -INFINITY;
    for (int j = lane; j < ns; j += 32) M = fmaxf(M, __ldcg(pm + 2 * j));
    M = warp_max(M);
    float S = 0.f;
    for (int j = lane; j < ns; j += 32) {
        const float sj = __ldcg(pm + 2 * j + 1);
        if (sj > 0.f) S += sj * expf(__ldcg(pm + 2 * j) - M);
    }
    S = warp_sum(S);
    const float lse = M + logf(S);
    // tau: the largest k-th value over slabs
    float tau = -INFINITY;
    for (int j = lane; j < ns; j += 32) tau = fmaxf(tau, __ldcg(pv + (size_t)j * k + k - 1));
    tau = warp_max(tau);
    if (lane == 0) *scount = 0;
    __syncwarp();
    bool overflow = false;
    for (int j = lane; j < ns; j += 32) {
        for (int r = 0; r < k; ++r) {
            const float v = __ldcg(pv + (size_t)j * k + r);
            if (v < tau) break;  // slab lists are sorted, descending
            const int pos = atomicAdd(scount, 1);
            if (pos < kMergeCap) {
                sv[pos] = v;
                si[pos] = __ldcg(pi + (size_t)j * k + r);
            } else {
                overflow = true;
            }
        }
    }
    overflow = __any_sync(0xffffffffu, overflow);
    __syncwarp();
    const int n = overflow ? ns * k : min(*scount, kMergeCap);
    // k rounds of a warp arg-max (desc value, asc id); taken entries flagged in a bitmap
    for (int w = lane; w < (n + 31) / 32; w += 32) taken[w] = 0u;
    __syncwarp();
    const int i = zr / a.B, b = zr % a.B;
    const size_t ob = ((size_t)b * a.N + i) * k;
    for (int r = 0; r < k; ++r) {
        float bv = -INFINITY;
        int bi = INT_MAX, bp = -1;
        for (int j = lane; j < n; j += 32) {
            if (taken[j >> 5] & (1u << (j & 31))) continue;
            const float v = overflow ? __ldcg(pv + j) : sv[j];
            const int id = overflow ? __ldcg(pi + j) : si[j];
            if (bp < 0 || better(v, id, bv, bi)) { bv = v; bi = id; bp = j; }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
            const int op = __shfl_xor_sync(0xffffffffu, bp, o);
            if (op >= 0 && (bp < 0 || better(ov, oi, bv, bi))) { bv = ov; bi = oi; bp = op; }
        }
        if (lane == 0) {
            a.topk_id[ob + r] = bi;
            a.topk_logit[ob + r] = bv;
            a.topk_prob[ob + r] = expf(bv * a.inv_temp - lse);
            if (bp >= 0) taken[bp >> 5] |= 1u << (bp & 31);
        }
        __syncwarp();
    }
    if (lane == 0) a.lse[(size_t)b * a.N + i] = lse;
}

template <typename WT, int BT>
__global__ void __launch_bounds__(kStreamThreads, 1) lmhead_kernel(const LmHeadArgs a, int D) {
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ TopkState st;
    const int K = a.d;
    const int Kpad = (K + 3) & ~3;
    const int tile = blockIdx.y;
    const int b0 = tile * BT;
    const int nb = min(BT, a.R - b0);
    const int xrows = min(BT, a.R);
    StreamSmem s = carve_stream_smem(smem, D, xrows, Kpad, BT);
    __shared__ float cbuf[kLmTile * 32 * kGroupRows / 4 * 4];  // >= BT * chunk_groups(BT) * 4
    static_assert(BT * chunk_groups(BT) * kGroupRows <= kLmTile * 32 * kGroupRows / 4 * 4, "chunk buffer");
    if (threadIdx.x < kLmTile) st.cnt[threadIdx.x] = 0;

    const int GM = (a.V + kGroupRows - 1) / kGroupRows;
    const int sl = blockIdx.x;
    const int g0 = (int)(((int64_t)sl * GM) / gridDim.x);
    const int g1 = (int)(((int64_t)(sl + 1) * GM) / gridDim.x);

    ProParams pp{PRO_RMSNORM, a.hid, a.d, a.gamma, a.eps, nullptr, nullptr, 0, 0};
    stage_activations<WT>(pp, K, s.X, Kpad, b0, nb, a.status, s.red);
    __syncthreads();
    LmEpi<BT> ep{&a, &st, cbuf, b0, nb};
    stream_run<WT, BT>((const unsigned char*)a.W, K, g0, g1, s, D, Kpad, nb, a.status, ep);
    __syncthreads();

    // this slab's partial for each row of the tile (warp b <-> row b)
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    if (warp < nb) {
        const int zr = b0 + warp;
        const float m = warp_max(ep.m);
        float sum = ep.m == -INFINITY ? 0.f : ep.sum * expf(ep.m - m);
        sum = warp_sum(sum);
        const size_t base = (size_t)zr * a.n_slabs + sl;
        for (int j = lane; j < a.top_k; j += 32) {
            const bool ok = j < st.cnt[warp];
            a.part_id[base * a.top_k + j] = ok ? st.id[warp][j] : INT_MAX;
            a.part_val[base * a.top_k + j] = ok ? st.val[warp][j] : -INFINITY;
        }
        if (lane == 0) {
            a.part_ms[base * 2 + 0] = m;
            a.part_ms[base * 2 + 1] = sum;
        }
    }
    // the last slab CTA of this tile merges the tile's rows
    __threadfence();
    __syncthreads();
    if (t == 0) st.last = atomicAdd(&a.counters[tile], 1) == (int)gridDim.x - 1;
    __syncthreads();
    if (!st.last) return;
    __threadfence();
    // shared memory of the finished stream is reused: per warp kMergeCap values, ids, a
    // counter and a taken-bitmap sized for the overflow fallback
    const int bitmap_words = (a.n_slabs * a.top_k + 31) / 32;
    unsigned char* mbase = smem + (size_t)warp * (kMergeCap * 8 + 16 + bitmap_words * 4);
    float* sv = (float*)mbase;
    int* si = (int*)(sv + kMergeCap);
    int* scount = si + kMergeCap;
    unsigned* taken = (unsigned*)(scount + 4);
    if (warp < nb) merge_row(a, b0 + warp, sv, si, scount, taken);
    if (t == 0) a.counters[tile] = 0;
}

// ---- host side ----------------------------------------------------------------------------
namespace {
constexpr size_t kXBudget = 128 * 1024;
constexpr int kPreferredSlots = 2;
constexpr size_t kStaticReserve = sizeof(TopkState) + kLmTile * 32 * kGroupRows * sizeof(float) + 256;

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
    const size_t merge = (size_t)kLmTile * (kMergeCap * 8 + 16 + ((a.n_slabs * a.top_k + 31) / 32) * 4);
    int D = stream_slots(budget, stream_smem_bytes(0, xrows, Kpad, BT));
    D = D > kPreferredSlots ? kPreferredSlots : D;
    if (D < 1) return cudaErrorInvalidValue;
    size_t smem = stream_smem_bytes(D, xrows, Kpad, BT);
    if (smem < merge) smem = merge;
    if (smem > budget) return cudaErrorInvalidValue;
    dim3 grid(a.n_slabs, (a.R + BT - 1) / BT);
    lmhead_kernel<WT, BT><<<grid, kStreamThreads, smem, st>>>(a, D);
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

int lmhead_launches(int, int, const DeviceInfo&) { return 1; }

cudaError_t launch_lmhead(fe_dtype dt, const LmHeadArgs& a, const DeviceInfo& dev, cudaStream_t st) {
    if (a.top_k < 1 || a.top_k > kMaxTopK) return cudaErrorInvalidValue;
    return dt == FE_F32 ? launch_t<float>(a, dev, st) : launch_t<bf16_t>(a, dev, st);
}

}  // namespace fe

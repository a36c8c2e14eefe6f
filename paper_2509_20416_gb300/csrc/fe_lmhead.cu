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
#include "fe_sample.cuh"
#include "fe_stream.cuh"
#include "fe_tc.cuh"

namespace fe {

constexpr int kMaxTopK = 32;
constexpr int kLmTile = 8;           // rows of z per tile (BT <= 8)
constexpr int kMergeCap = 256;       // survivors per row kept in shared memory for the merge

__device__ __forceinline__ bool better(float va, int ia, float vb, int ib) {
    return va > vb || (va == vb && ia < ib);
}

// ---- exact top-k of a candidate list, by one warp ------------------------------------------
// A lone warp scanning shared memory pays a full load latency per dependent step, so the
// selection keeps the dependent steps few: one pass for each lane's best (value, id); the
// k-th largest of the 32 lane bests as a threshold T (k candidates are >= T, so the k best
// are too); one pass compacting the candidates >= T (ballot, no atomics); then k rounds of
// a warp arg-max over survivors held in registers. Order: larger value first, then smaller id.
constexpr int kSelPerLane = kMergeCap / 32;

__device__ __forceinline__ void warp_argmax(float& v, int& id) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, v, o);
        const int oi = __shfl_xor_sync(0xffffffffu, id, o);
        if (better(ov, oi, v, id)) { v = ov; id = oi; }
    }
}

// The k-th largest (1 <= k <= 32) of the warp's 32 values: a descending bitonic sort
// across the lanes, then lane k - 1's value.
__device__ __forceinline__ float warp_kth_largest(float x, int k) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            const float y = __shfl_xor_sync(0xffffffffu, x, stride);
            const bool desc = (lane & size) == 0, low = (lane & stride) == 0;
            x = (low == desc) ? fmaxf(x, y) : fminf(x, y);
        }
    }
    return __shfl_sync(0xffffffffu, x, k - 1);
}

// The value a candidate is ranked by: its logit (greedy top-k) ...
struct KeyLogit {
    __device__ __forceinline__ float operator()(float v, int) const { return v; }
    __device__ __forceinline__ bool may_reach(float, float) const { return true; }
};
// ... or its sampling key logit / T + G (stochastic drafting; fe_sample.cuh). may_reach is
// a cheap necessary condition for key >= th (G never exceeds kGumbelMax), so most
// candidates are ruled out without drawing their deviate.
struct KeySample {
    float inv_temp;
    unsigned long long seed;
    int row, V;
    __device__ __forceinline__ float operator()(float v, int id) const {
        return v == -INFINITY ? -INFINITY : sample_key(v, inv_temp, seed, row, V, id);
    }
    __device__ __forceinline__ bool may_reach(float v, float th) const { return fmaf(v, inv_temp, kGumbelMax) >= th; }
};

// Top-k of n candidates vals[j] with ids ids[j] (or id_base + j when ids is null), ranked
// by key(vals[j], id) (larger first, then smaller id), in shared memory; sv / si: this
// warp's scratch of kMergeCap entries. Calls out(q, key, id) on lane 0 for q < k; past the
// finite candidates the key is -inf and the id INT_MAX. With STATS, also returns (max, sum
// of exp(x - max)) of x = vals[j] * inv_temp over the finite candidates (all lanes). vals
// may be overwritten (a taken candidate becomes -inf), but only after out() reports it.
template <bool STATS, typename Key, typename Out>
__device__ __forceinline__ float2 warp_topk(float* vals, const int* ids, int id_base, int n, int k, float inv_temp,
                                            float* sv, int* si, const Key& key, Out&& out) {
    const int lane = threadIdx.x & 31;
    constexpr int U = 4;
    float lv = -INFINITY, m = -INFINITY, sum = 0.f;
    int li = INT_MAX;
    for (int j0 = 0; j0 < n; j0 += 32 * U) {
        float v[U];
        int id[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int j = j0 + 32 * u + lane;
            v[u] = j < n ? vals[j] : -INFINITY;
            id[u] = j < n ? (ids ? ids[j] : id_base + j) : INT_MAX;
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const float kv = key(v[u], id[u]);
            if (better(kv, id[u], lv, li)) { lv = kv; li = id[u]; }
            if (STATS && v[u] != -INFINITY) {
                const float x = v[u] * inv_temp;
                if (x > m) { sum = sum * expf(m - x) + 1.f; m = x; }
                else sum += expf(x - m);
            }
        }
    }
    if (STATS) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float om = __shfl_xor_sync(0xffffffffu, m, o), os = __shfl_xor_sync(0xffffffffu, sum, o);
            const float nm = fmaxf(m, om);
            sum = (m == -INFINITY ? 0.f : sum * expf(m - nm)) + (om == -INFINITY ? 0.f : os * expf(om - nm));
            m = nm;
        }
    }
    const float T = warp_kth_largest(lv, k);
    int cnt = 0;
    for (int j0 = 0; j0 < n; j0 += 32 * U) {
        float v[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int j = j0 + 32 * u + lane;
            v[u] = j < n ? vals[j] : -INFINITY;
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int j = j0 + 32 * u + lane;
            const int idj = j < n ? (ids ? ids[j] : id_base + j) : INT_MAX;
            float kv = -INFINITY;
            if (j < n && key.may_reach(v[u], T)) kv = key(v[u], idj);
            const bool p = j < n && kv >= T;
            const unsigned bal = __ballot_sync(0xffffffffu, p);
            const int pos = cnt + __popc(bal & ((1u << lane) - 1u));
            if (p && pos < kMergeCap) { sv[pos] = kv; si[pos] = idj; }
            cnt += __popc(bal);
        }
    }
    __syncwarp();
    if (cnt <= kMergeCap) {
        float rv[kSelPerLane];
        int ri[kSelPerLane];
        float bv = -INFINITY;
        int bi = INT_MAX;
#pragma unroll
        for (int q = 0; q < kSelPerLane; ++q) {
            const int j = lane + 32 * q;
            rv[q] = j < cnt ? sv[j] : -INFINITY;
            ri[q] = j < cnt ? si[j] : INT_MAX;
            if (better(rv[q], ri[q], bv, bi)) { bv = rv[q]; bi = ri[q]; }
        }
        for (int r = 0; r < k; ++r) {
            float wv = bv;
            int wi = bi;
            warp_argmax(wv, wi);
            if (lane == 0) out(r, wv, wv == -INFINITY ? INT_MAX : wi);
            if (wi == bi && wv == bv) {  // this lane held the winner: drop it, find its next best
                bv = -INFINITY;
                bi = INT_MAX;
#pragma unroll
                for (int q = 0; q < kSelPerLane; ++q) {
                    if (ri[q] == wi && rv[q] == wv) { rv[q] = -INFINITY; ri[q] = INT_MAX; }
                    if (better(rv[q], ri[q], bv, bi)) { bv = rv[q]; bi = ri[q]; }
                }
            }
        }
    } else {  // too many ties at T to hold: rounds over all candidates, marking the taken ones
        float bv = -INFINITY;
        int bi = INT_MAX, bp = -1;
        auto rescan = [&]() {
            bv = -INFINITY;
            bi = INT_MAX;
            bp = -1;
            for (int j = lane; j < n; j += 32) {
                const int id = ids ? ids[j] : id_base + j;
                const float v = key(vals[j], id);
                if (bp < 0 || better(v, id, bv, bi)) { bv = v; bi = id; bp = j; }
            }
        };
        rescan();
        for (int r = 0; r < k; ++r) {
            float wv = bv;
            int wi = bi;
            warp_argmax(wv, wi);
            if (lane == 0) out(r, wv, wv == -INFINITY ? INT_MAX : wi);
            if (bp >= 0 && wi == bi && wv == bv) {
                vals[bp] = -INFINITY;
                rescan();
            }
            __syncwarp();
        }
    }
    return make_float2(m, sum);
}

// A row's running top-k, sorted (larger value first, then smaller id). val is the value
// the row is ranked by (the logit, or the sampling key); lg the candidate's logit.
struct TopkState {
    int id[kLmTile][kMaxTopK];
    float val[kLmTile][kMaxTopK];
    float lg[kLmTile][kMaxTopK];
    int cnt[kLmTile];
    int last;
};

__device__ __forceinline__ void topk_insert(TopkState* st, int b, int k, float key, int v, float lg) {
    const int c = st->cnt[b];
    int pos;
    if (c < k) {
        pos = c;
        st->cnt[b] = c + 1;
    } else if (better(key, v, st->val[b][k - 1], st->id[b][k - 1])) {
        pos = k - 1;
    } else {
        return;
    }
    while (pos > 0 && better(key, v, st->val[b][pos - 1], st->id[b][pos - 1])) {
        st->val[b][pos] = st->val[b][pos - 1];
        st->id[b][pos] = st->id[b][pos - 1];
        st->lg[b][pos] = st->lg[b][pos - 1];
        --pos;
    }
    st->val[b][pos] = key;
    st->id[b][pos] = v;
    st->lg[b][pos] = lg;
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
            const int srow = sample_row(b0 + warp, a->B, a->N);
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
                // the value the row is ranked by: the logit, or (sampling) its key
                const bool full = st->cnt[warp] >= k;
                const float th = full ? st->val[warp][k - 1] : -INFINITY;
                float key = lg;
                if (a->sample && valid)
                    key = (!full || fmaf(lg, a->inv_temp, kGumbelMax) >= th)
                              ? sample_key(lg, a->inv_temp, a->seed, srow, a->V, v) : -INFINITY;
                const bool pass = valid && (!full || better(key, v, th, st->id[warp][k - 1]));
                unsigned mask = __ballot_sync(0xffffffffu, pass);
                while (mask) {
                    const int j = __ffs(mask) - 1;
                    mask &= mask - 1;
                    if (lane == j) topk_insert(st, warp, k, key, v, lg);
                    __syncwarp();
                }
            }
        }
    }
};

// Merge of all slabs' partials for rows [r0, r1), by every thread of the calling CTA.
// The rows' partials are first copied into shared memory (`buf`, the finished stream's
// ring) in one coalesced pass, in batches of rows that fit; then warp w merges row
// r0 + w, r0 + w + nwarps, ... of the batch from shared memory:
//   lse = M + log sum_j s_j e^(m_j - M) over the slabs' (max, sum of exp) pairs;
//   tau = the largest k-th value over slabs (a slab holds k candidates >= tau, so
//   nothing below tau can be among the k best); the candidates >= tau (all of them if
//   there are more than kMergeCap) go through k rounds of a warp arg-max (descending
//   value, ascending id); probabilities are exp(logit / T - lse).
// Stochastic drafting: the partials' values are sampling keys, and the k largest keys
// (in that order: the draw order) are the drawn candidates; their logits come from the
// partials' part_lg, and they are written ordered by logit (ties: smaller id) with each
// one's draw position in topk_rank.
constexpr size_t kMergeWarpBytes = (size_t)kMergeCap * 8 + 16 + 32 * 8;  // selection scratch + winners
constexpr int kMergeMaxSmem = 100 * 1024;  // dynamic shared memory of lmhead_merge_kernel, at most

__device__ void merge_rows(const LmHeadArgs& a, int r0, int r1, unsigned char* buf, size_t buf_bytes) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5, nw = blockDim.x >> 5;
    const int ns = a.n_slabs, k = a.top_k;
    const bool smp = a.sample != 0;
    const size_t per_row = (size_t)ns * ((smp ? 3 : 2) * k + 2) * 4;
    const size_t per_warp = kMergeWarpBytes;
    if (buf_bytes <= nw * per_warp + per_row) return;  // never happens: the host sizes the buffer
    const int batch = (int)((buf_bytes - nw * per_warp) / per_row);
    float* cand_v = (float*)(buf + nw * per_warp);  // [batch][ns * k]
    for (int rb = r0; rb < r1; rb += batch) {
        const int nr = min(batch, r1 - rb);
        float* bv_ = cand_v;
        int* bi_ = (int*)(cand_v + (size_t)nr * ns * k);
        float* bm_ = (float*)(bi_ + (size_t)nr * ns * k);
        float* bl_ = bm_ + (size_t)nr * ns * 2;  // sampling: the candidates' logits
        // 8 independent loads in flight per thread (a load-then-store loop would wait a full
        // L2 round trip per element)
        const size_t nc = (size_t)nr * ns * k, nm = (size_t)nr * ns * 2;
        for (size_t q0 = t; q0 < nc; q0 += 8 * (size_t)blockDim.x) {
            float v[8];
            int id[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const size_t q = q0 + u * (size_t)blockDim.x;
                v[u] = q < nc ? __ldcg(a.part_val + (size_t)rb * ns * k + q) : 0.f;
                id[u] = q < nc ? __ldcg(a.part_id + (size_t)rb * ns * k + q) : 0;
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const size_t q = q0 + u * (size_t)blockDim.x;
                if (q < nc) { bv_[q] = v[u]; bi_[q] = id[u]; }
            }
        }
        if (smp) {
            for (size_t q0 = t; q0 < nc; q0 += 8 * (size_t)blockDim.x) {
                float v[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const size_t q = q0 + u * (size_t)blockDim.x;
                    v[u] = q < nc ? __ldcg(a.part_lg + (size_t)rb * ns * k + q) : 0.f;
                }
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const size_t q = q0 + u * (size_t)blockDim.x;
                    if (q < nc) bl_[q] = v[u];
                }
            }
        }
        for (size_t q0 = t; q0 < nm; q0 += 8 * (size_t)blockDim.x) {
            float v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const size_t q = q0 + u * (size_t)blockDim.x;
                v[u] = q < nm ? __ldcg(a.part_ms + (size_t)rb * ns * 2 + q) : 0.f;
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const size_t q = q0 + u * (size_t)blockDim.x;
                if (q < nm) bm_[q] = v[u];
            }
        }
        __syncthreads();
        for (int rr = warp; rr < nr; rr += nw) {
            const int zr = rb + rr;
            float* pv = bv_ + (size_t)rr * ns * k;
            int* pi = bi_ + (size_t)rr * ns * k;
            const float* pm = bm_ + (size_t)rr * ns * 2;
            float* sv = (float*)(buf + warp * per_warp);
            int* si = (int*)(sv + kMergeCap);
            float M = -INFINITY;
            for (int j = lane; j < ns; j += 32) M = fmaxf(M, pm[2 * j]);
            M = warp_max(M);
            float S = 0.f;
            for (int j = lane; j < ns; j += 32)
                if (pm[2 * j + 1] > 0.f) S += pm[2 * j + 1] * expf(pm[2 * j] - M);
            S = warp_sum(S);
            const float lse = M + logf(S);
            const int i = zr / a.B, b = zr % a.B;
            const size_t ob = ((size_t)b * a.N + i) * k;
            if (!smp) {
                warp_topk<false>(pv, pi, 0, ns * k, k, a.inv_temp, sv, si, KeyLogit{}, [&](int q, float v, int id) {
                    a.topk_id[ob + q] = id;
                    a.topk_logit[ob + q] = v;
                    a.topk_prob[ob + q] = v == -INFINITY ? 0.f : expf(v * a.inv_temp - lse);
                    if (a.topk_rank) a.topk_rank[ob + q] = q;
                });
            } else {
                // the k largest keys, in draw order, into this warp's winner slots
                float* wl = (float*)(buf + warp * per_warp + (size_t)kMergeCap * 8 + 16);
                int* wi = (int*)(wl + 32);
                if (lane < 32) { wl[lane] = -INFINITY; wi[lane] = INT_MAX; }
                __syncwarp();
                warp_topk<false>(pv, pi, 0, ns * k, k, a.inv_temp, sv, si, KeyLogit{},
                                 [&](int q, float, int id) { wi[q] = id; });
                __syncwarp();
                // the winners' logits: every candidate id occurs once (the slabs are disjoint)
                const float* pl = bl_ + (size_t)rr * ns * k;
                for (int j = lane; j < ns * k; j += 32) {
                    const int idj = pi[j];
                    for (int q = 0; q < k; ++q)
                        if (wi[q] == idj && idj != INT_MAX) wl[q] = pl[j];
                }
                __syncwarp();
                const float lg = lane < k ? wl[lane] : -INFINITY;
                const int id = lane < k ? wi[lane] : INT_MAX;
                int pos = 0;  // this winner's place by (logit desc, id asc)
                for (int j = 0; j < k; ++j) {
                    const float oj = __shfl_sync(0xffffffffu, lg, j);
                    const int ij = __shfl_sync(0xffffffffu, id, j);
                    if (j != lane && better(oj, ij, lg, id)) ++pos;
                }
                if (lane < k) {
                    a.topk_id[ob + pos] = id;
                    a.topk_logit[ob + pos] = lg;
                    a.topk_prob[ob + pos] = lg == -INFINITY ? 0.f : expf(lg * a.inv_temp - lse);
                    if (a.topk_rank) a.topk_rank[ob + pos] = lane;
                }
                __syncwarp();
            }
            if (lane == 0) a.lse[(size_t)b * a.N + i] = lse;
        }
        __syncthreads();
    }
}

// shared memory merge_rows needs for at least one row at a time
__host__ __device__ inline size_t merge_smem_bytes(int nwarps, int n_slabs, int top_k, bool sample) {
    return (size_t)nwarps * kMergeWarpBytes + (size_t)n_slabs * ((sample ? 3 : 2) * top_k + 2) * 4 + 64;
}

template <typename WT, int BT>
__global__ void __launch_bounds__(kStreamThreads, 1) lmhead_kernel(const LmHeadArgs a, int D, size_t smem_bytes) {
    const LaunchStamp stamp(a.stamp);
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

    const int issued = stream_begin<WT>((const unsigned char*)a.W, K, g0, g1, s, D);
    griddep_launch_dependents();
    griddep_wait();
    ProParams pp{PRO_RMSNORM, a.hid, a.d, a.gamma, a.eps, nullptr, nullptr, 0, 0};
    stage_activations<WT>(pp, K, s.X, Kpad, b0, nb, a.status, s.red);
    __syncthreads();
    LmEpi<BT> ep{&a, &st, cbuf, b0, nb};
    stream_run<WT, BT>((const unsigned char*)a.W, K, g0, g1, s, D, Kpad, nb, a.status, ep, issued);
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
            if (a.sample) a.part_lg[base * a.top_k + j] = ok ? st.lg[warp][j] : -INFINITY;
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
    // the finished stream's shared memory holds the merge
    merge_rows(a, b0, b0 + nb, smem, smem_bytes);
    if (t == 0) a.counters[tile] = 0;
}

// ---- tensor-core LM head (bf16 storage, up to kMmaMaxRows hidden rows) --------------------
//
// z_r = RMSNorm(h_r; gamma_out) is split into z_hi = bf16(z) and z_lo = bf16(z - z_hi)
// (zprep_kernel), so W_lm z = W_lm z_hi + W_lm z_lo keeps ~16 more bits than one bf16
// rounding of z; both halves are the B operand [2 R_pad rows x d] of one M=128 x N=2 R_pad
// tcgen05.mma per 16 columns, accumulating in float32 in TMEM. Warp roles: warp 4 streams
// 16 KB weight blocks (and the matching B blocks) with bulk TMA copies into a ring of
// stages; warp 5 (one thread) issues the MMAs and commits each stage back to its producer;
// warps 0..3 read the double-buffered accumulator from TMEM (TMEM lane = vocabulary row)
// into a shared-memory buffer holding the slab's logits. After the slab, each of the 6
// warps takes rows: softmax statistics over the buffer, and the row's top-k by k rounds of
// a warp arg-max (each lane caches its best; only the round's winner rescans).
constexpr int kMmaMaxRows = 16;
constexpr int kMmaThreads = 6 * 32;
constexpr int kMmaMaxStages = 12;

// zb [d/64][N rows x 128 B] in the 128B-swizzled layout: rows [0, R_pad) hold z_hi, rows
// [R_pad, 2 R_pad) hold z_lo (N = 2 R_pad), or, without lo, z rounded to bf16 alone
// (N = R_pad); rows of padding (r >= R) are zero. One CTA per row r < R_pad;
// thread t owns the 16-byte chunks (8 values) t, t + 256, ... of the row, kept in
// registers between the sum of squares and the split (d <= kZprepMaxChunks * 8 * 256).
constexpr int kZprepMaxChunks = 8;

template <typename WT>
// hid is written by the previous kernel, which may still be running when this one starts
// (programmatic launch): it is read only after griddep_wait(), through L2 (ld.global.cg),
// and is deliberately not a __restrict__ pointer, whose loads the compiler may treat as
// invariant and move above the wait.
__global__ void __launch_bounds__(256) zprep_kernel(const float* hid, const WT* __restrict__ gamma, int R,
                                                    int R_pad, int d, float eps, uint16_t* zb, int with_lo,
                                                    unsigned long long* stamp_pair) {
    const LaunchStamp stamp(stamp_pair);
    static_assert(sizeof(WT) == 2, "the tensor-core LM head takes bf16 weights");
    const int r = blockIdx.x, t = threadIdx.x;
    const int N = with_lo ? 2 * R_pad : R_pad;
    const int nc = d / 8;  // 16-byte chunks of a bf16 row
    __shared__ float red[8];
    // the gains do not depend on the previous kernel
    uint4 gv[kZprepMaxChunks];
#pragma unroll
    for (int j = 0; j < kZprepMaxChunks; ++j) {
        const int c = t + 256 * j;
        gv[j] = c < nc ? reinterpret_cast<const uint4*>(gamma)[c] : make_uint4(0u, 0u, 0u, 0u);
    }
    griddep_launch_dependents();
    griddep_wait();
    float x[kZprepMaxChunks][8];
    float ss = 0.f;
#pragma unroll
    for (int j = 0; j < kZprepMaxChunks; ++j) {
        const int c = t + 256 * j;
        float4 a = make_float4(0.f, 0.f, 0.f, 0.f), b = a;
        if (r < R && c < nc) {
            const float4* hp = reinterpret_cast<const float4*>(hid + (size_t)r * d) + 2 * c;
            a = __ldcg(hp);
            b = __ldcg(hp + 1);
        }
        x[j][0] = a.x; x[j][1] = a.y; x[j][2] = a.z; x[j][3] = a.w;
        x[j][4] = b.x; x[j][5] = b.y; x[j][6] = b.z; x[j][7] = b.w;
#pragma unroll
        for (int e = 0; e < 8; ++e) ss = fmaf(x[j][e], x[j][e], ss);
    }
    ss = warp_sum(ss);
    if ((t & 31) == 0) red[t >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) tot += red[w];
    const float rs = r < R ? 1.0f / sqrtf(tot / (float)d + eps) : 0.f;
#pragma unroll
    for (int j = 0; j < kZprepMaxChunks; ++j) {
        const int c = t + 256 * j;
        if (c >= nc) continue;
        float g[8];
        Vec16<WT>::widen(gv[j], g);
        uint32_t hi[4], lo[4];
#pragma unroll
        for (int e = 0; e < 8; e += 2) {
            const float z0 = x[j][e] * rs * g[e], z1 = x[j][e + 1] * rs * g[e + 1];
            const uint16_t h0 = f32_to_bf16(z0), h1 = f32_to_bf16(z1);
            const uint16_t l0 = f32_to_bf16(z0 - bf16_to_f32(h0)), l1 = f32_to_bf16(z1 - bf16_to_f32(h1));
            hi[e / 2] = (uint32_t)h0 | ((uint32_t)h1 << 16);
            lo[e / 2] = (uint32_t)l0 | ((uint32_t)l1 << 16);
        }
        const int kb = c / 8, cc = c % 8;  // 64-column block, 16-byte chunk within it
        unsigned char* blk = (unsigned char*)zb + (size_t)kb * N * 128;
        *reinterpret_cast<uint4*>(blk + sw128_offset(r, cc)) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
        if (with_lo)
            *reinterpret_cast<uint4*>(blk + sw128_offset(R_pad + r, cc)) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
    }
}

__device__ __forceinline__ void st_release_gpu(int* p, int v) {
    asm volatile("st.release.gpu.global.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ int ld_acquire_gpu(const int* p) {
    int v;
    asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

struct MmaState {
    uint64_t full[kMmaMaxStages], empty[kMmaMaxStages], tfull[2], tempty[2], ebar;
    uint32_t tmem_base;
    int last, abort;
};

__global__ void __launch_bounds__(kMmaThreads, 1) lmhead_mma_kernel(const LmHeadArgs a, const uint16_t* zb, int R_pad,
                                                                    int S, int stage_bytes, uint32_t tmem_cols,
                                                                    int slab_cap) {
    const LaunchStamp stamp(a.stamp ? a.stamp + 2 : nullptr);
    extern __shared__ unsigned char dsm_raw[];
    __shared__ MmaState st;
    // 1024-byte aligned ring (the 128B swizzle pattern is a function of address bits 4..9),
    // then the slab's logits [R][slab_cap]
    unsigned char* ring = (unsigned char*)(((uintptr_t)dsm_raw + 1023) & ~(uintptr_t)1023);
    float* slab = (float*)(ring + (size_t)S * stage_bytes);
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int N = 2 * R_pad, R = a.R, k = a.top_k;
    const int nkb = a.d / 64;
    const int ntiles = (a.V + 127) / 128;
    // (tile, 64-column block) units in tile-major order, split evenly over the CTAs (whole
    // tiles without the split buffers). gridDim.x <= ntiles, so a CTA covers at least nkb
    // units and a tile is shared by two CTAs at most: a CTA whose range starts inside a
    // tile computes that tile's second part first and leaves it in split_part (the tile
    // belongs to the previous CTA, which streams the first part last); a CTA whose range
    // ends inside a tile owns it and adds the next CTA's part before the epilogue.
    const int64_t U = (int64_t)ntiles * nkb;
    const bool stream_k = a.split_part != nullptr;
    auto ubegin = [&](int c) -> int64_t {
        return stream_k ? (int64_t)c * U / gridDim.x : ((int64_t)c * ntiles / gridDim.x) * nkb;
    };
    const int64_t u0 = ubegin(blockIdx.x), u1 = ubegin(blockIdx.x + 1);
    const int tf = (int)(u0 / nkb), tl = (int)((u1 - 1) / nkb);  // first and last tile touched
    const bool head_part = u0 % nkb != 0;  // the first piece is another CTA's tile
    const bool tail_part = u1 % nkb != 0;  // the last tile's second part comes from CTA + 1
    const int t0 = head_part ? tf + 1 : tf, t1 = tl + 1;  // the tiles of this slab

    if (t == 0) {
        for (int i = 0; i < S; ++i) {
            mbar_init(&st.full[i], 1);
            mbar_init(&st.empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&st.tfull[i], 1);
            mbar_init(&st.tempty[i], 4);
        }
        mbar_init(&st.ebar, 4);  // the four epilogue warps (split-tile hand-offs)
        st.abort = 0;
        mbar_fence_init();
    }
    if (warp == 0) tc_alloc(&st.tmem_base, tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = st.tmem_base;

    griddep_launch_dependents();
    if (warp == 4) {  // ---- TMA producer
        if (lane == 0) {
            // the first stages' weight blocks do not depend on the previous kernel (zprep);
            // unit u's weight block sits at u * 16 KB (tile-major packing)
            const int total = (int)(u1 - u0);
            const int pre = min(S, total);
            const uint64_t wpol = l2_evict_first();  // the LM head is read once per draft
            for (int it = 0; it < pre; ++it) {
                mbar_arrive_expect_tx(&st.full[it], 16384u + (uint32_t)N * 128u);
                bulk_g2s_hint(ring + (size_t)it * stage_bytes, (const unsigned char*)a.W + (size_t)(u0 + it) * 16384,
                              16384, &st.full[it], wpol);
            }
            griddep_wait();
            // ring positions advance by counters, not by division (a single thread on the
            // stream's critical path)
            int kb = (int)(u0 % nkb);  // z block of the next copy: (u0 + it) % nkb
            for (int it = 0; it < pre; ++it) {
                bulk_g2s(ring + (size_t)it * stage_bytes + 16384, (const unsigned char*)zb + (size_t)kb * N * 128,
                         (uint32_t)N * 128, &st.full[it]);
                if (++kb == nkb) kb = 0;
            }
            // iteration it >= S reuses slot it % S after the MMAs of iteration it - S: completion
            // (it - S) / S of empty[slot]
            int slot = 0;
            uint32_t pe = 0;
            for (int it = pre; it < total; ++it) {
                if (!mbar_wait_abortable(&st.empty[slot], pe, a.status, &st.abort)) break;
                unsigned char* dst = ring + (size_t)slot * stage_bytes;
                mbar_arrive_expect_tx(&st.full[slot], 16384u + (uint32_t)N * 128u);
                bulk_g2s_hint(dst, (const unsigned char*)a.W + (size_t)(u0 + it) * 16384, 16384, &st.full[slot], wpol);
                bulk_g2s(dst + 16384, (const unsigned char*)zb + (size_t)kb * N * 128, (uint32_t)N * 128,
                         &st.full[slot]);
                if (++kb == nkb) kb = 0;
                if (++slot == S) { slot = 0; pe ^= 1u; }
            }
        }
    } else if (warp == 5) {  // ---- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, N);
            int slot = 0;
            uint32_t pf = 0;  // phase bit of full[slot]
            int64_t u = u0;
            for (int tile = tf, j = 0; tile <= tl; ++tile, ++j) {  // one piece (accumulator) per tile
                const int buf = j & 1;
                if (!mbar_wait_abortable(&st.tempty[buf], ((uint32_t)(j >> 1) & 1u) ^ 1u, a.status, &st.abort)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem + (uint32_t)(buf * N);
                const int64_t ue = min(u1, (int64_t)(tile + 1) * nkb);
                bool ok = true;
                for (bool first = true; u < ue; ++u, first = false) {
                    if (!mbar_wait_abortable(&st.full[slot], pf, a.status, &st.abort)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_u32(ring + (size_t)slot * stage_bytes);
                    const uint64_t adesc = sw128_desc(sa), bdesc = sw128_desc(sa + 16384);
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)  // K = 16 per MMA: +32 bytes inside the swizzled rows
                        tc_mma(d_tmem, adesc + 2 * kk, bdesc + 2 * kk, idesc, (!first || kk) ? 1u : 0u);
                    tc_commit(&st.empty[slot]);
                    if (++slot == S) { slot = 0; pf ^= 1u; }
                }
                if (!ok) break;
                tc_commit(&st.tfull[buf]);
            }
        }
    } else {  // ---- epilogue warps 0..3: TMEM lanes 32 w .. 32 w + 31 = vocabulary rows of the tile
        const int tr = warp * 32 + lane;  // row of the tile
        uint32_t eb = 0;                  // phases of st.ebar passed
        auto epi_sync = [&]() -> bool {   // the four epilogue warps; bounded like every wait
            __syncwarp();
            if (lane == 0) mbar_arrive(&st.ebar);
            return mbar_wait_abortable(&st.ebar, (eb++) & 1u, a.status, &st.abort);
        };
        for (int tile = tf, j = 0; tile <= tl; ++tile, ++j) {
            const int buf = j & 1;
            if (!mbar_wait_abortable(&st.tfull[buf], (uint32_t)(j >> 1) & 1u, a.status, &st.abort, 20000)) break;
            tc_fence_after();
            float acc[2 * kMmaMaxRows];
            const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)(buf * N);
            for (int c = 0; c < N; c += 16) tc_ld16(taddr + c, acc + c);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&st.tempty[buf]);
            if (tile == tf && head_part) {  // the previous CTA's tile: leave this part for it
                float* p = a.split_part + ((size_t)blockIdx.x * 128 + tr) * R_pad;
#pragma unroll
                for (int r = 0; r < kMmaMaxRows; r += 4)
                    if (r < R_pad)
                        *reinterpret_cast<float4*>(p + r) =
                            make_float4(acc[r] + acc[R_pad + r], acc[r + 1] + acc[R_pad + r + 1],
                                        acc[r + 2] + acc[R_pad + r + 2], acc[r + 3] + acc[R_pad + r + 3]);
                if (!epi_sync()) break;  // the four warps' parts are written
                if (t == 0) {
                    __threadfence();
                    st_release_gpu(a.split_flag + blockIdx.x, 1);
                }
                continue;
            }
            float add[kMmaMaxRows];  // the next CTA's part of this tile, when it has one
#pragma unroll
            for (int r = 0; r < kMmaMaxRows; ++r) add[r] = 0.f;
            if (tile == tl && tail_part) {
                if (t == 0) {  // bounded wait for CTA + 1 (resident: it launched before this one could end)
                    const uint64_t t_0 = globaltimer_ns();
                    while (ld_acquire_gpu(a.split_flag + blockIdx.x + 1) == 0) {
                        if ((int64_t)(globaltimer_ns() - t_0) > kWaitBudgetNs) {
                            atomicOr(a.status, ST_TIMEOUT);
                            break;
                        }
                        __nanosleep(64);
                    }
                    // (lmhead_merge_kernel clears the flags once every CTA has exited)
                }
                if (!epi_sync()) break;
                const float* p = a.split_part + ((size_t)(blockIdx.x + 1) * 128 + tr) * R_pad;
#pragma unroll
                for (int r = 0; r < kMmaMaxRows; r += 4)
                    if (r < R_pad) {
                        const float4 q = __ldcg(reinterpret_cast<const float4*>(p + r));
                        add[r] = q.x; add[r + 1] = q.y; add[r + 2] = q.z; add[r + 3] = q.w;
                    }
            }
            const int row = (tile - t0) * 128 + tr;  // row of the slab
            const int v = tile * 128 + tr;
            for (int r = 0; r < R; ++r) {
                const float lg = (acc[r] + acc[R_pad + r]) + add[r];
                slab[(size_t)r * slab_cap + row] = v < a.V ? lg : -INFINITY;
                if (v < a.V && a.dbg_logits) {
                    const int i = r / a.B, sb = r % a.B;
                    a.dbg_logits[((size_t)sb * a.N + i) * a.V + v] = lg;
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tc_dealloc(tmem, tmem_cols);

    // ---- this slab's partial per row (warp w: rows w, w + 6, ..): statistics and top-k;
    // the ring is free now and holds each warp's selection scratch
    {
        const int n = (t1 - t0) * 128;
        const int first = t0 * 128;
        float* sv = (float*)(ring + (size_t)warp * kMergeCap * 8);
        int* si = (int*)(sv + kMergeCap);
        for (int r = warp; r < R; r += kMmaThreads / 32) {
            const size_t base = (size_t)r * a.n_slabs + blockIdx.x;
            float* row = slab + (size_t)r * slab_cap;
            auto out = [&](int q, float v, int id) {
                a.part_id[base * k + q] = id;
                a.part_val[base * k + q] = v;
                if (a.sample) a.part_lg[base * k + q] = id == INT_MAX ? -INFINITY : row[id - first];
            };
            const float2 ms =
                a.sample ? warp_topk<true>(row, nullptr, first, n, k, a.inv_temp, sv, si,
                                           KeySample{a.inv_temp, a.seed, sample_row(r, a.B, a.N), a.V}, out)
                         : warp_topk<true>(row, nullptr, first, n, k, a.inv_temp, sv, si, KeyLogit{}, out);
            if (lane == 0) {
                a.part_ms[base * 2 + 0] = ms.x;
                a.part_ms[base * 2 + 1] = ms.y;
            }
        }
    }
    // (lmhead_merge_kernel, one CTA per row, merges the slabs)
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
    const size_t merge = merge_smem_bytes(kStreamThreads / 32, a.n_slabs, a.top_k, a.sample != 0);
    int D = stream_slots(budget, stream_smem_bytes(0, xrows, Kpad, BT));
    D = D > kPreferredSlots ? kPreferredSlots : D;
    if (D < 1) return cudaErrorInvalidValue;
    size_t smem = stream_smem_bytes(D, xrows, Kpad, BT);
    if (smem < merge) smem = merge;
    if (smem > budget) return cudaErrorInvalidValue;
    dim3 grid(a.n_slabs, (a.R + BT - 1) / BT);
    return launch_k(lmhead_kernel<WT, BT>, grid, dim3(kStreamThreads), smem, st, a.pdl, a, D, smem);
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


bool lmhead_mma_ok(const LmHeadArgs& a) {
    return a.R <= kMmaMaxRows && a.d % 64 == 0 && a.d <= kZprepMaxChunks * 8 * 256 && a.top_k <= kMaxTopK;
}

size_t lmhead_mma_zb_bytes(int R, int d) {
    const int R_pad = (R + 7) / 8 * 8;
    return (size_t)2 * R_pad * d * 2;
}

__global__ void __launch_bounds__(128) lmhead_merge_kernel(const LmHeadArgs a, size_t smem_bytes);

cudaError_t lmhead_mma_prepare(const DeviceInfo& dev) {
    const cudaError_t e = cudaFuncSetAttribute(lmhead_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               dev.max_smem_optin - (int)sizeof(MmaState) - 256);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(lmhead_merge_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kMergeMaxSmem);
}

cudaError_t launch_lmhead_mma(const LmHeadArgs& a, uint16_t* zb, const DeviceInfo& dev, cudaStream_t st,
                              cudaEvent_t after_prep, cudaEvent_t after_main) {
    if (!lmhead_mma_ok(a) || (reinterpret_cast<uintptr_t>(a.hid) & 15)) return cudaErrorInvalidValue;
    const int R_pad = (a.R + 7) / 8 * 8;
    const int N = 2 * R_pad;
    cudaError_t e = launch_k(zprep_kernel<bf16_t>, dim3(R_pad), dim3(256), 0, st, a.pdl, a.hid,
                             (const bf16_t*)a.gamma, a.R, R_pad, a.d, a.eps, zb, 1, a.stamp);
    if (e != cudaSuccess) return e;
    if (after_prep && (e = cudaEventRecord(after_prep, st)) != cudaSuccess) return e;
    const int stage_bytes = (16384 + N * 128 + 1023) / 1024 * 1024;
    const size_t budget = (size_t)dev.max_smem_optin - sizeof(MmaState) - 256;
    const int ntiles = (a.V + 127) / 128;
    if (a.n_slabs < 1 || a.n_slabs > ntiles || (a.split_part && !a.split_flag)) return cudaErrorInvalidValue;
    // rows of the largest slab: whole tiles, or (split units) the tiles a range of
    // ceil(U / n_slabs) units ends in, plus one
    const int nkb = a.d / 64;
    const int64_t U = (int64_t)ntiles * nkb;
    const int slab_cap = (a.split_part ? (int)(((U + a.n_slabs - 1) / a.n_slabs + nkb - 1) / nkb) + 1
                                       : (ntiles + a.n_slabs - 1) / a.n_slabs) * 128;
    const size_t slab_bytes = (size_t)a.R * slab_cap * sizeof(float);
    if (budget < 1024 + slab_bytes + 2 * (size_t)stage_bytes) return cudaErrorInvalidValue;
    int S = (int)((budget - 1024 - slab_bytes) / stage_bytes);
    S = S > kMmaMaxStages ? kMmaMaxStages : S;
    if (S < 2) return cudaErrorInvalidValue;
    const size_t msmem = merge_smem_bytes(4, a.n_slabs, a.top_k, a.sample != 0);
    if (msmem > kMergeMaxSmem) return cudaErrorInvalidValue;
    const size_t smem = 1024 + (size_t)S * stage_bytes + slab_bytes;
    uint32_t cols = 32;
    while (cols < (uint32_t)(2 * N)) cols <<= 1;
    e = launch_k(lmhead_mma_kernel, dim3(a.n_slabs), dim3(kMmaThreads), smem, st, a.pdl, a, (const uint16_t*)zb,
                 R_pad, S, stage_bytes, cols, slab_cap);
    if (e != cudaSuccess) return e;
    if (after_main && (e = cudaEventRecord(after_main, st)) != cudaSuccess) return e;
    // one CTA per row merges the slabs (a last-CTA merge would hold every row on one SM)
    return launch_k(lmhead_merge_kernel, dim3(a.R), dim3(128), msmem, st, a.pdl, a, msmem);
}


// ==== wide tensor-core LM head: up to 256 hidden rows (batched serving) =====================
// At B sequences x N depths the LM head sees R = N * B rows (192 at B = 32, N = 6). The
// 16-row kernel above keeps every slab logit in shared memory and splits z into bf16
// hi + lo; neither holds at this R. Here:
//   - z is rounded once to bf16 (N = R_pad MMA columns, R_pad <= 256); every product is
//     accumulated in float32. The logit error this leaves is of the order of
//     |W_v| |z| 2^-9 / sqrt(3), a few 1e-3 at d = 4096 with weights ~ N(0, 0.02^2).
//   - The weight blocks and the z blocks travel in two rings of their own: a weight block
//     comes from HBM and a z block from L2 (every CTA reads all of z once per tile), so the
//     weight ring runs as many stages ahead as shared memory allows (the bytes in flight
//     that keep HBM busy) while a few stages cover the z block's L2 latency.
//   - TMEM holds two R_pad-column accumulators, so the epilogue of tile j overlaps the
//     MMAs of tile j + 1.
//   - Eight epilogue warps, one hidden row per thread: warps 4 g .. 4 g + 3 own rows
//     128 g .. 128 g + 127. A tile's accumulator has the vocabulary entries as TMEM lanes
//     and the rows as columns, so each row group transposes it through shared memory in
//     rounds of kWideRound entries x 128 rows (the warps whose lanes hold those entries copy
//     them; a small round leaves shared memory to the weight ring). A thread then reads its
//     row's logits in batches of 32 held in registers: the
//     batch max, a mask of the entries that reach the running top-k list's k-th value (only
//     those run through the list's insertion network), the sum of exp against the batch
//     max (base 2, on the hardware's 2^x) and one rescale of the running (max, sum). The
//     list is sorted in registers (larger value first, ties to the smaller id); there is no
//     cross-thread reduction. At the end of the slab each thread writes its row's partial.
//   - lmhead_merge_kernel (one CTA per row) then merges the slabs as merge_rows does.
constexpr int kWideKMax = 16;     // top_k limit of this kernel (a sorted list in registers)
constexpr int kWideRowsMax = 256;
constexpr int kWideLoRows = 16;   // up to this many (padded) rows z is split into bf16 hi + lo
constexpr int kWideGroup = 128;   // rows of a row group (one per thread of its four warps)
constexpr int kWideRound = 32;    // vocabulary entries staged per transpose round (a quarter of a tile)
constexpr int kWideRoundWarps = kWideRound / 32;  // the warps that stage one round
constexpr int kWideTileStride = kWideGroup + 1;  // floats per staged vocabulary entry (no bank conflicts)
constexpr int kWideMaxW = 12;     // weight-ring stages (16 KB each)
constexpr int kWideMaxZ = 3;      // z-ring stages at most (R_pad x 128 B each)
constexpr int kWideThreads = 10 * 32;  // 8 epilogue warps, 1 producer warp, 1 MMA warp

struct WideState {
    uint64_t wfull[kWideMaxW], zfull[kWideMaxW], done[kWideMaxW], tfull[2], tempty[2],
        ebar[2][2];
    uint32_t tmem_base;
    int abort;
};

// insertion into the sorted list as a branch-free compare-exchange down the list
template <int KM>
__device__ __forceinline__ void wide_insert(float (&tv)[KM], int (&ti)[KM], int k, float x, int id) {
#pragma unroll
    for (int q = 0; q < KM; ++q) {
        const bool sw = q < k && better(x, id, tv[q], ti[q]);
        const float ov = tv[q];
        const int oi = ti[q];
        tv[q] = sw ? x : ov;
        ti[q] = sw ? id : oi;
        x = sw ? ov : x;
        id = sw ? oi : id;
    }
}

// the same, carrying each entry's logit beside its key (stochastic drafting)
template <int KM>
__device__ __forceinline__ void wide_insert(float (&tv)[KM], int (&ti)[KM], float (&tl)[KM], int k, float x, int id,
                                            float lx) {
#pragma unroll
    for (int q = 0; q < KM; ++q) {
        const bool sw = q < k && better(x, id, tv[q], ti[q]);
        const float ov = tv[q], ol = tl[q];
        const int oi = ti[q];
        tv[q] = sw ? x : ov;
        ti[q] = sw ? id : oi;
        tl[q] = sw ? lx : ol;
        x = sw ? ov : x;
        id = sw ? oi : id;
        lx = sw ? ol : lx;
    }
}

// Stochastic drafting: the smallest 23-bit deviate code m (U = (m + 1/2) / 2^23) with which
// a logit at most M can still give a key logit / T + G >= th, minus a safety margin. With
// c = th - M / T, G >= c needs U >= exp(-exp(-c)); the bound is taken from 1 - U <=
// -expm1(-exp(-(c - 1e-3))), which errs towards admitting more (1e-3 in c moves the bound
// by a relative 1e-3, far above the functions' rounding). A tile's entries with a smaller
// code cannot enter the list and skip their logarithms.
__device__ __forceinline__ uint32_t sample_code_floor(float th, float M_scaled) {
    if (th == -INFINITY) return 0u;
    const float c = th - M_scaled - 1e-3f;
    if (c <= -30.f) return 0u;
    const float tail = -expm1f(-expf(-c));                    // an upper bound on 1 - U
    const float f = floorf(8388607.5f - tail * 8388608.0f) - 1.0f;
    return f <= 0.f ? 0u : (uint32_t)f;
}

// A running (softmax statistics, top-k) state of one hidden row: the first k of the KM
// entries form the sorted list (larger value first, ties to the smaller id; the rest stay
// -inf); (m, s) are the max and sum of exp of logit / T so far.
template <int KM>
struct WideRow {
    float v[KM];  // the values the list is ranked by: logits, or sampling keys
    int i[KM];
    float l[KM];  // sampling only: the entries' logits
    float m, s;
    __device__ __forceinline__ void init() {
#pragma unroll
        for (int q = 0; q < KM; ++q) { v[q] = -INFINITY; i[q] = INT_MAX; l[q] = -INFINITY; }
        m = -INFINITY;
        s = 0.f;
    }
};

// One batch of up to 32 of a round's entries (round entries e0 .. e0 + 31, vocabulary ids
// id0 + e) for the thread's row state w (inside lmhead_wide_kernel's epilogue).
// col[e * kWideTileStride] is the row's logit of round entry e; nv entries of the round are
// valid. Expanded textually: written as a function taking the state by reference, the
// compiler keeps the state in local memory.
#define FE_WIDE_BATCH(e0)                                                                          \
    do {                                                                                           \
        if ((e0) >= nv) break;                                                                     \
        float x[32];                                                                               \
        _Pragma("unroll") for (int u = 0; u < 32; ++u)                                             \
            x[u] = (e0) + u < nv ? col[(size_t)((e0) + u) * kWideTileStride] : -INFINITY;          \
        float m4[4] = {x[0], x[1], x[2], x[3]};                                                    \
        _Pragma("unroll") for (int u = 4; u < 32; ++u) m4[u & 3] = fmaxf(m4[u & 3], x[u]);         \
        const float M = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));                           \
        /* the list's k-th value (-inf until k entries are in): its smallest of the first k */    \
        float th = w.v[0];                                                                         \
        _Pragma("unroll") for (int q = 1; q < KM; ++q) th = q < k ? fminf(th, w.v[q]) : th;        \
        uint32_t bits = 0u; /* entries that can enter the list */                                  \
        if (!SMP) {                                                                                \
            _Pragma("unroll") for (int u = 0; u < 32; ++u)                                         \
                bits |= ((e0) + u < nv && x[u] >= th ? 1u : 0u) << u;                              \
        } else { /* keys: a deviate code per entry, logarithms only past the code floor */         \
            const int srow = sample_row(r, a.B, a.N);                                              \
            const uint32_t mlo = sample_code_floor(th, M * a.inv_temp);                            \
            _Pragma("unroll") for (int u = 0; u < 32; ++u) {                                       \
                if ((e0) + u < nv) {                                                               \
                    const uint32_t m23 = (uint32_t)(splitmix64_at(a.seed,                          \
                        sample_counter(srow, a.V, id0 + (e0) + u)) >> 41);                         \
                    if (m23 >= mlo) {                                                              \
                        const float key = fmaf(x[u], a.inv_temp,                                   \
                            gumbel_of(((float)m23 + 0.5f) * (1.0f / 8388608.0f)));                 \
                        bits |= (key >= th ? 1u : 0u) << u;                                        \
                    }                                                                              \
                }                                                                                  \
            }                                                                                      \
        }                                                                                          \
        while (bits) {                                                                             \
            const int e = (e0) + __ffs(bits) - 1;                                                  \
            bits &= bits - 1u;                                                                     \
            const float xe = col[(size_t)e * kWideTileStride];                                     \
            if (SMP)                                                                               \
                wide_insert(w.v, w.i, w.l, k, sample_key(xe, a.inv_temp, a.seed,                   \
                            sample_row(r, a.B, a.N), a.V, id0 + e), id0 + e, xe);                  \
            else                                                                                   \
                wide_insert(w.v, w.i, k, xe, id0 + e);                                             \
        }                                                                                          \
        /* sum of exp(x / T - M / T) in base 2: 2^(x c - M c), c = log2(e) / T */                 \
        const float c2 = a.inv_temp * kLog2e, mc = M * c2;                                         \
        float s4[4] = {0.f, 0.f, 0.f, 0.f};                                                        \
        _Pragma("unroll") for (int u = 0; u < 32; ++u) s4[u & 3] += ex2_approx(fmaf(x[u], c2, -mc)); \
        const float S = (s4[0] + s4[1]) + (s4[2] + s4[3]);                                         \
        const float Mt = M * a.inv_temp;                                                           \
        const float nm = fmaxf(w.m, Mt);                                                           \
        w.s = (w.m == -INFINITY ? 0.f : w.s * ex2_approx((w.m - nm) * kLog2e)) + S * ex2_approx((Mt - nm) * kLog2e); \
        w.m = nm;                                                                                  \
    } while (0)

template <int KM, bool SMP, bool LO>
__global__ void __launch_bounds__(kWideThreads, 1) lmhead_wide_kernel(const LmHeadArgs a, const uint16_t* zb, int R_pad,
                                                                      int SW, int SZ, uint32_t tmem_cols) {
    const LaunchStamp stamp(a.stamp ? a.stamp + 2 : nullptr);
    extern __shared__ unsigned char dsm_raw[];
    __shared__ WideState st;
    // LO: z as bf16 hi (rows [0, R_pad)) + lo (rows [R_pad, 2 R_pad)) parts, NZ = 2 R_pad MMA
    // columns, the epilogue adding the two accumulator columns of a row; else z in bf16 alone
    const int NZ = LO ? 2 * R_pad : R_pad;
    const uint32_t zbytes = (uint32_t)NZ * 128u;
    // [weight ring: SW x 16 KB][z ring: SZ x zbytes][transpose buffers: one per row group]
    unsigned char* wring = (unsigned char*)(((uintptr_t)dsm_raw + 1023) & ~(uintptr_t)1023);
    unsigned char* zring = wring + (size_t)SW * 16384;
    float* tbuf = (float*)(zring + (size_t)SZ * zbytes);  // [group][64 vocab][kWideTileStride]
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int R = a.R, k = a.top_k;
    const int nkb = a.d / 64;
    const int ntiles = (a.V + 127) / 128;
    const int t0 = (int)(((int64_t)blockIdx.x * ntiles) / gridDim.x);
    const int t1 = (int)(((int64_t)(blockIdx.x + 1) * ntiles) / gridDim.x);
    const int ngroups = (R_pad + kWideGroup - 1) / kWideGroup;

    if (t == 0) {
        for (int i = 0; i < SW; ++i) {
            mbar_init(&st.wfull[i], 1);
            mbar_init(&st.zfull[i], 1);
            mbar_init(&st.done[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&st.tfull[i], 1);
            mbar_init(&st.tempty[i], 4 * ngroups);  // every warp of a present row group
            mbar_init(&st.ebar[i][0], 4);
            mbar_init(&st.ebar[i][1], 4);
        }
        st.abort = 0;
        mbar_fence_init();
    }
    if (warp == 0) tc_alloc(&st.tmem_base, tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = st.tmem_base;
    griddep_launch_dependents();

    // Ring positions advance by counters (slot, phase bit), not by division: the producer and
    // the MMA issuer are single threads whose every instruction is on the stream's critical
    // path.
    if (warp == 8) {  // ---- TMA producer
        if (lane == 0) {
            const int total = (t1 - t0) * nkb;  // iteration it: weight block t0 * nkb + it, z block it % nkb
            const unsigned char* Wsrc = (const unsigned char*)a.W + (size_t)t0 * nkb * 16384;
            const unsigned char* Zsrc = (const unsigned char*)zb;
            const int prew = min(SW, total), prez = min(SZ, total);
            const uint64_t wpol = l2_evict_first();  // the LM head is read once per draft
            // the weights do not depend on earlier kernels: the first stages go out at once
            for (int it = 0; it < prew; ++it) {
                mbar_arrive_expect_tx(&st.wfull[it], 16384u);
                bulk_g2s_hint(wring + (size_t)it * 16384, Wsrc + (size_t)it * 16384, 16384, &st.wfull[it], wpol);
            }
            griddep_wait();
            int kz = 0;  // z block of the next z copy
            for (int it = 0; it < prez; ++it) {
                mbar_arrive_expect_tx(&st.zfull[it], zbytes);
                bulk_g2s(zring + (size_t)it * zbytes, Zsrc + (size_t)kz * zbytes, zbytes, &st.zfull[it]);
                if (++kz == nkb) kz = 0;
            }
            // once the MMAs of iteration c are done (done[c % SW]), its z slot takes iteration
            // c + SZ and its weight slot iteration c + SW
            int cw = 0, cz = 0;  // c % SW, c % SZ
            uint32_t pd = 0;     // phase bit of done[cw]
            for (int c = 0; c + SZ < total; ++c) {
                if (!mbar_wait_abortable(&st.done[cw], pd, a.status, &st.abort)) break;
                mbar_arrive_expect_tx(&st.zfull[cz], zbytes);
                bulk_g2s(zring + (size_t)cz * zbytes, Zsrc + (size_t)kz * zbytes, zbytes, &st.zfull[cz]);
                if (++kz == nkb) kz = 0;
                if (c + SW < total) {
                    mbar_arrive_expect_tx(&st.wfull[cw], 16384u);
                    bulk_g2s_hint(wring + (size_t)cw * 16384, Wsrc + (size_t)(c + SW) * 16384, 16384, &st.wfull[cw], wpol);
                }
                if (++cz == SZ) cz = 0;
                if (++cw == SW) { cw = 0; pd ^= 1u; }
            }
        }
    } else if (warp == 9) {  // ---- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, NZ);
            int sw = 0, sz = 0;          // it % SW, it % SZ
            uint32_t pw = 0, pz = 0;     // phase bits of wfull[sw], zfull[sz]
            for (int tile = t0, j = 0; tile < t1; ++tile, ++j) {
                const int buf = j & 1;
                if (!mbar_wait_abortable(&st.tempty[buf], ((uint32_t)(j >> 1) & 1u) ^ 1u, a.status, &st.abort)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem + (uint32_t)(buf * NZ);
                bool ok = true;
                for (int kb = 0; kb < nkb; ++kb) {
                    if (!mbar_wait_abortable(&st.wfull[sw], pw, a.status, &st.abort) ||
                        !mbar_wait_abortable(&st.zfull[sz], pz, a.status, &st.abort)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t adesc = sw128_desc(smem_u32(wring + (size_t)sw * 16384));
                    const uint64_t bdesc = sw128_desc(smem_u32(zring + (size_t)sz * zbytes));
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) tc_mma(d_tmem, adesc + 2 * kk, bdesc + 2 * kk, idesc, (kb | kk) != 0);
                    tc_commit(&st.done[sw]);
                    if (++sw == SW) { sw = 0; pw ^= 1u; }
                    if (++sz == SZ) { sz = 0; pz ^= 1u; }
                }
                if (!ok) break;
                tc_commit(&st.tfull[buf]);
            }
        }
    } else if ((warp >> 2) < ngroups) {  // ---- epilogue warps of row group g = warp / 4
        const int g = warp >> 2, qd = warp & 3;  // row group; TMEM lane quadrant 32 qd .. 32 qd + 31
        const int r = g * kWideGroup + qd * 32 + lane;  // this thread's hidden row
        float* tb = tbuf + (size_t)g * kWideRound * kWideTileStride;
        const float* col = tb + qd * 32 + lane;  // the row's column of the staged entries
        griddep_wait();
        WideRow<KM> w;
        w.init();
        uint32_t eb = 0;  // group barriers passed (two mbarriers used alternately)
        auto epi_sync = [&]() -> bool {
            __syncwarp();
            uint64_t* bar = &st.ebar[g][eb & 1];
            if (lane == 0) mbar_arrive(bar);
            const bool ok = mbar_wait_abortable(bar, (eb >> 1) & 1u, a.status, &st.abort);
            ++eb;
            return ok;
        };
        bool ok = true;
        for (int tile = t0, j = 0; tile < t1 && ok; ++tile, ++j) {
            const int buf = j & 1;
            if (!mbar_wait_abortable(&st.tfull[buf], (uint32_t)(j >> 1) & 1u, a.status, &st.abort)) break;
            tc_fence_after();
            // the group's 128 columns of this warp's 32 lanes (vocabulary entries)
            const uint32_t taddr = tmem + ((uint32_t)(qd * 32) << 16) + (uint32_t)(buf * NZ + g * kWideGroup);
            const int ncols = min(kWideGroup, R_pad - g * kWideGroup);
#pragma unroll
            for (int h = 0; h < 128 / kWideRound; ++h) {
                if (!ok) break;
                if (qd / kWideRoundWarps == h) {  // stage: this warp's 32 entries x the group's rows
                    float* trow = tb + (size_t)((qd % kWideRoundWarps) * 32 + lane) * kWideTileStride;
                    for (int c0 = 0; c0 < ncols; c0 += 32) {
                        float v32[32];
                        tc_ld32(taddr + (uint32_t)c0, v32);
                        if (LO) {  // (hi + lo, the same sum the 16-row kernel forms)
                            float l32[32];
                            tc_ld32(taddr + (uint32_t)(R_pad + c0), l32);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v32[i] += l32[i];
                        }
#pragma unroll
                        for (int i = 0; i < 32; ++i) trow[c0 + i] = v32[i];
                    }
                    // this warp's last read of the accumulator: hand it back to the MMA warp
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&st.tempty[buf]);
                }
                if (!(ok = epi_sync())) break;
                if (r < R) {
                    const int id0 = tile * 128 + h * kWideRound;
                    const int nv = min(kWideRound, a.V - id0);
                    FE_WIDE_BATCH(0);
                    if (kWideRound > 32) FE_WIDE_BATCH(32);
                    if (a.dbg_logits) {
                        const int rb = r % a.B, ri = r / a.B;
                        for (int u = 0; u < nv; ++u)
                            a.dbg_logits[((size_t)rb * a.N + ri) * a.V + id0 + u] = col[(size_t)u * kWideTileStride];
                    }
                }
                ok = epi_sync();
            }
        }
        // ---- the slab's partial of this thread's row
        if (ok && r < R) {
            const size_t base = (size_t)r * a.n_slabs + blockIdx.x;
#pragma unroll
            for (int q = 0; q < KM; ++q) {
                if (q < k) {
                    a.part_id[base * k + q] = w.v[q] == -INFINITY ? INT_MAX : w.i[q];
                    a.part_val[base * k + q] = w.v[q];
                    if (SMP) a.part_lg[base * k + q] = w.l[q];
                }
            }
            a.part_ms[base * 2 + 0] = w.m;
            a.part_ms[base * 2 + 1] = w.s;
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tc_dealloc(tmem, tmem_cols);
}

#undef FE_WIDE_BATCH

// One CTA per row: merges every slab's partial of that row (merge_rows).
__global__ void __launch_bounds__(128) lmhead_merge_kernel(const LmHeadArgs a, size_t smem_bytes) {
    const LaunchStamp stamp(a.stamp ? a.stamp + 4 : nullptr);
    extern __shared__ __align__(16) unsigned char msm[];
    griddep_launch_dependents();
    griddep_wait();
    // Every CTA of the product kernel has exited, so no split-tile flag can be set after
    // this: clear them for the next launch here (a CTA that gave up waiting on a flag
    // cannot leave it set for the next launch to take as ready).
    if (a.split_flag && blockIdx.x == 0)
        for (int j = threadIdx.x; j < a.n_slabs; j += blockDim.x) a.split_flag[j] = 0;
    merge_rows(a, blockIdx.x, blockIdx.x + 1, msm, smem_bytes);
}

bool lmhead_wide_ok(const LmHeadArgs& a) {
    return a.R > 0 && a.R <= kWideRowsMax && a.d % 64 == 0 && a.d <= kZprepMaxChunks * 8 * 256 &&
           a.top_k >= 1 && a.top_k <= kWideKMax;
}

size_t lmhead_mma_split_bytes(int R, const DeviceInfo& dev) {
    return (size_t)dev.num_sms * 128 * ((R + 7) / 8 * 8) * sizeof(float);
}

// rows of at most kWideLoRows take z as bf16 hi + lo (twice the rows of the operand)
size_t lmhead_wide_zb_bytes(int R, int d) {
    const int R_pad = (R + 15) / 16 * 16;
    return (size_t)(R_pad <= kWideLoRows ? 2 * R_pad : R_pad) * d * 2;
}

int lmhead_wide_slabs(int V, const DeviceInfo& dev) {
    const int ntiles = (V + 127) / 128;
    return ntiles < dev.num_sms ? ntiles : dev.num_sms;
}

cudaError_t lmhead_wide_prepare(const DeviceInfo& dev) {
    const int wsm = dev.max_smem_optin - (int)sizeof(WideState) - 256;
    cudaError_t e;
    for (auto k : {lmhead_wide_kernel<8, false, false>, lmhead_wide_kernel<16, false, false>,
                   lmhead_wide_kernel<8, true, false>, lmhead_wide_kernel<16, true, false>,
                   lmhead_wide_kernel<8, false, true>, lmhead_wide_kernel<16, false, true>,
                   lmhead_wide_kernel<8, true, true>, lmhead_wide_kernel<16, true, true>})
        if ((e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, wsm)) != cudaSuccess) return e;
    return cudaFuncSetAttribute(lmhead_merge_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kMergeMaxSmem);
}

cudaError_t launch_lmhead_wide(const LmHeadArgs& a, uint16_t* zb, const DeviceInfo& dev, cudaStream_t st,
                               cudaEvent_t after_prep, cudaEvent_t after_main) {
    if (!lmhead_wide_ok(a) || (reinterpret_cast<uintptr_t>(a.hid) & 15)) return cudaErrorInvalidValue;
    const int R_pad = (a.R + 15) / 16 * 16;
    const bool lo = R_pad <= kWideLoRows;  // z as bf16 hi + lo
    const int NZ = lo ? 2 * R_pad : R_pad;
    cudaError_t e = launch_k(zprep_kernel<bf16_t>, dim3(R_pad), dim3(256), 0, st, a.pdl, a.hid,
                             (const bf16_t*)a.gamma, a.R, R_pad, a.d, a.eps, zb, lo ? 1 : 0, a.stamp);
    if (e != cudaSuccess) return e;
    if (after_prep && (e = cudaEventRecord(after_prep, st)) != cudaSuccess) return e;
    // shared memory: the transpose buffers (one per row group), then up to kWideMaxZ z stages
    // (R_pad x 128 B) and the rest to the weight ring (at least as many stages)
    const size_t zst = (size_t)NZ * 128;
    const size_t tbytes = (size_t)((R_pad + kWideGroup - 1) / kWideGroup) * kWideRound * kWideTileStride * sizeof(float);
    const size_t budget = (size_t)dev.max_smem_optin - sizeof(WideState) - 256;
    if (budget < 1024 + tbytes + 2 * (16384 + zst)) return cudaErrorInvalidValue;
    const size_t avail = budget - 1024 - tbytes;
    int SZ = (int)(avail / (16384 + zst));
    SZ = SZ > kWideMaxZ ? kWideMaxZ : SZ;
    int SW = (int)((avail - SZ * zst) / 16384);
    SW = SW > kWideMaxW ? kWideMaxW : SW;
    const size_t zring = SZ * zst;
    const size_t smem = 1024 + (size_t)SW * 16384 + zring + tbytes;
    // TMEM: two NZ-column accumulators; the epilogue reads 32 columns at a time from a row
    // group's first column (and, with lo, from R_pad columns further on)
    const uint32_t need = (uint32_t)(NZ + (lo ? R_pad : 0) + ((std::min(R_pad, kWideGroup) + 31) / 32) * 32);
    uint32_t cols = 32;
    while (cols < (uint32_t)(2 * NZ) || cols < need) cols <<= 1;
    if (cols > 512) return cudaErrorInvalidValue;
    auto kern = lo ? (a.sample ? (a.top_k <= 8 ? lmhead_wide_kernel<8, true, true> : lmhead_wide_kernel<16, true, true>)
                               : (a.top_k <= 8 ? lmhead_wide_kernel<8, false, true> : lmhead_wide_kernel<16, false, true>))
                   : (a.sample ? (a.top_k <= 8 ? lmhead_wide_kernel<8, true, false> : lmhead_wide_kernel<16, true, false>)
                               : (a.top_k <= 8 ? lmhead_wide_kernel<8, false, false> : lmhead_wide_kernel<16, false, false>));
    e = launch_k(kern, dim3(a.n_slabs), dim3(kWideThreads), smem, st, a.pdl, a, (const uint16_t*)zb, R_pad, SW, SZ, cols);
    if (e != cudaSuccess) return e;
    if (after_main && (e = cudaEventRecord(after_main, st)) != cudaSuccess) return e;
    const size_t msmem = merge_smem_bytes(4, a.n_slabs, a.top_k, a.sample != 0);
    if (msmem > kMergeMaxSmem) return cudaErrorInvalidValue;
    return launch_k(lmhead_merge_kernel, dim3(a.R), dim3(128), msmem, st, a.pdl, a, msmem);
}

}  // namespace fe

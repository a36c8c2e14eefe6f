// Decode attention of each cascade layer L_i (Eq. 2) for the drafted row of every
// sequence, over that layer's own prefix K/V cache (the per-layer cache the paper's
// vLLM study refers to, Sec. 3.2) plus the row's own key and value.
//
// One kernel, split-KV: work item (split s, KV head g, sequence b) covers keys
// [s*split, min((s+1)*split, P_b + 1)) for the G = H / Hkv query heads sharing KV head g,
// so each K/V row is read once for all of its query heads. Four warps take 32-key chunks:
//   - scores: lane j owns key j of the chunk and streams its row with independent 16-byte
//     loads (no per-key dependency chain), dotting it with the G rotated, pre-scaled
//     queries read from shared memory (broadcast);
//   - online softmax per head across chunks (warp max / warp sum);
//   - P.V: lane j owns hd/32 dimensions; V rows are read coalesced, one per key.
// The warps' states merge into one partial (max, sum, accumulator) per head. The last
// split to finish for a (sequence, KV head) — an atomic counter — merges the splits with
// the usual max-shifted weights and writes o. The item holding key P_b also rotates the
// new key and writes the row's key and value into cache slot P_b.
#include "fe_kernels.h"
#include "fe_common.cuh"

namespace fe {

// address of cache row `pos` of sequence b, KV head g (null if the page id is invalid)
template <typename CT>
__device__ __forceinline__ CT* cache_row(CT* base, const AttnArgs& a, int b, int g, int pos, int hd) {
    if (a.page_table) {
        const int pg = a.page_table[(size_t)b * a.max_pages + pos / a.page_size];
        if (pg < 0 || pg >= a.n_pages) return nullptr;
        return base + (((size_t)pg * a.Hkv + g) * a.page_size + pos % a.page_size) * hd;
    }
    return base + (((size_t)b * a.Hkv + g) * a.max_seq + pos) * hd;
}

template <typename CT>
__device__ __forceinline__ void widen16(const uint4& v, float* f);
template <>
__device__ __forceinline__ void widen16<bf16_t>(const uint4& v, float* f) { Vec16<bf16_t>::widen(v, f); }
template <>
__device__ __forceinline__ void widen16<float>(const uint4& v, float* f) { Vec16<float>::widen(v, f); }

template <typename CT, int DPL>
__device__ __forceinline__ void load_dims(const CT* p, float* out) {
#pragma unroll
    for (int e = 0; e < DPL; ++e) out[e] = Storage<CT>::load(p, e);
}
template <>
__device__ __forceinline__ void load_dims<bf16_t, 4>(const bf16_t* p, float* out) {
    const uint2 v = *reinterpret_cast<const uint2*>(p);
    out[0] = __uint_as_float(v.x << 16); out[1] = __uint_as_float(v.x & 0xFFFF0000u);
    out[2] = __uint_as_float(v.y << 16); out[3] = __uint_as_float(v.y & 0xFFFF0000u);
}
template <>
__device__ __forceinline__ void load_dims<float, 4>(const float* p, float* out) {
    const float4 v = *reinterpret_cast<const float4*>(p);
    out[0] = v.x; out[1] = v.y; out[2] = v.z; out[3] = v.w;
}

constexpr int kAttnWarps = 4;

template <typename CT, int HD, int G>
__global__ void __launch_bounds__(kAttnWarps * 32) attn_kernel(const AttnArgs a) {
    constexpr int HALF = HD / 2;
    constexpr int DPL = HD / 32;               // dims per lane in P.V
    constexpr int VE = 16 / sizeof(CT);        // elements per 16-byte vector
    constexpr int NV = HD / VE;                // vectors per key row
    const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int P = a.prefix_len[b];
    const int ldq = (a.H + 2 * a.Hkv) * HD;

    __shared__ __align__(16) float qs[G][HD];
    __shared__ __align__(16) float kn[HD];
    __shared__ __align__(16) float vn[HD];
    __shared__ float pw[kAttnWarps][G][32];
    __shared__ float wm[kAttnWarps][G], wl[kAttnWarps][G];
    __shared__ float wacc[kAttnWarps][G][HD];
    __shared__ int s_last;

    float* out = a.out + (size_t)b * a.H * HD + (size_t)g * G * HD;
    const bool valid = P >= 0 && P + 1 <= a.max_seq;
    if (!valid) {
        if (s == 0) {
            if (g == 0 && t == 0) atomicOr(a.status, ST_CAPACITY);
            for (int i = t; i < G * HD; i += blockDim.x) out[i] = 0.f;
        }
        return;
    }
    const int t0 = s * a.split;
    if (t0 > P) return;  // beyond this sequence's keys: not an active split
    const int t1 = min(t0 + a.split, P + 1);
    const int n_act = min(a.n_split, P / a.split + 1);

    // queries of the group, rotated at position P and pre-scaled by 1/sqrt(hd)
    const float* cs = a.rope_cs + (size_t)P * HALF * 2;
    const float scale = 1.0f / sqrtf((float)HD);
    for (int idx = t; idx < G * HALF; idx += blockDim.x) {
        const int j = idx / HALF, i = idx % HALF;
        const float* q = a.qkv + (size_t)b * ldq + (size_t)(g * G + j) * HD;
        const float x1 = q[i], x2 = q[i + HALF], c = cs[2 * i], sn = cs[2 * i + 1];
        qs[j][i] = (x1 * c - x2 * sn) * scale;
        qs[j][i + HALF] = (x2 * c + x1 * sn) * scale;
    }
    if (t1 == P + 1) {  // this item holds the row's own key: rotate it and append k, v at slot P
        const float* kq = a.qkv + (size_t)b * ldq + (size_t)a.H * HD + (size_t)g * HD;
        const float* vq = kq + (size_t)a.Hkv * HD;
        CT* krow = cache_row<CT>((CT*)a.kc, a, b, g, P, HD);
        CT* vrow = cache_row<CT>((CT*)a.vc, a, b, g, P, HD);
        if ((!krow || !vrow) && t == 0) atomicOr(a.status, ST_DEVICE);
        for (int i = t; i < HALF; i += blockDim.x) {
            const float x1 = kq[i], x2 = kq[i + HALF], c = cs[2 * i], sn = cs[2 * i + 1];
            const float r1 = x1 * c - x2 * sn, r2 = x2 * c + x1 * sn;
            kn[i] = r1;
            kn[i + HALF] = r2;
            if (krow) {
                Storage<CT>::store(krow, i, r1);
                Storage<CT>::store(krow, i + HALF, r2);
            }
        }
        for (int i = t; i < HD; i += blockDim.x) {
            vn[i] = vq[i];
            if (vrow) Storage<CT>::store(vrow, i, vq[i]);
        }
    }
    __syncthreads();

    float m[G], l[G], acc[G][DPL];
#pragma unroll
    for (int j = 0; j < G; ++j) {
        m[j] = -INFINITY;
        l[j] = 0.f;
#pragma unroll
        for (int e = 0; e < DPL; ++e) acc[j][e] = 0.f;
    }
    bool bad_page = false;
    for (int base = t0 + warp * 32; base < t1; base += kAttnWarps * 32) {
        // ---- scores: lane owns key base + lane
        const int key = base + lane;
        bool kval = key < t1;
        float sc[G];
#pragma unroll
        for (int j = 0; j < G; ++j) sc[j] = 0.f;
        if (kval) {
            const CT* kr = nullptr;
            if (key < P) {
                kr = cache_row<CT>((CT*)a.kc, a, b, g, key, HD);
                if (!kr) { kval = false; bad_page = true; }
            }
            if (kval) {
#pragma unroll 4
                for (int v = 0; v < NV; ++v) {
                    float kk[VE];
                    if (kr) {
                        widen16<CT>(*reinterpret_cast<const uint4*>(kr + v * VE), kk);
                    } else {
#pragma unroll
                        for (int e = 0; e < VE; ++e) kk[e] = kn[v * VE + e];
                    }
#pragma unroll
                    for (int j = 0; j < G; ++j)
#pragma unroll
                        for (int e = 0; e < VE; ++e) sc[j] = fmaf(qs[j][v * VE + e], kk[e], sc[j]);
                }
            }
        }
        // ---- online softmax per head over this chunk
#pragma unroll
        for (int j = 0; j < G; ++j) {
            const float sj = kval ? sc[j] : -INFINITY;
            const float mn = fmaxf(m[j], warp_max(sj));
            const float c = m[j] == -INFINITY ? 0.f : expf(m[j] - mn);
            const float p = kval ? expf(sj - mn) : 0.f;
            l[j] = l[j] * c + warp_sum(p);
#pragma unroll
            for (int e = 0; e < DPL; ++e) acc[j][e] *= c;
            m[j] = mn;
            pw[warp][j][lane] = p;
        }
        __syncwarp();
        // ---- P.V: lane owns dims lane*DPL .. lane*DPL + DPL - 1
        const int nk = min(32, t1 - base);
#pragma unroll 4
        for (int kk = 0; kk < nk; ++kk) {
            const int pos = base + kk;
            float vv[DPL];
            if (pos < P) {
                const CT* vr = cache_row<CT>((CT*)a.vc, a, b, g, pos, HD);
                if (!vr) continue;
                load_dims<CT, DPL>(vr + lane * DPL, vv);
            } else {
#pragma unroll
                for (int e = 0; e < DPL; ++e) vv[e] = vn[lane * DPL + e];
            }
#pragma unroll
            for (int j = 0; j < G; ++j) {
                const float p = pw[warp][j][kk];
#pragma unroll
                for (int e = 0; e < DPL; ++e) acc[j][e] = fmaf(p, vv[e], acc[j][e]);
            }
        }
        __syncwarp();
    }
    if (bad_page) atomicOr(a.status, ST_DEVICE);  // any lane may have owned the bad key

    // ---- merge the warps into this split's partial per head
#pragma unroll
    for (int j = 0; j < G; ++j) {
#pragma unroll
        for (int e = 0; e < DPL; ++e) wacc[warp][j][lane * DPL + e] = acc[j][e];
        if (lane == 0) { wm[warp][j] = m[j]; wl[warp][j] = l[j]; }
    }
    __syncthreads();
    for (int idx = t; idx < G * HD; idx += blockDim.x) {
        const int j = idx / HD, dd = idx % HD;
        float M = wm[0][j];
        for (int w = 1; w < kAttnWarps; ++w) M = fmaxf(M, wm[w][j]);
        float v = 0.f, L = 0.f;
        for (int w = 0; w < kAttnWarps; ++w) {
            if (wm[w][j] == -INFINITY) continue;
            const float f = expf(wm[w][j] - M);
            v = fmaf(f, wacc[w][j][dd], v);
            L = fmaf(f, wl[w][j], L);
        }
        float* pp = a.part + (((size_t)b * a.H + g * G + j) * a.n_split + s) * (HD + 2);
        pp[dd] = v;
        if (dd == 0) { pp[HD] = M; pp[HD + 1] = L; }
    }
    // ---- the last active split of (b, g) combines all splits
    __threadfence();
    __syncthreads();
    if (t == 0) s_last = atomicAdd(&a.counters[b * a.Hkv + g], 1) == n_act - 1;
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    for (int idx = t; idx < G * HD; idx += blockDim.x) {
        const int j = idx / HD, dd = idx % HD;
        const float* pb = a.part + (((size_t)b * a.H + g * G + j) * a.n_split) * (HD + 2);
        float M = -INFINITY;
        for (int q = 0; q < n_act; ++q) M = fmaxf(M, __ldcg(pb + (size_t)q * (HD + 2) + HD));
        float v = 0.f, L = 0.f;
        for (int q = 0; q < n_act; ++q) {
            const float* p = pb + (size_t)q * (HD + 2);
            const float mq = __ldcg(p + HD);
            if (mq == -INFINITY) continue;
            const float f = expf(mq - M);
            v = fmaf(f, __ldcg(p + dd), v);
            L = fmaf(f, __ldcg(p + HD + 1), L);
        }
        out[(size_t)j * HD + dd] = L > 0.f ? v / L : 0.f;
    }
    if (t == 0) a.counters[b * a.Hkv + g] = 0;
}

// Keys per work item: aim at ~4 small CTAs per SM over all (sequence, KV head) pairs, in
// whole 32-key chunks, at least 64 keys.
int attn_split(int B, int Hkv, int max_seq, const DeviceInfo& dev) {
    const int items = B * Hkv;
    int per = (4 * dev.num_sms + items - 1) / items;  // splits per (sequence, KV head)
    if (per < 1) per = 1;
    int split = (max_seq + per - 1) / per;
    split = ((split + 31) / 32) * 32;
    return split < 64 ? 64 : split;
}

template <typename CT, int HD, int G>
static cudaError_t launch_g(const AttnArgs& a, cudaStream_t st) {
    dim3 grid(a.n_split, a.Hkv, a.B);
    attn_kernel<CT, HD, G><<<grid, kAttnWarps * 32, 0, st>>>(a);
    return cudaGetLastError();
}

template <typename CT, int HD>
static cudaError_t launch_hd(const AttnArgs& a, cudaStream_t st) {
    switch (a.H / a.Hkv) {
        case 1: return launch_g<CT, HD, 1>(a, st);
        case 2: return launch_g<CT, HD, 2>(a, st);
        case 4: return launch_g<CT, HD, 4>(a, st);
        case 8: return launch_g<CT, HD, 8>(a, st);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_attention(fe_dtype dt, const AttnArgs& a, cudaStream_t st) {
    if (dt == FE_F32) return a.hd == 64 ? launch_hd<float, 64>(a, st) : launch_hd<float, 128>(a, st);
    return a.hd == 64 ? launch_hd<bf16_t, 64>(a, st) : launch_hd<bf16_t, 128>(a, st);
}

}  // namespace fe

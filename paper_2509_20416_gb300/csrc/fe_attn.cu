// Decode attention of each cascade layer L_i (Eq. 2) for the drafted row of every
// sequence, over that layer's own prefix K/V cache (the per-layer cache of the paper's
// Sec. 3.2 vLLM study) plus the row's own key and value.
//
// Split-KV: work item (split s, KV head g, sequence b) covers keys [s*split, min((s+1)*split,
// P_b + 1)) for the G = H / Hkv query heads that share KV head g, so each K/V row is read
// once for all of its query heads. Four warps take keys round-robin; each lane holds hd/32
// dimensions; a warp computes q.k for the G heads with shuffles and keeps a running
// (max, sum, accumulator) per head (online softmax). The warps' states are merged through
// shared memory into one partial per head; attn_combine_kernel then merges the splits with
// the usual max-shifted weights. The item holding key P_b also rotates the new key and
// writes the row's key and value into cache slot P_b.
#include "fe_kernels.h"
#include "fe_common.cuh"

namespace fe {

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

template <typename CT, int HD, int G>
__global__ void __launch_bounds__(128) attn_split_kernel(const AttnArgs a) {
    constexpr int DPL = HD / 32;
    constexpr int HALF = HD / 2;
    const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int P = a.prefix_len[b];
    const int ldq = (a.H + 2 * a.Hkv) * HD;

    __shared__ float qs[G][HD];
    __shared__ float kn[HD], vn[HD];
    __shared__ float wm[4][G], wl[4][G];
    __shared__ float wacc[4][G][HD];

    auto part = [&](int j) { return a.part + (((size_t)b * a.H + g * G + j) * a.n_split + s) * (HD + 2); };
    const bool valid = P >= 0 && P + 1 <= a.max_seq;
    const int t0 = s * a.split;
    if (!valid || t0 > P) {
        if (!valid && s == 0 && g == 0 && t == 0) atomicOr(a.status, ST_CAPACITY);
        if (t < G) { part(t)[HD] = -INFINITY; part(t)[HD + 1] = 0.f; }
        return;
    }
    const int t1 = min(t0 + a.split, P + 1);
    const bool own = (t1 == P + 1);

    // queries of the group, rotated at position P and pre-scaled by 1/sqrt(hd)
    const float* cs = a.rope_cs + (size_t)P * HALF * 2;
    const float scale = 1.0f / sqrtf((float)HD);
    for (int idx = t; idx < G * HALF; idx += 128) {
        const int j = idx / HALF, i = idx % HALF;
        const float* q = a.qkv + (size_t)b * ldq + (size_t)(g * G + j) * HD;
        const float x1 = q[i], x2 = q[i + HALF], c = cs[2 * i], sn = cs[2 * i + 1];
        qs[j][i] = (x1 * c - x2 * sn) * scale;
        qs[j][i + HALF] = (x2 * c + x1 * sn) * scale;
    }
    if (own) {
        const float* kq = a.qkv + (size_t)b * ldq + (size_t)a.H * HD + (size_t)g * HD;
        const float* vq = kq + (size_t)a.Hkv * HD;
        CT* krow = cache_row<CT>((CT*)a.kc, a, b, g, P, HD);
        CT* vrow = cache_row<CT>((CT*)a.vc, a, b, g, P, HD);
        if (!krow || !vrow) {
            if (t == 0) atomicOr(a.status, ST_DEVICE);
        }
        for (int i = t; i < HALF; i += 128) {
            const float x1 = kq[i], x2 = kq[i + HALF], c = cs[2 * i], sn = cs[2 * i + 1];
            const float r1 = x1 * c - x2 * sn, r2 = x2 * c + x1 * sn;
            kn[i] = r1;
            kn[i + HALF] = r2;
            if (krow) {
                Storage<CT>::store(krow, i, r1);
                Storage<CT>::store(krow, i + HALF, r2);
            }
        }
        for (int i = t; i < HD; i += 128) {
            vn[i] = vq[i];
            if (vrow) Storage<CT>::store(vrow, i, vq[i]);
        }
    }
    __syncthreads();

    float qv[G][DPL];
#pragma unroll
    for (int j = 0; j < G; ++j)
#pragma unroll
        for (int e = 0; e < DPL; ++e) qv[j][e] = qs[j][lane * DPL + e];
    float m[G], l[G], acc[G][DPL];
#pragma unroll
    for (int j = 0; j < G; ++j) {
        m[j] = -INFINITY;
        l[j] = 0.f;
#pragma unroll
        for (int e = 0; e < DPL; ++e) acc[j][e] = 0.f;
    }

    bool bad_page = false;
    for (int pos = t0 + warp; pos < t1; pos += 4) {
        float kv[DPL], vv[DPL];
        if (pos < P) {
            const CT* kr = cache_row<CT>((CT*)a.kc, a, b, g, pos, HD);
            const CT* vr = cache_row<CT>((CT*)a.vc, a, b, g, pos, HD);
            if (!kr || !vr) { bad_page = true; continue; }
            load_dims<CT, DPL>(kr + lane * DPL, kv);
            load_dims<CT, DPL>(vr + lane * DPL, vv);
        } else {
#pragma unroll
            for (int e = 0; e < DPL; ++e) { kv[e] = kn[lane * DPL + e]; vv[e] = vn[lane * DPL + e]; }
        }
#pragma unroll
        for (int j = 0; j < G; ++j) {
            float d = 0.f;
#pragma unroll
            for (int e = 0; e < DPL; ++e) d = fmaf(qv[j][e], kv[e], d);
            d = warp_sum(d);
            const float mn = fmaxf(m[j], d);
            const float c = expf(m[j] - mn);
            const float p = expf(d - mn);
            l[j] = l[j] * c + p;
#pragma unroll
            for (int e = 0; e < DPL; ++e) acc[j][e] = fmaf(acc[j][e], c, p * vv[e]);
            m[j] = mn;
        }
    }
    if (bad_page && lane == 0) atomicOr(a.status, ST_DEVICE);

#pragma unroll
    for (int j = 0; j < G; ++j) {
#pragma unroll
        for (int e = 0; e < DPL; ++e) wacc[warp][j][lane * DPL + e] = acc[j][e];
        if (lane == 0) { wm[warp][j] = m[j]; wl[warp][j] = l[j]; }
    }
    __syncthreads();
    for (int idx = t; idx < G * HD; idx += 128) {
        const int j = idx / HD, dd = idx % HD;
        float M = wm[0][j];
        for (int w = 1; w < 4; ++w) M = fmaxf(M, wm[w][j]);
        float v = 0.f, L = 0.f;
        for (int w = 0; w < 4; ++w) {
            if (wm[w][j] == -INFINITY) continue;
            const float f = expf(wm[w][j] - M);
            v = fmaf(f, wacc[w][j][dd], v);
            L = fmaf(f, wl[w][j], L);
        }
        float* pp = part(j);
        pp[dd] = v;
        if (dd == 0) { pp[HD] = M; pp[HD + 1] = L; }
    }
}

// o[b, h*hd + d] = sum_s e^(m_s - M) acc_s[d] / sum_s e^(m_s - M) l_s
__global__ void attn_combine_kernel(const AttnArgs a) {
    const int h = blockIdx.x, b = blockIdx.y;
    const int hd = a.hd;
    const int P = a.prefix_len[b];
    float* o = a.out + (size_t)b * a.H * hd + (size_t)h * hd;
    if (P < 0 || P + 1 > a.max_seq) {
        for (int dd = threadIdx.x; dd < hd; dd += blockDim.x) o[dd] = 0.f;
        return;
    }
    const int ns = min(a.n_split, P / a.split + 1);
    const float* base = a.part + ((size_t)b * a.H + h) * a.n_split * (hd + 2);
    float M = -INFINITY;
    for (int s = 0; s < ns; ++s) M = fmaxf(M, base[(size_t)s * (hd + 2) + hd]);
    for (int dd = threadIdx.x; dd < hd; dd += blockDim.x) {
        float v = 0.f, L = 0.f;
        for (int s = 0; s < ns; ++s) {
            const float* p = base + (size_t)s * (hd + 2);
            if (p[hd] == -INFINITY) continue;
            const float f = expf(p[hd] - M);
            v = fmaf(f, p[dd], v);
            L = fmaf(f, p[hd + 1], L);
        }
        o[dd] = L > 0.f ? v / L : 0.f;
    }
}

int attn_split(int B, int Hkv, int max_seq, const DeviceInfo& dev) {
    const int items = B * Hkv;
    int per = (2 * dev.num_sms + items - 1) / items;  // splits per (sequence, KV head)
    if (per < 1) per = 1;
    int split = (max_seq + per - 1) / per;
    split = ((split + 15) / 16) * 16;
    if (split < 32) split = 32;
    return split;
}

template <typename CT, int HD, int G>
static cudaError_t launch_g(const AttnArgs& a, cudaStream_t st) {
    dim3 grid(a.n_split, a.Hkv, a.B);
    attn_split_kernel<CT, HD, G><<<grid, 128, 0, st>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    attn_combine_kernel<<<dim3(a.H, a.B), HD, 0, st>>>(a);
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

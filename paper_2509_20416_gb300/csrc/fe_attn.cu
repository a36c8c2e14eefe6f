// Decode attention of each cascade layer L_i (Eq. 2) for the drafted row of every
// sequence, over that layer's own prefix K/V cache (the per-layer cache the paper's
// vLLM study refers to, Sec. 3.2) plus the row's own key and value.
//
// One kernel, split-KV. Work item (split s, KV head g, sequence b) covers keys
// [s*split, min((s+1)*split, P_b + 1)) for the G = H / Hkv query heads sharing KV head g,
// so each K/V row is read once for all of its query heads.
//   - Each of the 4 warps runs its own pipeline over 32-key chunks of the item: lane 0
//     issues bulk TMA copies (cp.async.bulk) of the chunk's K and V rows into the warp's
//     shared-memory slots — one copy per contiguous run of rows (the whole chunk when the
//     cache is contiguous, one per page when it is paged) — completing on the slot's
//     mbarrier; with two slots the next chunk streams in while the warp computes.
//   - Scores: lane l holds dimensions l*hd/32 .. of every query head in registers, reads
//     the same dimensions of each key row from shared memory (conflict-free), and the
//     32 / G keys x G heads partial dots of a batch are summed across lanes with one
//     transposing shuffle reduction (31 shuffles for 32 scores).
//   - Online softmax per head across chunks; P.V from shared memory, lane l owning the
//     same hd/32 dimensions of the output.
// The warps' states merge into one partial (max, sum, accumulator) per head. The last
// split to finish for a (sequence, KV head) — an atomic counter — merges the splits with
// the usual max-shifted weights and writes o. The item holding key P_b also rotates the
// new key and writes the row's key and value into cache slot P_b (keys are cached after
// RoPE); the own row is used from shared memory, unrounded.
#include "fe_kernels.h"
#include "fe_common.cuh"
#include "fe_stream.cuh"

namespace fe {

constexpr int kAttnWarps = 4;
constexpr int kChunkKeys = 32;
constexpr int kAttnMaxSlots = 2;
constexpr int kAttnPageSmem = 32 * 1024;  // dynamic shared memory reserved for an item's page ids

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
__device__ __forceinline__ void load_dims<bf16_t, 2>(const bf16_t* p, float* out) {
    const uint32_t v = *reinterpret_cast<const uint32_t*>(p);
    out[0] = __uint_as_float(v << 16); out[1] = __uint_as_float(v & 0xFFFF0000u);
}
template <>
__device__ __forceinline__ void load_dims<float, 4>(const float* p, float* out) {
    const float4 v = *reinterpret_cast<const float4*>(p);
    out[0] = v.x; out[1] = v.y; out[2] = v.z; out[3] = v.w;
}
template <>
__device__ __forceinline__ void load_dims<float, 2>(const float* p, float* out) {
    const float2 v = *reinterpret_cast<const float2*>(p);
    out[0] = v.x; out[1] = v.y;
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
__global__ void __launch_bounds__(kAttnWarps * 32) attn_kernel(const AttnArgs a, int S) {
    constexpr int HALF = HD / 2;
    constexpr int DPL = HD / 32;                  // dims per lane
    constexpr int KB = 32 / G;                    // keys per score batch (KB * G = 32 scores)
    constexpr int NB = kChunkKeys / KB;           // batches per chunk
    constexpr uint32_t ROWB = HD * sizeof(CT);    // bytes per cache row
    constexpr uint32_t CHB = kChunkKeys * ROWB;   // bytes per chunk of K (or V)
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ __align__(16) float qs[G][HD];
    __shared__ __align__(16) float kn[HD];
    __shared__ __align__(16) float vn[HD];
    __shared__ float pw[kAttnWarps][kChunkKeys * G];
    __shared__ float wm[kAttnWarps][G], wl[kAttnWarps][G];
    __shared__ __align__(8) uint64_t bars[kAttnWarps][kAttnMaxSlots];
    __shared__ int s_last, s_abort;

    const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int P = a.prefix_len[b];
    const int ldq = (a.H + 2 * a.Hkv) * HD;

    float* out = a.out + (size_t)b * a.H * HD + (size_t)g * G * HD;
    const bool valid = P >= 0 && P + 1 <= a.max_seq;
    if (!valid) {
        griddep_launch_dependents();
        griddep_wait();
        if (s == 0) {
            if (g == 0 && t == 0) atomicOr(a.status, ST_CAPACITY);
            for (int i = t; i < G * HD; i += blockDim.x) out[i] = 0.f;
        }
        return;
    }
    const int t0 = s * a.split;
    if (t0 > P) {  // beyond this sequence's keys: not an active split
        griddep_launch_dependents();
        return;
    }
    const int t1 = min(t0 + a.split, P + 1);
    const int n_act = min(a.n_split, P / a.split + 1);
    const int nchunks = (t1 - t0 + kChunkKeys - 1) / kChunkKeys;

    unsigned char* kbuf = dsm + (size_t)warp * S * 2 * CHB;  // [S][K chunk, V chunk]
    uint64_t* bar = bars[warp];
    if (lane == 0) {
        for (int i = 0; i < S; ++i) mbar_init(&bar[i], 1);
        mbar_fence_init();
    }
    if (t == 0) s_abort = 0;
    // Paged caches: this item's page ids, read once into shared memory (after the K/V slots;
    // -1 marks an invalid id), so that issuing a chunk needs no round trip to the table.
    int* spg = reinterpret_cast<int*>(dsm + (size_t)kAttnWarps * S * 2 * CHB);
    const int pg0 = a.page_table ? t0 / a.page_size : 0;
    if (a.page_table) {
        const int last_row = min(t1, P) - 1;  // cached rows are < P
        const int npg = last_row >= t0 ? last_row / a.page_size - pg0 + 1 : 0;
        for (int i = t; i < npg; i += blockDim.x) {
            const int pg = a.page_table[(size_t)b * a.max_pages + pg0 + i];
            spg[i] = (pg < 0 || pg >= a.n_pages) ? -1 : pg;
        }
    }
    // address of cached row `pos` (< P) of this item from the staged page ids (null if invalid)
    auto prow = [&](CT* base, int pos) -> CT* {
        const int pg = spg[pos / a.page_size - pg0];
        if (pg < 0) return nullptr;
        return base + (((size_t)pg * a.Hkv + g) * a.page_size + pos % a.page_size) * HD;
    };

    // Chunk j of this warp covers keys [c0, c0 + 32), c0 = t0 + (warp + 4 j) * 32; its rows
    // below P come from the cache. Returns the mask of rows whose page id was invalid.
    auto issue = [&](int j, int slot) -> uint32_t {
        const int c0 = t0 + (warp + kAttnWarps * j) * kChunkKeys;
        const int rows = max(0, min(kChunkKeys, min(t1, P) - c0));
        unsigned char* kd = kbuf + (size_t)slot * 2 * CHB;
        unsigned char* vd = kd + CHB;
        uint32_t bad = 0, bytes = 0;
        if (a.page_table) {
            for (int p = c0; p < c0 + rows;) {
                const int n = min(a.page_size - p % a.page_size, c0 + rows - p);
                if (spg[p / a.page_size - pg0] >= 0) bytes += 2u * n * ROWB;
                else bad |= (n >= 32 ? 0xffffffffu : ((1u << n) - 1u)) << (p - c0);
                p += n;
            }
        } else {
            bytes = 2u * rows * ROWB;
        }
        mbar_arrive_expect_tx(&bar[slot], bytes);
        if (a.page_table) {
            for (int p = c0; p < c0 + rows;) {
                const int n = min(a.page_size - p % a.page_size, c0 + rows - p);
                const CT* kr = prow((CT*)a.kc, p);
                const CT* vr = prow((CT*)a.vc, p);
                if (kr && vr) {
                    bulk_g2s(kd + (size_t)(p - c0) * ROWB, kr, n * ROWB, &bar[slot]);
                    bulk_g2s(vd + (size_t)(p - c0) * ROWB, vr, n * ROWB, &bar[slot]);
                }
                p += n;
            }
        } else if (rows > 0) {
            bulk_g2s(kd, cache_row<CT>((CT*)a.kc, a, b, g, c0, HD), rows * ROWB, &bar[slot]);
            bulk_g2s(vd, cache_row<CT>((CT*)a.vc, a, b, g, c0, HD), rows * ROWB, &bar[slot]);
        }
        return bad;
    };
    const int my_chunks = warp < nchunks ? (nchunks - warp + kAttnWarps - 1) / kAttnWarps : 0;
    uint32_t badmask[kAttnMaxSlots] = {0u, 0u};  // per slot, meaningful on lane 0
    int issued = 0;
    __syncthreads();  // barriers initialised
    // cached prefix rows (< P) are not written by the earlier kernels of this draft: copy
    // them before waiting for the QKV projection
    if (lane == 0)
        for (int j = 0; j < S && j < my_chunks; ++j, ++issued) badmask[j] = issue(j, j);
    griddep_launch_dependents();
    griddep_wait();

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
    using R = WarpMultiSum<32>;
    const int head = lane % G;
    for (int j = 0; j < my_chunks; ++j) {
        const int slot = j % S;
        const int c0 = t0 + (warp + kAttnWarps * j) * kChunkKeys;
        const int nk = min(kChunkKeys, t1 - c0);
        const uint32_t bad = __shfl_sync(0xffffffffu, badmask[slot], 0);
        if (bad && lane == 0) atomicOr(a.status, ST_DEVICE);
        mbar_wait_abortable(&bar[slot], (uint32_t)(j / S) & 1u, a.status, &s_abort);
        const CT* kc = (const CT*)(kbuf + (size_t)slot * 2 * CHB);
        const CT* vc = (const CT*)(kbuf + (size_t)slot * 2 * CHB + CHB);
        // ---- scores: batch bt holds keys bt*KB .. bt*KB + KB - 1 for all G heads; after the
        // reduction lane l holds (key bt*KB + l / G, head l % G)
        float sc[NB];
#pragma unroll
        for (int bt = 0; bt < NB; ++bt) {
            float part[32];
#pragma unroll
            for (int kk = 0; kk < KB; ++kk) {
                const int key = bt * KB + kk;
                float kv[DPL];
                if (key < nk && c0 + key < P) {
                    load_dims<CT, DPL>(kc + (size_t)key * HD + lane * DPL, kv);
                } else {
#pragma unroll
                    for (int e = 0; e < DPL; ++e) kv[e] = key < nk ? kn[lane * DPL + e] : 0.f;
                }
#pragma unroll
                for (int hh = 0; hh < G; ++hh) {
                    float d = 0.f;
#pragma unroll
                    for (int e = 0; e < DPL; ++e) d = fmaf(qv[hh][e], kv[e], d);
                    part[kk * G + hh] = d;
                }
            }
            R::run(part, lane);
            const int key = bt * KB + lane / G;
            const bool ok = key < nk && !((bad >> key) & 1u);
            sc[bt] = ok ? part[0] : -INFINITY;
        }
        // ---- online softmax per head (lanes with lane % G == h hold head h's scores)
        float cm = -INFINITY;
#pragma unroll
        for (int bt = 0; bt < NB; ++bt) cm = fmaxf(cm, sc[bt]);
#pragma unroll
        for (int o = 16; o >= G; o >>= 1) cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, o));
        float mnew[G], corr[G];
        float mine = 0.f;
#pragma unroll
        for (int hh = 0; hh < G; ++hh) {
            const float cmh = __shfl_sync(0xffffffffu, cm, hh);
            mnew[hh] = fmaxf(m[hh], cmh);
            corr[hh] = m[hh] == -INFINITY ? 0.f : expf(m[hh] - mnew[hh]);
            if (head == hh) mine = mnew[hh];
        }
        float csum = 0.f;
#pragma unroll
        for (int bt = 0; bt < NB; ++bt) {
            const float p = sc[bt] == -INFINITY ? 0.f : expf(sc[bt] - mine);
            csum += p;
            pw[warp][(bt * KB + lane / G) * G + head] = p;
        }
#pragma unroll
        for (int o = 16; o >= G; o >>= 1) csum += __shfl_xor_sync(0xffffffffu, csum, o);
#pragma unroll
        for (int hh = 0; hh < G; ++hh) {
            l[hh] = l[hh] * corr[hh] + __shfl_sync(0xffffffffu, csum, hh);
#pragma unroll
            for (int e = 0; e < DPL; ++e) acc[hh][e] *= corr[hh];
            m[hh] = mnew[hh];
        }
        __syncwarp();
        // ---- P.V for the chunk
        for (int key = 0; key < nk; ++key) {
            if ((bad >> key) & 1u) continue;
            float vv[DPL];
            if (c0 + key < P) {
                load_dims<CT, DPL>(vc + (size_t)key * HD + lane * DPL, vv);
            } else {
#pragma unroll
                for (int e = 0; e < DPL; ++e) vv[e] = vn[lane * DPL + e];
            }
#pragma unroll
            for (int hh = 0; hh < G; ++hh) {
                const float p = pw[warp][key * G + hh];
#pragma unroll
                for (int e = 0; e < DPL; ++e) acc[hh][e] = fmaf(p, vv[e], acc[hh][e]);
            }
        }
        __syncwarp();
        // refill the slot with this warp's chunk j + S
        if (lane == 0 && j + S < my_chunks && !*(volatile int*)&s_abort) {
            badmask[slot] = issue(j + S, slot);
            ++issued;
        }
        __syncwarp();
    }
    // never leave with copies in flight (only possible after an aborted wait)
    if (lane == 0 && *(volatile int*)&s_abort)
        for (int j = max(0, issued - S); j < issued; ++j) mbar_wait(&bar[j % S], (uint32_t)(j / S) & 1u, a.status, 100000000LL);

    // ---- merge the warps into this split's partial per head (the K/V slots are free now
    // and hold the warps' accumulators)
    float (*wacc)[G][HD] = reinterpret_cast<float (*)[G][HD]>(dsm);
    __syncthreads();
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
#pragma unroll
        for (int e = 0; e < DPL; ++e) wacc[warp][hh][lane * DPL + e] = acc[hh][e];
        if (lane == 0) { wm[warp][hh] = m[hh]; wl[warp][hh] = l[hh]; }
    }
    __syncthreads();
    for (int idx = t; idx < G * HD; idx += blockDim.x) {
        const int hh = idx / HD, dd = idx % HD;
        float M = wm[0][hh];
        for (int w = 1; w < kAttnWarps; ++w) M = fmaxf(M, wm[w][hh]);
        float v = 0.f, L = 0.f;
        for (int w = 0; w < kAttnWarps; ++w) {
            if (wm[w][hh] == -INFINITY) continue;
            const float f = expf(wm[w][hh] - M);
            v = fmaf(f, wacc[w][hh][dd], v);
            L = fmaf(f, wl[w][hh], L);
        }
        float* pp = a.part + (((size_t)b * a.H + g * G + hh) * a.n_split + s) * (HD + 2);
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
    // Each split's (max, sum) per head goes to shared memory (the K/V slots are free now) in
    // one round trip; each head's weights exp(M_q - M) are formed there; each output then
    // sums its splits with eight loads in flight (a load-then-accumulate loop would wait a
    // full L2 round trip per split).
    const float* pb0 = a.part + ((size_t)b * a.H + g * G) * a.n_split * (HD + 2);
    float* wq = reinterpret_cast<float*>(dsm);  // [n_act][G] weights, then [n_act][G] sums
    float* lq = wq + n_act * G;
    __shared__ float hl[G];
    if ((size_t)2 * n_act * G * sizeof(float) <= (size_t)kAttnWarps * S * 2 * CHB) {
        for (int idx = t; idx < n_act * G; idx += blockDim.x) {
            const int q = idx / G, hh = idx % G;
            const float* p = pb0 + ((size_t)hh * a.n_split + q) * (HD + 2) + HD;
            wq[idx] = __ldcg(p);
            lq[idx] = __ldcg(p + 1);
        }
        __syncthreads();
        for (int hh = warp; hh < G; hh += kAttnWarps) {
            float M = -INFINITY;
            for (int q = lane; q < n_act; q += 32) M = fmaxf(M, wq[q * G + hh]);
            M = warp_max(M);
            float L = 0.f;
            for (int q = lane; q < n_act; q += 32) {
                const float mq = wq[q * G + hh];
                const float f = mq == -INFINITY ? 0.f : expf(mq - M);
                wq[q * G + hh] = f;
                L = fmaf(f, lq[q * G + hh], L);
            }
            L = warp_sum(L);
            if (lane == 0) hl[hh] = L;
        }
        __syncthreads();
        // thread t owns outputs t, t + 128, ... (NO of them) and loads QB splits of each at once
        constexpr int NO = (G * HD + kAttnWarps * 32 - 1) / (kAttnWarps * 32);
        constexpr int QB = NO >= 32 ? 1 : 32 / NO;
        float v[NO];
#pragma unroll
        for (int o = 0; o < NO; ++o) v[o] = 0.f;
        for (int q0 = 0; q0 < n_act; q0 += QB) {
            float x[NO][QB];
#pragma unroll
            for (int o = 0; o < NO; ++o) {
                const int idx = t + o * kAttnWarps * 32, hh = idx / HD, dd = idx % HD;
                const float* p = pb0 + (size_t)hh * a.n_split * (HD + 2) + dd;
#pragma unroll
                for (int u = 0; u < QB; ++u)
                    x[o][u] = idx < G * HD && q0 + u < n_act ? __ldcg(p + (size_t)(q0 + u) * (HD + 2)) : 0.f;
            }
#pragma unroll
            for (int o = 0; o < NO; ++o) {
                const int idx = t + o * kAttnWarps * 32, hh = (idx / HD) % G;
#pragma unroll
                for (int u = 0; u < QB; ++u)
                    if (q0 + u < n_act) v[o] = fmaf(wq[(q0 + u) * G + hh], x[o][u], v[o]);
            }
        }
#pragma unroll
        for (int o = 0; o < NO; ++o) {
            const int idx = t + o * kAttnWarps * 32;
            if (idx < G * HD) {
                const int hh = idx / HD, dd = idx % HD;
                out[(size_t)hh * HD + dd] = hl[hh] > 0.f ? v[o] / hl[hh] : 0.f;
            }
        }
    } else {  // more splits than the slots hold: the same sums, one split at a time
        for (int idx = t; idx < G * HD; idx += blockDim.x) {
            const int hh = idx / HD, dd = idx % HD;
            const float* pb = pb0 + (size_t)hh * a.n_split * (HD + 2);
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
            out[(size_t)hh * HD + dd] = L > 0.f ? v / L : 0.f;
        }
    }
    if (t == 0) a.counters[b * a.Hkv + g] = 0;
}

// Keys per work item: aim at ~4 CTAs per SM over all (sequence, KV head) pairs, in whole
// multiples of one chunk per warp (128 keys), so that every warp of a CTA has work and the
// last split's combine has few partials to read.
int attn_split(int B, int Hkv, int max_seq, const DeviceInfo& dev) {
    constexpr int unit = kAttnWarps * kChunkKeys;
    const int items = B * Hkv;
    int per = (4 * dev.num_sms + items - 1) / items;  // splits per (sequence, KV head)
    if (per < 1) per = 1;
    int split = (max_seq + per - 1) / per;
    split = ((split + unit - 1) / unit) * unit;
    return split < unit ? unit : split;
}

// Pipeline slots per warp: two when a warp has more than one chunk and a chunk of K (or
// V) is at most 8 KB (bf16, hd 128), else one; at most 128 KB of dynamic shared memory.
// One slot per warp: a CTA then needs ~70 KB (bf16, hd 128) and three fit on an SM. The
// per-chunk work is a chain of shared-memory loads and shuffles, latency-bound in one warp,
// so more warps per SM (other CTAs) hide it better than a second slot per warp does.
static int max_slots(int, int) { return 1; }
static int attn_slots(int, int, int) { return 1; }

static size_t attn_smem(int hd, int es, int S) { return (size_t)kAttnWarps * S * 2 * kChunkKeys * hd * es; }
// page ids one work item covers (paged caches)
static size_t attn_page_ints(const AttnArgs& a) {
    return a.page_table ? (size_t)(a.split + a.page_size - 1) / a.page_size + 1 : 0;
}

template <typename CT, int HD, int G>
static cudaError_t prepare_g() {
    return cudaFuncSetAttribute(attn_kernel<CT, HD, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)attn_smem(HD, sizeof(CT), max_slots(HD, sizeof(CT))) + kAttnPageSmem);
}

template <typename CT, int HD, int G>
static cudaError_t launch_g(const AttnArgs& a, cudaStream_t st) {
    const int S = attn_slots(a.split, HD, sizeof(CT));
    const size_t pg = attn_page_ints(a) * sizeof(int);
    if (pg > (size_t)kAttnPageSmem) return cudaErrorInvalidValue;
    dim3 grid(a.n_split, a.Hkv, a.B);
    return launch_k(attn_kernel<CT, HD, G>, grid, dim3(kAttnWarps * 32), attn_smem(HD, sizeof(CT), S) + pg, st, a.pdl,
                    a, S);
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

template <typename CT, int HD>
static cudaError_t prepare_hd() {
    cudaError_t e;
    if ((e = prepare_g<CT, HD, 1>()) != cudaSuccess) return e;
    if ((e = prepare_g<CT, HD, 2>()) != cudaSuccess) return e;
    if ((e = prepare_g<CT, HD, 4>()) != cudaSuccess) return e;
    return prepare_g<CT, HD, 8>();
}

cudaError_t attention_prepare() {
    cudaError_t e;
    if ((e = prepare_hd<float, 64>()) != cudaSuccess) return e;
    if ((e = prepare_hd<float, 128>()) != cudaSuccess) return e;
    if ((e = prepare_hd<bf16_t, 64>()) != cudaSuccess) return e;
    return prepare_hd<bf16_t, 128>();
}

cudaError_t launch_attention(fe_dtype dt, const AttnArgs& a, cudaStream_t st) {
    if (dt == FE_F32) return a.hd == 64 ? launch_hd<float, 64>(a, st) : launch_hd<float, 128>(a, st);
    return a.hd == 64 ? launch_hd<bf16_t, 64>(a, st) : launch_hd<bf16_t, 128>(a, st);
}

}  // namespace fe

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
#include <cstdlib>

#include "fe_kernels.h"
#include "fe_common.cuh"
#include "fe_stream.cuh"
#include "fe_tc.cuh"
#include "fe_splitk.cuh"

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

// Output `head`, dimension dd of row qrow: into `out`, or (a.xb) as the bf16 hi + lo pair of
// the O projection's operand (x = hi + lo to ~16 significant bits, as the operand prep
// splits it), column head * HD + dd, in the 128-byte-swizzled K-major layout.
// A QKV phase that deferred its split tiles (a.qprev): the finished (pre-RoPE) query
// columns of heads [g G, g G + G) of row qrow into q (G x HD, heads consecutive) and, when
// `own`, the row's key and value into kn / vn, each 8-column chunk summed from the phase's
// shares in CTA order (its own fix-up). Thread t takes chunks t, t + blockDim.x, ...
template <int HD, int G>
__device__ __forceinline__ void load_qkv(const AttnArgs& a, size_t qrow, int g, bool own, float* q, float* kn,
                                         float* vn) {
    constexpr int NQ = G * HD / 8, NO = HD / 8;
    constexpr int NC = (NQ + 2 * NO + kAttnWarps * 32 - 1) / (kAttnWarps * 32);
    const int n = NQ + (own ? 2 * NO : 0);
    auto column = [&](int c) {  // first qkv column of chunk c
        return c < NQ ? g * G * HD + 8 * c
                      : (c < NQ + NO ? (a.H + g) * HD + 8 * (c - NQ) : (a.H + a.Hkv + g) * HD + 8 * (c - NQ - NO));
    };
    float v[NC][8];
#pragma unroll
    for (int j = 0; j < NC; ++j) {
        const int c = threadIdx.x + j * kAttnWarps * 32;
        if (c >= n) break;
        prev_finish_t<false, false>(a.qprev, a.qprev_bpad, (int)qrow, column(c), v[j]);
    }
#pragma unroll
    for (int j = 0; j < NC; ++j) {
        const int c = threadIdx.x + j * kAttnWarps * 32;
        if (c >= n) break;
        float* dst = c < NQ ? q + 8 * c : (c < NQ + NO ? kn + 8 * (c - NQ) : vn + 8 * (c - NQ - NO));
        reinterpret_cast<float4*>(dst)[0] = make_float4(v[j][0], v[j][1], v[j][2], v[j][3]);
        reinterpret_cast<float4*>(dst)[1] = make_float4(v[j][4], v[j][5], v[j][6], v[j][7]);
    }
}

template <int HD>
__device__ __forceinline__ void put_out(const AttnArgs& a, size_t qrow, int head, int dd, float v) {
    if (a.xb) {
        const int k = head * HD + dd;
        const uint16_t hi = f32_to_bf16(v), lo = f32_to_bf16(v - bf16_to_f32(hi));
        unsigned char* blk = (unsigned char*)a.xb + (size_t)(k >> 6) * (2 * a.xb_bpad) * 128;
        const uint32_t ch = (uint32_t)(k & 63) >> 3, el = (uint32_t)(k & 7);
        *reinterpret_cast<uint16_t*>(blk + sw128_offset((uint32_t)qrow, ch) + 2 * el) = hi;
        *reinterpret_cast<uint16_t*>(blk + sw128_offset((uint32_t)(a.xb_bpad + qrow), ch) + 2 * el) = lo;
    } else {
        a.out[qrow * a.H * HD + (size_t)head * HD + dd] = v;
    }
}

// A split's partial per head: the weighted value sum [HD], then its max and its sum of
// weights, padded to a multiple of four floats so that rows start on 16-byte boundaries.
template <int HD>
constexpr int part_row() { return HD + 4; }

// The last split of (sequence, KV head) combines every active split's partials into the
// G heads' outputs: out = sum_q w_q acc_q / sum_q w_q l_q with w_q = exp(m_q - max m). The
// partial rows of as many heads as `smem` holds are staged into shared memory by bulk
// copies (one per head: its splits' rows are contiguous), then each head's weights are
// formed once and every output sums its splits from shared memory. BASE2: the maxima are
// in base 2 (scores pre-scaled by log2 e).
template <int HD, int G, bool BASE2>
__device__ __forceinline__ void combine_splits(const AttnArgs& a, const float* pb0, int n_act, size_t qrow, int head0,
                                               unsigned char* smem, size_t smem_bytes) {
    constexpr int RS = part_row<HD>();
    constexpr int NW = kAttnWarps;
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    __shared__ float hl[G];
    const size_t per_head = (size_t)n_act * (RS + 1) * sizeof(float);  // its rows and weights
    const int Hp = (int)min((size_t)G, smem_bytes / per_head);
    if (Hp < 1) {  // more splits than shared memory holds: one split at a time from L2
        for (int idx = t; idx < G * HD; idx += NW * 32) {
            const int hh = idx / HD, dd = idx % HD;
            const float* pb = pb0 + (size_t)hh * a.n_split * RS;
            float M = -INFINITY;
            for (int q = 0; q < n_act; ++q) M = fmaxf(M, __ldcg(pb + (size_t)q * RS + HD));
            float v = 0.f, L = 0.f;
            for (int q = 0; q < n_act; ++q) {
                const float* p = pb + (size_t)q * RS;
                const float mq = __ldcg(p + HD);
                if (mq == -INFINITY) continue;
                const float f = BASE2 ? exp2f(mq - M) : expf(mq - M);
                v = fmaf(f, __ldcg(p + dd), v);
                L = fmaf(f, __ldcg(p + HD + 1), L);
            }
            put_out<HD>(a, qrow, head0 + hh, dd, L > 0.f ? v / L : 0.f);
        }
        return;
    }
    float* rows = reinterpret_cast<float*>(smem);  // [hn][n_act][RS]
    __shared__ uint64_t cbar;                      // completion of a pass's bulk copies
    if (t == 0) {
        mbar_init(&cbar, 1);
        mbar_fence_init();
    }
    __syncthreads();
    for (int h0 = 0, pass = 0; h0 < G; h0 += Hp, ++pass) {
        const int hn = min(Hp, G - h0);
        float* wq = rows + (size_t)hn * n_act * RS;  // [hn][n_act] weights
        // a head's rows of every split are contiguous: one bulk copy per head
        if (t == 0) {
            const uint32_t hb = (uint32_t)(n_act * RS * sizeof(float));
            // the partials were written by other CTAs (generic proxy) and this shared memory
            // was last written by this CTA's threads: both before the async-proxy copies
            asm volatile("fence.proxy.async.global;" ::: "memory");
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            mbar_arrive_expect_tx(&cbar, hb * hn);
            for (int hh = 0; hh < hn; ++hh)
                bulk_g2s(rows + (size_t)hh * n_act * RS, pb0 + (size_t)(h0 + hh) * a.n_split * RS, hb, &cbar);
        }
        if (!mbar_wait(&cbar, (uint32_t)pass & 1u, a.status)) return;  // (bounded; ST_TIMEOUT recorded)
        for (int hh = warp; hh < hn; hh += NW) {
            const float* hr = rows + (size_t)hh * n_act * RS;
            float M = -INFINITY;
            for (int q = lane; q < n_act; q += 32) M = fmaxf(M, hr[(size_t)q * RS + HD]);
            M = warp_max(M);
            float L = 0.f;
            for (int q = lane; q < n_act; q += 32) {
                const float mq = hr[(size_t)q * RS + HD];
                const float f = mq == -INFINITY ? 0.f : (BASE2 ? exp2f(mq - M) : expf(mq - M));
                wq[hh * n_act + q] = f;
                L = fmaf(f, hr[(size_t)q * RS + HD + 1], L);
            }
            L = warp_sum(L);
            if (lane == 0) hl[hh] = L;
        }
        __syncthreads();
        // thread t owns outputs t, t + 128, ...: the splits in the outer loop, so that its
        // outputs' sums advance together
        constexpr int NO = (G * HD + NW * 32 - 1) / (NW * 32);
        float v[NO];
#pragma unroll
        for (int o = 0; o < NO; ++o) v[o] = 0.f;
        for (int q = 0; q < n_act; ++q) {
#pragma unroll
            for (int o = 0; o < NO; ++o) {
                const int idx = t + o * NW * 32;
                if (idx < hn * HD) {
                    const int hh = idx / HD, dd = idx - hh * HD;
                    v[o] = fmaf(wq[hh * n_act + q], rows[((size_t)hh * n_act + q) * RS + dd], v[o]);
                }
            }
        }
#pragma unroll
        for (int o = 0; o < NO; ++o) {
            const int idx = t + o * NW * 32;
            if (idx < hn * HD) {
                const int hh = idx / HD, dd = idx - hh * HD;
                put_out<HD>(a, qrow, head0 + h0 + hh, dd, hl[hh] > 0.f ? v[o] / hl[hh] : 0.f);
            }
        }
        __syncthreads();  // the next pass overwrites the rows
    }
}

template <typename CT, int HD, int G>
__global__ void __launch_bounds__(kAttnWarps * 32) attn_kernel(const AttnArgs a, int S) {
    const LaunchStamp stamp(a.stamp);
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
    // (a commit launch handles row index pos_add of every sequence: its position is
    // prefix_len + pos_add, and sequences with fewer rows to commit have no work here)
    if (a.n_rows && a.pos_add >= a.n_rows[b]) {
        griddep_launch_dependents();
        return;
    }
    const int P = a.prefix_len[b] + a.pos_add;
    const size_t qrow = (size_t)b * a.row_stride + a.row_off;  // this row in qkv and out

    const bool valid = P >= 0 && P + 1 <= a.max_seq;
    if (!valid) {
        griddep_launch_dependents();
        griddep_wait();
        if (s == 0) {
            if (g == 0 && t == 0) atomicOr(a.status, ST_CAPACITY);
            for (int i = t; i < G * HD; i += blockDim.x) put_out<HD>(a, qrow, g * G + i / HD, i % HD, 0.f);
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
    int* spg = reinterpret_cast<int*>(dsm + (size_t)a.combine_smem);  // (after the slots / combine area)
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
                    bulk_g2s_hint(kd + (size_t)(p - c0) * ROWB, kr, n * ROWB, &bar[slot], l2_evict_first());
                    bulk_g2s_hint(vd + (size_t)(p - c0) * ROWB, vr, n * ROWB, &bar[slot], l2_evict_first());
                }
                p += n;
            }
        } else if (rows > 0) {
            bulk_g2s_hint(kd, cache_row<CT>((CT*)a.kc, a, b, g, c0, HD), rows * ROWB, &bar[slot], l2_evict_first());
            bulk_g2s_hint(vd, cache_row<CT>((CT*)a.vc, a, b, g, c0, HD), rows * ROWB, &bar[slot], l2_evict_first());
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

    // queries of the group, rotated at position P and pre-scaled by 1/sqrt(hd). A deferred
    // QKV phase's columns are first finished into qs / kn / vn (then rotated in place);
    // otherwise they are read from qkv here.
    const float* cs = a.rope_cs + (size_t)P * HALF * 2;
    const float scale = 1.0f / sqrtf((float)HD);
    const bool own = t1 == P + 1;  // this item holds the row's own key
    const bool dq = a.qprev.active;
    if (dq) {
        load_qkv<HD, G>(a, qrow, g, own, &qs[0][0], kn, vn);
        __syncthreads();
    }
    const float* qrow_p = a.qkv + qrow * (size_t)((a.H + 2 * a.Hkv) * HD);
    // (two loops: in the one reading qkv no load may wait for an earlier iteration's store)
    if (dq) {
        for (int idx = t; idx < G * HALF; idx += blockDim.x) {
            const int j = idx / HALF, i = idx % HALF;
            const float x1 = qs[j][i], x2 = qs[j][i + HALF], c = cs[2 * i], sn = cs[2 * i + 1];
            qs[j][i] = (x1 * c - x2 * sn) * scale;
            qs[j][i + HALF] = (x2 * c + x1 * sn) * scale;
        }
    } else {
        for (int idx = t; idx < G * HALF; idx += blockDim.x) {
            const int j = idx / HALF, i = idx % HALF;
            const float* q = qrow_p + (size_t)(g * G + j) * HD;
            const float x1 = q[i], x2 = q[i + HALF], c = cs[2 * i], sn = cs[2 * i + 1];
            qs[j][i] = (x1 * c - x2 * sn) * scale;
            qs[j][i + HALF] = (x2 * c + x1 * sn) * scale;
        }
    }
    if (own) {  // rotate the row's own key and append k, v at slot P
        const float* kq = qrow_p + (size_t)a.H * HD + (size_t)g * HD;
        const float* vq = kq + (size_t)a.Hkv * HD;
        CT* krow = cache_row<CT>((CT*)a.kc, a, b, g, P, HD);
        CT* vrow = cache_row<CT>((CT*)a.vc, a, b, g, P, HD);
        if ((!krow || !vrow) && t == 0) atomicOr(a.status, ST_DEVICE);
        for (int i = t; i < HALF; i += blockDim.x) {
            const float x1 = dq ? kn[i] : kq[i], x2 = dq ? kn[i + HALF] : kq[i + HALF];
            const float c = cs[2 * i], sn = cs[2 * i + 1];
            const float r1 = x1 * c - x2 * sn, r2 = x2 * c + x1 * sn;
            kn[i] = r1;
            kn[i + HALF] = r2;
            if (krow) {
                Storage<CT>::store(krow, i, r1);
                Storage<CT>::store(krow, i + HALF, r2);
            }
        }
        for (int i = t; i < HD; i += blockDim.x) {
            const float x = dq ? vn[i] : vq[i];
            vn[i] = x;
            if (vrow) Storage<CT>::store(vrow, i, x);
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
        float* pp = a.part + (((size_t)b * a.H + g * G + hh) * a.n_split + s) * part_row<HD>();
        pp[dd] = v;
        if (dd == 0) { pp[HD] = M; pp[HD + 1] = L; }
    }
    // ---- the last active split of (b, g) combines all splits. Thread 0's acquire-release
    // add publishes the CTA's partial (ordered before it by the barrier) and, in the last
    // split, orders the combine's reads after every other split's.
    __syncthreads();
    if (t == 0) s_last = atom_add_acq_rel_gpu(&a.counters[b * a.Hkv + g], 1) == n_act - 1;
    __syncthreads();
    if (!s_last) return;
    const float* pb0 = a.part + ((size_t)b * a.H + g * G) * a.n_split * part_row<HD>();
    combine_splits<HD, G, false>(a, pb0, n_act, qrow, g * G, dsm, (size_t)a.combine_smem);
    if (t == 0) a.counters[b * a.Hkv + g] = 0;
}

// ---- tensor-core attention (bf16 caches, hd = 128, G = 1..8 query heads per KV head) ---------
// The same work items, chunk ownership, own-row append and split combine as attn_kernel;
// the per-chunk arithmetic runs on mma.sync (m16n8k16, bf16 operands, float32 accumulate)
// with the keys and the head dimensions as the long matrix sides:
//   S^T (32 keys x 8 heads) = K (32 x 128) . Q^T            2 key tiles x 8 k-steps
//   O^T (128 dims x 8 heads) += V^T (128 x 32) . P^T          8 dim tiles x 2 k-steps
// so a KV head's G <= 8 query heads fill the 8-wide side (with G = 1 seven columns idle: the
// products are still far cheaper than the CUDA-core kernel's shuffle reductions). Q and P enter as bf16 hi + lo
// pairs (two products each), which keeps scores and outputs at float32-level accuracy; K
// and V are bf16 in the cache already.
//   - Rows arrive by cp.async (16 bytes per lane, two rows per warp instruction, each lane
//     with its own address), so every row can go to its own place: 16-byte chunk c of row
//     r lands at chunk c ^ (r % 8), which puts the eight rows an ldmatrix phase reads into
//     eight different bank groups. Rows without a key are zero-filled by the copy itself.
//   - K and V of a chunk are separate copy groups: the next chunk's K rows are requested as
//     soon as S is formed and its V rows as soon as P.V is done, so each copy overlaps the
//     other half of the chunk's arithmetic.
//   - P^T changes fragment layout by shuffles within the warp.
//   - Softmax runs in base 2 (log2 e is folded into the query scale).
//   - The row's own key and value (position P, float32) enter as the first key of warp
//     0's online softmax.
constexpr uint32_t kTcHalfBytes = kChunkKeys * 256;  // the K (or V) rows of one chunk

// x0 -> bits 0..15, x1 -> bits 16..31, rounded to nearest even
__device__ __forceinline__ uint32_t bf16x2_rn(float x0, float x1) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(x1), "f"(x0));
    return r;
}

// (x0, x1) as bf16x2 hi + lo words: x = hi + lo to about 16 significant bits
__device__ __forceinline__ void split_pack(float x0, float x1, uint32_t& hi, uint32_t& lo) {
    hi = bf16x2_rn(x0, x1);
    lo = bf16x2_rn(x0 - __uint_as_float(hi << 16), x1 - __uint_as_float(hi & 0xFFFF0000u));
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr)
                 : "memory");
}

__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr)
                 : "memory");
}

// d += A B for one m16n8k16 tile (A row-major 16 x 16, B column-major 16 x 8)
__device__ __forceinline__ void mma_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// 16 bytes global -> shared, bypassing L1; src_bytes = 0 writes 16 zero bytes instead
// with an L2 cache policy (the cached prefix is read once per draft: l2_evict_first())
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes, uint64_t pol) {
    asm volatile("cp.async.cg.shared.global.L2::cache_hint [%0], [%1], 16, %2, %3;" ::"r"(dst), "l"(src), "r"(src_bytes),
                 "l"(pol)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

template <int G, bool DQ>
__global__ void __launch_bounds__(kAttnWarps * 32, 3) attn_tc_kernel(const AttnArgs a) {
    const LaunchStamp stamp(a.stamp);
    using CT = bf16_t;
    constexpr int HD = 128;
    constexpr int HALF = HD / 2;
    static_assert(kAttnWarps * 32 == HD, "one thread per head dimension (the own key and value)");
    constexpr uint32_t CB = kTcHalfBytes;
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ __align__(16) float qs[G][HD];
    __shared__ __align__(16) float kn[HD];
    __shared__ __align__(16) float vn[HD];
    __shared__ float wm[kAttnWarps][G], wl[kAttnWarps][G];
    __shared__ float s_own[G];  // the own key's score per head (base 2)
    __shared__ int s_last;

    const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    // (a commit launch handles row index pos_add of every sequence: its position is
    // prefix_len + pos_add, and sequences with fewer rows to commit have no work here)
    if (a.n_rows && a.pos_add >= a.n_rows[b]) {
        griddep_launch_dependents();
        return;
    }
    const int P = a.prefix_len[b] + a.pos_add;
    const size_t qrow = (size_t)b * a.row_stride + a.row_off;  // this row in qkv and out

    const bool valid = P >= 0 && P + 1 <= a.max_seq;
    if (!valid) {
        griddep_launch_dependents();
        griddep_wait();
        if (s == 0) {
            if (g == 0 && t == 0) atomicOr(a.status, ST_CAPACITY);
            for (int i = t; i < G * HD; i += blockDim.x) put_out<HD>(a, qrow, g * G + i / HD, i % HD, 0.f);
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
    const int tc = min(t1, P);  // cached keys [t0, tc); key P, when t1 > P, is the row's own
    const int nchunks = tc > t0 ? (tc - t0 + kChunkKeys - 1) / kChunkKeys : 0;

    unsigned char* kc = dsm + (size_t)warp * 2 * CB;  // this warp's 32 K rows, then its 32 V rows
    unsigned char* vc = kc + CB;
    // Paged caches: this item's page ids, read once into shared memory after the K/V rows
    // (-1 marks an invalid id)
    int* spg = reinterpret_cast<int*>(dsm + (size_t)a.combine_smem);  // (after the slots / combine area)
    const int pg0 = a.page_table ? t0 / a.page_size : 0;
    if (a.page_table) {
        const int npg = tc > t0 ? (tc - 1) / a.page_size - pg0 + 1 : 0;
        for (int i = t; i < npg; i += blockDim.x) {
            const int pg = a.page_table[(size_t)b * a.max_pages + pg0 + i];
            spg[i] = (pg < 0 || pg >= a.n_pages) ? -1 : pg;
        }
    }
    __syncthreads();  // page ids staged

    // Chunk j of this warp covers keys [c0, c0 + 32), c0 = t0 + (warp + 4 j) * 32; lane r
    // looks up row c0 + r. Returns 1 and the row's index in the cache (in rows of hd
    // elements) when it holds a cached key, 0 past the item's keys, -1 on an invalid page id.
    // (power-of-two page sizes take shifts instead of divisions)
    const int ps_shift = a.page_table && !(a.page_size & (a.page_size - 1)) ? __ffs(a.page_size) - 1 : -1;
    auto plan = [&](int j, uint32_t& ri) -> int {
        const int pos = t0 + (warp + kAttnWarps * j) * kChunkKeys + lane;
        ri = 0;  // rows without a key copy from row 0 with zero source bytes
        if (pos >= tc) return 0;
        if (a.page_table) {
            const int lp = ps_shift >= 0 ? pos >> ps_shift : pos / a.page_size;
            const int in = ps_shift >= 0 ? pos & (a.page_size - 1) : pos % a.page_size;
            const int pg = spg[lp - pg0];
            if (pg < 0) return -1;
            ri = (uint32_t)(((size_t)pg * a.Hkv + g) * a.page_size + in);
        } else {
            ri = (uint32_t)(((size_t)b * a.Hkv + g) * a.max_seq + pos);
        }
        return 1;
    };
    // One half (K or V) of a chunk as one copy group: warp instruction i moves rows 2 i and
    // 2 i + 1, lane l chunk l % 16 of row 2 i + l / 16 (row indices come from their lanes).
    // The swizzle c ^ (r % 8) repeats every four instructions.
    const int hrow = lane >> 4, cchunk = lane & 15;
    uint32_t xo[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) xo[k] = (uint32_t)(hrow * 256 + ((cchunk ^ ((2 * k + hrow) & 7)) << 4));
    const uint64_t kvpol = l2_evict_first();
    auto copy_half = [&](unsigned char* dst, const void* cache, uint32_t ri, uint32_t live) {
        const uint32_t d0 = smem_u32(dst);
        const unsigned char* src0 = (const unsigned char*)cache + cchunk * 16;
        const uint32_t lh = live >> hrow;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const uint32_t rr = __shfl_sync(0xffffffffu, ri, 2 * i + hrow);
            cp_async16(d0 + 2 * i * 256 + xo[i & 3], src0 + (size_t)rr * 256, (lh >> (2 * i)) & 1u ? 16u : 0u, kvpol);
        }
        cp_async_commit();
    };
    const int my_chunks = warp < nchunks ? (nchunks - warp + kAttnWarps - 1) / kAttnWarps : 0;
    uint32_t ri = 0, live = 0, bad = 0;  // lane's row index; the chunk's rows holding a key / on invalid pages
    // cached prefix rows are not written by the earlier kernels of this draft: copy the
    // first chunk before waiting for the QKV projection
    if (my_chunks > 0) {
        const int code = plan(0, ri);
        live = __ballot_sync(0xffffffffu, code > 0);
        bad = __ballot_sync(0xffffffffu, code < 0);
        copy_half(kc, a.kc, ri, live);
        copy_half(vc, a.vc, ri, live);
    }
    griddep_launch_dependents();
    griddep_wait();

    // queries of the group, rotated at position P and pre-scaled by log2(e) / sqrt(hd); the
    // item holding key P loads the row's own key and value with them (one round trip). A
    // deferred QKV phase's columns are first finished into qs / kn / vn (then rotated in
    // place); otherwise they are read from qkv here.
    const float* cs = a.rope_cs + (size_t)P * HALF * 2;
    const float scale = 1.4426950408889634f / sqrtf((float)HD);
    const bool own = t1 == P + 1;  // this item holds the row's own key
    constexpr bool dq = DQ;  // (a.qprev.active: a separate instantiation)
    if (dq) {
        load_qkv<HD, G>(a, qrow, g, own, &qs[0][0], kn, vn);
        __syncthreads();
    }
    const float* qrow_p = a.qkv + qrow * (size_t)((a.H + 2 * a.Hkv) * HD);
    const float* kq = qrow_p + (size_t)a.H * HD + (size_t)g * HD;
    const float* vq = kq + (size_t)a.Hkv * HD;
    float ok1 = 0.f, ok2 = 0.f, okc = 0.f, oks = 0.f, ov = 0.f;  // (blockDim.x == HD: one element each)
    if (own) {
        if (t < HALF) {
            ok1 = dq ? kn[t] : kq[t];
            ok2 = dq ? kn[t + HALF] : kq[t + HALF];
            okc = cs[2 * t];
            oks = cs[2 * t + 1];
        }
        ov = dq ? vn[t] : vq[t];
    }
    // (two loops: in the one reading qkv no load may wait for an earlier iteration's store)
    if (dq) {
        for (int idx = t; idx < G * HALF; idx += blockDim.x) {
            const int j = idx / HALF, i = idx % HALF;
            const float x1 = qs[j][i], x2 = qs[j][i + HALF], c = cs[2 * i], sn = cs[2 * i + 1];
            qs[j][i] = (x1 * c - x2 * sn) * scale;
            qs[j][i + HALF] = (x2 * c + x1 * sn) * scale;
        }
    } else {
        for (int idx = t; idx < G * HALF; idx += blockDim.x) {
            const int j = idx / HALF, i = idx % HALF;
            const float* q = qrow_p + (size_t)(g * G + j) * HD;
            const float x1 = q[i], x2 = q[i + HALF], c = cs[2 * i], sn = cs[2 * i + 1];
            qs[j][i] = (x1 * c - x2 * sn) * scale;
            qs[j][i + HALF] = (x2 * c + x1 * sn) * scale;
        }
    }
    if (own) {  // rotate the new key and append k, v at slot P
        CT* krow = cache_row<CT>((CT*)a.kc, a, b, g, P, HD);
        CT* vrow = cache_row<CT>((CT*)a.vc, a, b, g, P, HD);
        if ((!krow || !vrow) && t == 0) atomicOr(a.status, ST_DEVICE);
        if (t < HALF) {
            const float r1 = ok1 * okc - ok2 * oks, r2 = ok2 * okc + ok1 * oks;
            kn[t] = r1;
            kn[t + HALF] = r2;
            if (krow) {
                Storage<CT>::store(krow, t, r1);
                Storage<CT>::store(krow, t + HALF, r2);
            }
        }
        vn[t] = ov;
        if (vrow) Storage<CT>::store(vrow, t, ov);
    }
    __syncthreads();
    if (own)  // the own key's score per head: warp w takes heads w, w + 4
        for (int h = warp; h < G; h += kAttnWarps) {
            float v = 0.f;
#pragma unroll
            for (int i = lane; i < HD; i += 32) v = fmaf(qs[h][i], kn[i], v);
            v = warp_sum(v);
            if (lane == 0) s_own[h] = v;
        }
    __syncthreads();

    // Fragment ownership: gid = lane / 4, tig = lane % 4. Thread (gid, tig) holds Q^T's
    // B fragments for head gid (zero for gid >= G) and accumulates heads 2 tig and 2 tig + 1.
    const int gid = lane >> 2, tig = lane & 3;
    uint32_t qh[8][2], ql[8][2];  // k-step ks: dims 16 ks + 2 tig (+1) and 16 ks + 8 + 2 tig (+1)
#pragma unroll
    for (int ks = 0; ks < 8; ++ks)
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
            const int c = ks * 16 + hf * 8 + tig * 2;
            split_pack(gid < G ? qs[gid][c] : 0.f, gid < G ? qs[gid][c + 1] : 0.f, qh[ks][hf], ql[ks][hf]);
        }
    // Running state of heads 2 tig + e (base 2). Warp 0 of the item holding key P starts
    // from the row's own key and value (float32, unrounded) as its first key.
    const bool first = own && warp == 0;
    float m[2], l[2];
#pragma unroll
    for (int e = 0; e < 2; ++e) {
        m[e] = first ? s_own[min(2 * tig + e, G - 1)] : -INFINITY;
        l[e] = first && gid == 0 ? 1.f : 0.f;  // (one lane of the column holds the own key's share)
    }
    float o[8][4];  // dim tile mt: (16 mt + gid, heads 2 tig, 2 tig + 1), (16 mt + gid + 8, same heads)
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
        const float v0 = first ? vn[16 * mt + gid] : 0.f, v1 = first ? vn[16 * mt + gid + 8] : 0.f;
        o[mt][0] = o[mt][1] = v0;
        o[mt][2] = o[mt][3] = v1;
    }

    // ldmatrix addresses (chunk c of row r sits at chunk c ^ (r % 8), and r % 8 = lane % 8
    // for every row a lane addresses): K as the A operand, 16 keys x 16 dims per x4, lane l
    // naming row (l % 8) + 8 ((l / 8) % 2) at dims 8 (l / 16) ..; V^T through .trans, lane l
    // naming key 8 (l / 16) + l % 8 at dims 8 ((l / 8) % 2) ..
    const int sw = lane & 7;
    const uint32_t rowa = smem_u32(kc) + (uint32_t)(sw + 8 * ((lane >> 3) & 1)) * 256;
    const uint32_t rowv = smem_u32(vc) + (uint32_t)(8 * (lane >> 4) + sw) * 256;
    const int ca = lane >> 4, cv = (lane >> 3) & 1;
    // P^T's B fragments gather keys 2 tig and 2 tig + 1 of every 8 from lanes 4 (2 tig) +
    // gid / 2 and 4 (2 tig + 1) + gid / 2, value e = gid % 2 of theirs
    const int src0 = 4 * (2 * tig) + (gid >> 1), src1 = src0 + 4;
    const bool odd = gid & 1;
    for (int j = 0; j < my_chunks; ++j) {
        if (bad && lane == 0) atomicOr(a.status, ST_DEVICE);
        const bool more = j + 1 < my_chunks;
        uint32_t nri = 0, nlive = 0, nbad = 0;
        if (more) {
            const int code = plan(j + 1, nri);
            nlive = __ballot_sync(0xffffffffu, code > 0);
            nbad = __ballot_sync(0xffffffffu, code < 0);
        }
        // this chunk's K rows (groups in flight: K(j), V(j))
        cp_async_wait<1>();
        __syncwarp();
        // S^T = K Q^T; four independent accumulators (key tile x hi/lo)
        float sc[2][4];
        {
            float acc[4][4];
#pragma unroll
            for (int i = 0; i < 4; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
                const uint32_t col = (uint32_t)((2 * ks + ca) ^ sw) << 4;
                uint32_t a0[4], a1[4];
                ldsm_x4(rowa + col, a0);
                ldsm_x4(rowa + 16 * 256 + col, a1);
                mma_16816(acc[0], a0, qh[ks][0], qh[ks][1]);
                mma_16816(acc[1], a1, qh[ks][0], qh[ks][1]);
                mma_16816(acc[2], a0, ql[ks][0], ql[ks][1]);
                mma_16816(acc[3], a1, ql[ks][0], ql[ks][1]);
            }
#pragma unroll
            for (int mt = 0; mt < 2; ++mt)
#pragma unroll
                for (int i = 0; i < 4; ++i) sc[mt][i] = acc[mt][i] + acc[2 + mt][i];
        }
        __syncwarp();  // every lane's K reads are done: the K rows may be refilled
        if (more) copy_half(kc, a.kc, nri, nlive);
        // online softmax: head 2 tig + e sees keys 8 q + gid (q = 2 mt + hi) here and in the
        // 7 other lanes of its column (lanes tig, tig + 4, ...)
        bool kl[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) kl[q] = (live >> (8 * q + gid)) & 1u;
        float p[2][4], corr[2];
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            float mx = -INFINITY;
#pragma unroll
            for (int q = 0; q < 4; ++q)
                if (kl[q]) mx = fmaxf(mx, sc[q >> 1][2 * (q & 1) + e]);
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
            const float mn = fmaxf(m[e], mx);
            corr[e] = m[e] == mn ? 1.f : ex2_approx(m[e] - mn);  // (0 when m was -inf)
            // l[e] holds this lane's share of the sum (its keys); the column's lanes add
            // their shares once, after the last chunk
            float rs = 0.f;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float pv = kl[q] ? ex2_approx(sc[q >> 1][2 * (q & 1) + e] - mn) : 0.f;
                p[q >> 1][2 * (q & 1) + e] = pv;
                rs += pv;
            }
            l[e] = l[e] * corr[e] + rs;
            m[e] = mn;
        }
        // rescale the accumulators only when some head's maximum moved
        if (__any_sync(0xffffffffu, corr[0] != 1.f || corr[1] != 1.f)) {
#pragma unroll
            for (int mt = 0; mt < 8; ++mt) {
                o[mt][0] *= corr[0];
                o[mt][1] *= corr[1];
                o[mt][2] *= corr[0];
                o[mt][3] *= corr[1];
            }
        }
        // P^T's B fragments: word w[q][e] = key 8 q + gid of head 2 tig + e as bf16 (hi, lo);
        // k-step kk, half hf takes keys 16 kk + 8 hf + 2 tig (+1) of head gid
        uint32_t w[4][2];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            uint32_t hi, lo;
            split_pack(p[q >> 1][2 * (q & 1)], p[q >> 1][2 * (q & 1) + 1], hi, lo);
            w[q][0] = __byte_perm(hi, lo, 0x5410);
            w[q][1] = __byte_perm(hi, lo, 0x7632);
        }
        uint32_t pb[4][2];  // [q = 2 kk + hf][hi / lo]
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint32_t x0 = __shfl_sync(0xffffffffu, w[q][0], src0), y0 = __shfl_sync(0xffffffffu, w[q][1], src0);
            const uint32_t x1 = __shfl_sync(0xffffffffu, w[q][0], src1), y1 = __shfl_sync(0xffffffffu, w[q][1], src1);
            const uint32_t v0 = odd ? y0 : x0, v1 = odd ? y1 : x1;
            pb[q][0] = __byte_perm(v0, v1, 0x5410);
            pb[q][1] = __byte_perm(v0, v1, 0x7632);
        }
        // this chunk's V rows (groups in flight: V(j), and K(j + 1) unless this is the last)
        if (more) cp_async_wait<1>();
        else cp_async_wait<0>();
        __syncwarp();
        // O^T += V^T P^T, four dim tiles at a time: each accumulator's two products are four
        // MMAs apart
#pragma unroll
        for (int kk = 0; kk < 2; ++kk)
#pragma unroll
            for (int mg = 0; mg < 2; ++mg) {
                uint32_t af[4][4];
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    ldsm_x4_trans(rowv + kk * 16 * 256 + ((uint32_t)((2 * (4 * mg + i) + cv) ^ sw) << 4), af[i]);
#pragma unroll
                for (int i = 0; i < 4; ++i) mma_16816(o[4 * mg + i], af[i], pb[2 * kk][0], pb[2 * kk + 1][0]);
#pragma unroll
                for (int i = 0; i < 4; ++i) mma_16816(o[4 * mg + i], af[i], pb[2 * kk][1], pb[2 * kk + 1][1]);
            }
        __syncwarp();  // every lane's V reads are done
        if (more) copy_half(vc, a.vc, nri, nlive);
        live = nlive;
        bad = nbad;
    }

    // the sums of exp over each head's keys: add the shares of the column's 8 lanes
#pragma unroll
    for (int e = 0; e < 2; ++e) {
        l[e] += __shfl_xor_sync(0xffffffffu, l[e], 4);
        l[e] += __shfl_xor_sync(0xffffffffu, l[e], 8);
        l[e] += __shfl_xor_sync(0xffffffffu, l[e], 16);
    }
    // ---- merge the warps into this split's partial per head (every copy group has been
    // waited for: the K/V rows are free and hold the warps' accumulators)
    float (*wacc)[G][HD] = reinterpret_cast<float (*)[G][HD]>(dsm);
    __syncthreads();
#pragma unroll
    for (int e = 0; e < 2; ++e) {
        const int h = 2 * tig + e;
        if (h < G) {
#pragma unroll
            for (int mt = 0; mt < 8; ++mt) {
                wacc[warp][h][16 * mt + gid] = o[mt][e];
                wacc[warp][h][16 * mt + gid + 8] = o[mt][2 + e];
            }
            if (gid == 0) {
                wm[warp][h] = m[e];
                wl[warp][h] = l[e];
            }
        }
    }
    __syncthreads();
    for (int idx = t; idx < G * HD; idx += blockDim.x) {
        const int hh = idx / HD, dd = idx % HD;
        float M = wm[0][hh];
        for (int w = 1; w < kAttnWarps; ++w) M = fmaxf(M, wm[w][hh]);
        float v = 0.f, L = 0.f;
        for (int w = 0; w < kAttnWarps; ++w) {
            if (wm[w][hh] == -INFINITY) continue;
            const float f = exp2f(wm[w][hh] - M);
            v = fmaf(f, wacc[w][hh][dd], v);
            L = fmaf(f, wl[w][hh], L);
        }
        float* pp = a.part + (((size_t)b * a.H + g * G + hh) * a.n_split + s) * part_row<HD>();
        pp[dd] = v;
        if (dd == 0) { pp[HD] = M; pp[HD + 1] = L; }
    }
    // ---- the last active split of (b, g) combines all splits. Thread 0's acquire-release
    // add publishes the CTA's partial (ordered before it by the barrier) and, in the last
    // split, orders the combine's reads after every other split's.
    __syncthreads();
    if (t == 0) s_last = atom_add_acq_rel_gpu(&a.counters[b * a.Hkv + g], 1) == n_act - 1;
    __syncthreads();
    if (!s_last) return;
    const float* pb0 = a.part + ((size_t)b * a.H + g * G) * a.n_split * part_row<HD>();
    combine_splits<HD, G, true>(a, pb0, n_act, qrow, g * G, dsm, (size_t)a.combine_smem);
    if (t == 0) a.counters[b * a.Hkv + g] = 0;
}

// Keys per work item: aim at ~8 CTAs per SM over all (sequence, KV head) pairs, in whole
// multiples of one chunk per warp (128 keys), so that every warp of a CTA has work. About
// three CTAs are resident per SM, so ragged prefixes leave several waves of items that the
// block scheduler balances; the last split's combine still has few partials to read.
int attn_split(int B, int Hkv, int max_seq, const DeviceInfo& dev) {
    constexpr int unit = kAttnWarps * kChunkKeys;
    const int items = B * Hkv;
    int per = (8 * dev.num_sms + items - 1) / items;  // splits per (sequence, KV head)
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

// bf16 at hd 128 runs on the tensor-core kernel unless FE_DRAFT_ATTN_TC=0 selects
// the CUDA-core kernel (kept for comparison)
static bool attn_tc_enabled() {
    const char* e = getenv("FE_DRAFT_ATTN_TC");
    return !(e && e[0] == '0');
}

// The combine's shared memory: the K/V slots (`slots` bytes), grown to hold every split's
// partial rows at once (one staging pass) when that fits beside the page ids within the
// kernel's limit (slots + kAttnPageSmem); the page ids then follow it.
template <int HD, int G>
static size_t combine_bytes(const AttnArgs& a, size_t slots, size_t pg) {
    const size_t all = (size_t)G * a.n_split * (part_row<HD>() + 1) * sizeof(float);
    const size_t cap = slots + (size_t)kAttnPageSmem - pg;
    return all <= slots ? slots : (all <= cap ? (all + 15) & ~(size_t)15 : slots);
}

template <typename CT, int HD, int G>
static cudaError_t launch_g(const AttnArgs& a0, cudaStream_t st) {
    AttnArgs a = a0;
    const int S = attn_slots(a.split, HD, sizeof(CT));
    const size_t pg = attn_page_ints(a) * sizeof(int);
    if (pg > (size_t)kAttnPageSmem) return cudaErrorInvalidValue;
    if constexpr (sizeof(CT) == 2 && HD == 128) {
        if (attn_tc_enabled()) {
            const size_t slots = (size_t)kAttnWarps * 2 * kTcHalfBytes;
            a.combine_smem = (int)combine_bytes<HD, G>(a, slots, pg);
            return launch_k(a.qprev.active ? attn_tc_kernel<G, true> : attn_tc_kernel<G, false>,
                            dim3(a.n_split, a.Hkv, a.B), dim3(kAttnWarps * 32),
                            (size_t)a.combine_smem + pg, st, a.pdl, a);
        }
    }
    const size_t slots = attn_smem(HD, sizeof(CT), S);
    a.combine_smem = (int)combine_bytes<HD, G>(a, slots, pg);
    dim3 grid(a.n_split, a.Hkv, a.B);
    return launch_k(attn_kernel<CT, HD, G>, grid, dim3(kAttnWarps * 32), (size_t)a.combine_smem + pg, st, a.pdl, a, S);
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
    for (auto k : {attn_tc_kernel<1, false>, attn_tc_kernel<2, false>, attn_tc_kernel<4, false>,
                   attn_tc_kernel<8, false>, attn_tc_kernel<1, true>, attn_tc_kernel<2, true>,
                   attn_tc_kernel<4, true>, attn_tc_kernel<8, true>})
        if ((e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)(kAttnWarps * 2 * kTcHalfBytes) + kAttnPageSmem)) != cudaSuccess)
            return e;
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

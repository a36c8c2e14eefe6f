// Weight-streaming core shared by every matrix-vector phase of the drafter.
//
// At batch 1 each phase of the cascade (Eq. 1 FCs, the QKV / O / gate-up / down
// projections of every layer L_i in Eq. 2, the LM head of Sec. 2.1) reads a weight
// matrix once and does 2 flops per weight: the phases are bound by HBM bandwidth, not
// by arithmetic. The CTA is built around keeping HBM busy with as little consumer
// overhead as possible:
//
//   - Weights are tile-packed at init (fe_pack.cu): each matrix is cut into groups of 4
//     rows, and each group into K-slices of kKS columns; the 4 x width block of one
//     (group, slice) — a tile, at most 8 KB — is stored contiguously, so every copy is
//     one contiguous bulk transfer. A CTA owns a contiguous range of groups, i.e. a
//     contiguous range of tiles.
//   - Every warp runs its own pipeline: warp w takes tiles w, w+8, w+16, ... of the CTA's
//     range; its lane 0 issues cp.async.bulk (TMA) copies into the warp's own D slots,
//     each slot completing on its own mbarrier, and refills a slot as soon as the warp
//     has read it. No warp ever waits for another inside the stream.
//   - A lane multiplies 16-byte column vectors of all 4 rows of a tile by the activations
//     X (float32 in shared memory for the whole phase, staged once with a fused
//     prologue), so each X vector is reused for 4 weight rows. When a warp moves to
//     another row group it reduces its 4 x BT partial sums across lanes (a transposing
//     shuffle reduction) into its own slot of a per-chunk buffer. Every kChunk groups the
//     CTA synchronises once, and the phase's epilogue combines the 8 warps' slots.
//
// Measured on GB300 for a 283 MB bf16 matrix: 6.25 TB/s with compute, against 6.46 TB/s
// for the same copies with no compute (one shared producer and a CTA-wide barrier per
// row group reached 4.9 TB/s).
//
// Accumulation is float32 FMA on CUDA cores: at 1..8 activation rows the tensor pipe
// would idle, and this keeps fp32 weights (the small parity workload) on exact fp32
// arithmetic, never TF32.
#pragma once

#include "fe_common.cuh"

namespace fe {

constexpr int kWarps = 8;
constexpr int kStreamThreads = kWarps * 32;  // 256
constexpr int kGroupRows = 4;                // weight rows per group
constexpr int kTileBytes = 8192;             // 4 rows x 2 KB
constexpr int kChunk = 32;                   // row groups per epilogue round (BT <= 2)

// Row groups per epilogue round for BT activation rows: the per-warp partial sums of a
// chunk take kWarps * 4 * BT floats per group, so larger BT gets shorter chunks.
__host__ __device__ constexpr int chunk_groups(int BT) { return BT >= 8 ? 8 : BT >= 4 ? 16 : kChunk; }
constexpr int kMaxSlots = 3;                 // pipeline depth per warp

template <typename WT>
struct StreamGeom {
    static constexpr int kES = Storage<WT>::kBytes;
    static constexpr int kVec = Vec16<WT>::kN;                   // elements per 16 B
    static constexpr int kKS = kTileBytes / (kGroupRows * kES);  // columns per full slice
};

// Element offset of tile (group g, slice s) in a tile-packed [ceil(M/4)*4, K] matrix.
template <typename WT>
__host__ __device__ __forceinline__ int64_t tile_offset(int g, int s, int K) {
    return (int64_t)g * kGroupRows * K + (int64_t)s * kGroupRows * StreamGeom<WT>::kKS;
}

struct StreamSmem {
    unsigned char* ring;  // [kWarps][D][kTileBytes] (128-byte aligned)
    float* X;             // [xrows][Kpad] activations
    float* red;           // [chunk_groups(BT)][kWarps][4 * BT] per-warp partial sums of the current chunk
    uint64_t* full;       // [kWarps][D]
    int* abort;           // set when any wait of this CTA gave up
};

// Bytes of dynamic shared memory a streaming CTA needs (before any epilogue extras).
__host__ __device__ inline size_t stream_smem_bytes(int D, int xrows, int Kpad, int BT) {
    size_t b = (size_t)kWarps * D * kTileBytes;
    b += (size_t)xrows * Kpad * sizeof(float);
    b += (size_t)chunk_groups(BT) * kWarps * kGroupRows * BT * sizeof(float);
    b = (b + 15) & ~(size_t)15;
    b += (size_t)kWarps * D * sizeof(uint64_t) + 16;
    return b;
}

__device__ inline StreamSmem carve_stream_smem(unsigned char* smem, int D, int xrows, int Kpad, int BT) {
    StreamSmem s;
    s.ring = smem;
    s.X = (float*)(smem + (size_t)kWarps * D * kTileBytes);
    s.red = s.X + (size_t)xrows * Kpad;
    size_t off = (size_t)kWarps * D * kTileBytes +
                 ((size_t)xrows * Kpad + (size_t)chunk_groups(BT) * kWarps * kGroupRows * BT) * sizeof(float);
    off = (off + 15) & ~(size_t)15;
    s.full = (uint64_t*)(smem + off);
    s.abort = (int*)(s.full + kWarps * D);
    return s;
}

// Wait on a phase of `bar`; gives up when the CTA's abort flag is raised or after the
// wall-clock budget (then raises the flag and records ST_TIMEOUT). With sleep_ns > 0 the
// thread sleeps (up to sleep_ns per try) instead of spinning.
__device__ __forceinline__ bool mbar_wait_abortable(uint64_t* bar, uint32_t parity, int* status, int* abort,
                                                    uint32_t sleep_ns = 0) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (sleep_ns ? mbar_try_wait_sleep(bar, parity, sleep_ns) : mbar_try_wait(bar, parity)) return true;
        if (*(volatile int*)abort) return false;
        if ((int64_t)(globaltimer_ns() - t0) > kWaitBudgetNs) {
            atomicOr(status, ST_TIMEOUT);
            *(volatile int*)abort = 1;
            return false;
        }
    }
}

// Transposing warp reduction of V = 4 * BT values per lane: afterwards lane l holds, in
// v[0], the warp-wide sum of value index (l >> (5 - log2 V)). V - 1 + 5 - log2(V)
// shuffles instead of 5 V.
template <int V>
struct WarpMultiSum {
    template <int N, int O>
    __device__ __forceinline__ static void step(float* v, int lane) {
        if constexpr (N > 1) {
            constexpr int H = N / 2;
            const bool upper = (lane & O) != 0;
#pragma unroll
            for (int i = 0; i < H; ++i) {
                const float send = upper ? v[i] : v[i + H];
                const float keep = upper ? v[i + H] : v[i];
                v[i] = keep + __shfl_xor_sync(0xffffffffu, send, O);
            }
            step<H, O / 2>(v, lane);
        } else {
#pragma unroll
            for (int o = O; o >= 1; o >>= 1) v[0] += __shfl_xor_sync(0xffffffffu, v[0], o);
        }
    }
    __device__ __forceinline__ static void run(float* v, int lane) { step<V, 16>(v, lane); }
    static constexpr int kLog = V >= 32 ? 5 : V >= 16 ? 4 : V >= 8 ? 3 : V >= 4 ? 2 : V >= 2 ? 1 : 0;
    // which lanes hold a result, and for which value index
    __device__ __forceinline__ static bool owner(int lane) { return (lane & ((32 >> kLog) - 1)) == 0; }
    __device__ __forceinline__ static int index(int lane) { return lane >> (5 - kLog); }
};

// Value of (row r of group g, batch column b) of the current chunk: the sum of the 8 warps.
template <int BT>
__device__ __forceinline__ float chunk_value(const float* red, int g_in_chunk, int r, int b) {
    const float* p = red + (size_t)g_in_chunk * kWarps * kGroupRows * BT + r * BT + b;
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) v += p[w * kGroupRows * BT];
    return v;
}

// One tile: 4 weight rows x `width` columns (rows at stride `width`) starting at column kc.
template <typename WT, int BT>
__device__ __forceinline__ void tile_compute(const unsigned char* st, const float* X, int Kpad, int kc, int width,
                                             int nb, int lane, float (&acc)[kGroupRows][BT]) {
    using G = StreamGeom<WT>;
    constexpr int V = G::kVec;
    const size_t rs = (size_t)width * G::kES;
    const int nv = width / V;
    for (int v = lane; v < nv; v += 32) {
        float f[kGroupRows][V];
#pragma unroll
        for (int r = 0; r < kGroupRows; ++r)
            Vec16<WT>::widen(*reinterpret_cast<const uint4*>(st + r * rs + (size_t)v * 16), f[r]);
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            if (b < nb) {
                const float4* xp = reinterpret_cast<const float4*>(X + (size_t)b * Kpad + kc + (size_t)v * V);
                float xv[V];
#pragma unroll
                for (int q = 0; q < V / 4; ++q) {
                    const float4 x4 = xp[q];
                    xv[4 * q] = x4.x; xv[4 * q + 1] = x4.y; xv[4 * q + 2] = x4.z; xv[4 * q + 3] = x4.w;
                }
#pragma unroll
                for (int r = 0; r < kGroupRows; ++r)
#pragma unroll
                    for (int j = 0; j < V; ++j) acc[r][b] = fmaf(f[r][j], xv[j], acc[r][b]);
            }
        }
    }
}

// Stage activations X[b][k] (b < nb, k < K) into shared memory (see Prologue).
struct ProParams {
    int pro;
    const void* x;
    int ldx;
    const void* gamma;
    float eps;
    const void* embed;
    const int* tok;
    int d_split;
    int vocab;
};

// Copy n values of src (storage type T, global) widened to float into dst (shared); returns
// this thread's sum of squares when SQ. Uses 16-byte loads with up to 8 in flight per
// thread when both ends are 16-byte aligned and n is a whole number of vectors: the
// activations are read after griddep_wait(), and a latency-bound prologue would leave the
// weight stream idle once the first copies have landed. src may have been written by the
// previous kernel: it is read through L2 (ld.global.cg) and is not a __restrict__ pointer,
// so no load can be treated as invariant and moved above griddep_wait().
template <typename T, bool SQ>
__device__ __forceinline__ float stage_span(const T* src, float* dst, int n) {
    constexpr int V = Vec16<T>::kN;
    constexpr int U = 8;
    float ss = 0.f;
    const bool vec = ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15) == 0 && n % V == 0;
    if (vec) {
        const uint4* s4 = reinterpret_cast<const uint4*>(src);
        const int nv = n / V;
        for (int base = threadIdx.x; base < nv; base += kStreamThreads * U) {
            uint4 r[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int i = base + u * kStreamThreads;
                r[u] = i < nv ? __ldcg(s4 + i) : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int i = base + u * kStreamThreads;
                if (i < nv) {
                    float f[V];
                    Vec16<T>::widen(r[u], f);
                    if (SQ) {
#pragma unroll
                        for (int j = 0; j < V; ++j) ss = fmaf(f[j], f[j], ss);
                    }
                    float4* d4 = reinterpret_cast<float4*>(dst + (size_t)i * V);
#pragma unroll
                    for (int q = 0; q < V / 4; ++q) d4[q] = make_float4(f[4 * q], f[4 * q + 1], f[4 * q + 2], f[4 * q + 3]);
                }
            }
        }
    } else {
        for (int k = threadIdx.x; k < n; k += kStreamThreads) {
            const float v = Storage<T>::load(src, k);
            dst[k] = v;
            if (SQ) ss = fmaf(v, v, ss);
        }
    }
    return ss;
}

// dst[k] = dst[k] * rs * gamma[k] for k < n (dst shared, gamma global storage type), with
// the gains read as 16-byte vectors, 8 in flight per thread, when aligned.
template <typename T>
__device__ __forceinline__ void scale_span(const T* __restrict__ gamma, float* dst, int n, float rs) {
    constexpr int V = Vec16<T>::kN;
    constexpr int U = 8;
    const bool vec = ((reinterpret_cast<uintptr_t>(gamma) | reinterpret_cast<uintptr_t>(dst)) & 15) == 0 && n % V == 0;
    if (vec) {
        const uint4* g4 = reinterpret_cast<const uint4*>(gamma);
        const int nv = n / V;
        for (int base = threadIdx.x; base < nv; base += kStreamThreads * U) {
            uint4 r[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int i = base + u * kStreamThreads;
                r[u] = i < nv ? g4[i] : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int i = base + u * kStreamThreads;
                if (i < nv) {
                    float f[V];
                    Vec16<T>::widen(r[u], f);
                    float* d = dst + (size_t)i * V;
#pragma unroll
                    for (int j = 0; j < V; ++j) d[j] = d[j] * rs * f[j];
                }
            }
        }
    } else {
        for (int k = threadIdx.x; k < n; k += kStreamThreads) dst[k] = dst[k] * rs * Storage<T>::load(gamma, k);
    }
}

// The part of the prologue that reads nothing an earlier kernel writes, for a caller to run
// before griddep_wait(): the RMSNorm gains, widened into X (the rows' activations then need
// one read of x and one pass over shared memory), or the token-embedding half of a
// concatenation. Returns true when it ran; stage_activations must then get pre = true.
// (For RMSNorm only when a row fits the single-round register path: K <= 8192, aligned.)
template <typename WT>
__device__ bool stage_pre(const ProParams& p, int K, float* X, int Kpad, int b0, int nb, int* status) {
    const int t = threadIdx.x;
    if (p.pro == PRO_RMSNORM) {
        if (K % 4 != 0 || K / 4 > kStreamThreads * 8 || p.ldx % 4 != 0 ||
            (reinterpret_cast<uintptr_t>(p.x) & 15) != 0)
            return false;
        for (int b = 0; b < nb; ++b) stage_span<WT, false>((const WT*)p.gamma, X + (size_t)b * Kpad, K);
        return true;
    }
    if (p.pro == PRO_CONCAT_EMB) {
        const int de = K - p.d_split;
        for (int b = 0; b < nb; ++b) {
            float* Xb = X + (size_t)b * Kpad;
            int tok = p.tok[b0 + b];
            if (tok < 0 || tok >= p.vocab) {
                if (t == 0) atomicOr(status, ST_DEVICE);
                for (int k = t; k < de; k += kStreamThreads) Xb[p.d_split + k] = 0.f;
            } else {
                stage_span<WT, false>((const WT*)p.embed + (size_t)tok * de, Xb + p.d_split, de);
            }
        }
        return true;
    }
    return false;
}

template <typename WT>
__device__ void stage_activations(const ProParams& p, int K, float* X, int Kpad, int b0, int nb, int* status,
                                  float* scratch /* >= kWarps floats */, bool pre = false) {
    const int t = threadIdx.x;
    for (int b = 0; b < nb; ++b) {
        const int row = b0 + b;
        float* Xb = X + (size_t)b * Kpad;
        if (pre && p.pro == PRO_CONCAT_EMB) {  // the embedding half is in place
            stage_span<float, false>((const float*)p.x + (size_t)row * p.ldx, Xb, p.d_split);
        } else if (pre && p.pro == PRO_RMSNORM) {
            // Xb holds gamma: one round of up to 8 float4 loads of x per thread, the sum of
            // squares in the same order as stage_span, then Xb = (x * rs) * gamma in place
            const float4* x4 = reinterpret_cast<const float4*>((const float*)p.x + (size_t)row * p.ldx);
            const int nv = K / 4;
            float4 r[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int i = t + u * kStreamThreads;
                r[u] = i < nv ? __ldcg(x4 + i) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
            float ss = 0.f;
#pragma unroll
            for (int u = 0; u < 8; ++u)
                if (t + u * kStreamThreads < nv) {
                    ss = fmaf(r[u].x, r[u].x, ss);
                    ss = fmaf(r[u].y, r[u].y, ss);
                    ss = fmaf(r[u].z, r[u].z, ss);
                    ss = fmaf(r[u].w, r[u].w, ss);
                }
            ss = warp_sum(ss);
            if ((t & 31) == 0) scratch[t >> 5] = ss;
            __syncthreads();
            float tot = 0.f;
#pragma unroll
            for (int w = 0; w < kWarps; ++w) tot += scratch[w];
            const float rs = 1.0f / sqrtf(tot / (float)K + p.eps);
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int i = t + u * kStreamThreads;
                if (i < nv) {
                    float4* d = reinterpret_cast<float4*>(Xb) + i;
                    const float4 gm = *d;
                    *d = make_float4(r[u].x * rs * gm.x, r[u].y * rs * gm.y, r[u].z * rs * gm.z, r[u].w * rs * gm.w);
                }
            }
            __syncthreads();  // scratch reuse by the next row
        } else if (p.pro == PRO_F32) {
            stage_span<float, false>((const float*)p.x + (size_t)row * p.ldx, Xb, K);
        } else if (p.pro == PRO_STORAGE) {
            stage_span<WT, false>((const WT*)p.x + (size_t)row * p.ldx, Xb, K);
        } else if (p.pro == PRO_CONCAT_EMB) {
            int tok = p.tok[row];
            if (tok < 0 || tok >= p.vocab) {
                if (t == 0) atomicOr(status, ST_DEVICE);
                tok = -1;
            }
            const int de = K - p.d_split;
            stage_span<float, false>((const float*)p.x + (size_t)row * p.ldx, Xb, p.d_split);
            if (tok >= 0)
                stage_span<WT, false>((const WT*)p.embed + (size_t)tok * de, Xb + p.d_split, de);
            else
                for (int k = t; k < de; k += kStreamThreads) Xb[p.d_split + k] = 0.f;
        } else {  // PRO_RMSNORM
            float ss = stage_span<float, true>((const float*)p.x + (size_t)row * p.ldx, Xb, K);
            ss = warp_sum(ss);
            if ((t & 31) == 0) scratch[t >> 5] = ss;
            __syncthreads();
            float tot = 0.f;
#pragma unroll
            for (int w = 0; w < kWarps; ++w) tot += scratch[w];
            const float rs = 1.0f / sqrtf(tot / (float)K + p.eps);
            scale_span<WT>((const WT*)p.gamma, Xb, K, rs);
            __syncthreads();  // scratch reuse by the next row
        }
    }
    // zero the padding columns so vector loads past K read zeros
    for (int b = 0; b < nb; ++b)
        for (int k = K + t; k < Kpad; k += kStreamThreads) X[(size_t)b * Kpad + k] = 0.f;
}

// Item i of a CTA's range is tile (g, ks). With the activations staged in one pass the
// items run group-major (the n0 = nks slices of group g0, then of g0 + 1, ...). When X holds
// only the first n0 < nks slices' columns at a time, they run pass-major: slices [0, n0) of
// every group, then slices [n0, nks) of every group (items0 = groups x n0 items first).
__device__ __forceinline__ void stream_item(int i, int g0, int nks, int n0, int items0, int& g, int& ks) {
    if (i < items0) {
        g = g0 + i / n0;
        ks = i % n0;
    } else {
        const int n1 = nks - n0, i1 = i - items0;
        g = g0 + i1 / n1;
        ks = n0 + i1 % n1;
    }
}

// Issue copy i (the warp's item i of the CTA's tile range) into the warp's slot.
template <typename WT>
__device__ __forceinline__ void stream_issue(const unsigned char* Wt, int K, int g0, int nks, int n0, int items0,
                                             int i, int slot, uint64_t* full, unsigned char* ring) {
    using G = StreamGeom<WT>;
    int g, ks;
    stream_item(i, g0, nks, n0, items0, g, ks);
    const uint32_t bytes = (uint32_t)kGroupRows * (uint32_t)min(G::kKS, K - ks * G::kKS) * G::kES;
    mbar_arrive_expect_tx(&full[slot], bytes);
    // weights are read once per draft: evict first, keeping L2 for the activations
    bulk_g2s_hint(ring + (size_t)slot * kTileBytes, Wt + tile_offset<WT>(g, ks, K) * G::kES, bytes, &full[slot],
                  l2_evict_first());
}

// First half of a stream: initialise the per-warp barriers and issue every warp's first D
// copies. Touches only the (read-only) weights, so it may run before griddep_wait().
// Must be called by all 256 threads; returns the number of copies this warp issued.
// `again`: a later stream of the same CTA (persistent kernel): the barriers are retired
// first (the previous stream consumed every copy) and the abort flag is kept. `n0`: slices
// per activation pass (0: one pass over all of K; see stream_item).
template <typename WT>
__device__ int stream_begin(const unsigned char* Wt, int K, int g0, int g1, StreamSmem& s, int D,
                            bool again = false, int n0 = 0) {
    using G = StreamGeom<WT>;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nks = (K + G::kKS - 1) / G::kKS;
    const int total = (g1 - g0) * nks;
    if (n0 <= 0 || n0 > nks) n0 = nks;
    const int items0 = (g1 - g0) * n0;
    uint64_t* full = s.full + warp * D;
    unsigned char* ring = s.ring + (size_t)warp * D * kTileBytes;
    int issued = 0;
    if (lane == 0) {
        for (int d = 0; d < D; ++d) {
            if (again) mbar_inval(&full[d]);
            mbar_init(&full[d], 1);
        }
        if (warp == 0 && !again) *s.abort = 0;
        mbar_fence_init();
        for (int j = 0; j < D && warp + kWarps * j < total; ++j, ++issued)
            stream_issue<WT>(Wt, K, g0, nks, n0, items0, warp + kWarps * j, j, full, ring);
    }
    return issued;
}

// Second half, the main loop: stream the row groups [g0, g1) of the tile-packed W through
// the per-warp pipelines. Must be called by all 256 threads after X is staged. Calls
// epi.chunk(cg0, cg1, red) on all threads once per chunk of up to kChunk groups; the
// epilogue reads values with chunk_value<BT>(red, g - cg0, r, b). `issued` is
// stream_begin's return value. Two activation
// passes (n0 > 0, pass1 set): X holds columns [0, n0 kKS) at first; once every warp is
// past its pass-0 items the CTA stages columns [n0 kKS, K) in their place (pass1 gives
// that prologue; plain float32 or storage-type rows only) and the pass-1 items read them.
// The caller guarantees that the CTA's groups fit one chunk (g1 - g0 <= chunk_groups(BT)),
// so the epilogue runs once, after both passes, and every partial sum of a group, from
// either pass, lands in its warp's slot of the chunk buffer.
template <typename WT, int BT, typename Epi>
__device__ void stream_run(const unsigned char* Wt, int K, int g0, int g1, StreamSmem& s, int D, int Kpad, int nb,
                           int* status, Epi& epi, int issued, int n0 = 0, const ProParams* pass1 = nullptr,
                           int b0 = 0) {
    using G = StreamGeom<WT>;
    using R = WarpMultiSum<kGroupRows * BT>;
    constexpr int RV = kGroupRows * BT;
    constexpr int CH = chunk_groups(BT);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nks = (K + G::kKS - 1) / G::kKS;
    const int total = (g1 - g0) * nks;
    if (n0 <= 0 || n0 > nks || !pass1) n0 = nks;
    const int items0 = (g1 - g0) * n0;
    const int kx0 = n0 * G::kKS;  // the first column of pass 1
    bool crossed = n0 == nks;
    uint64_t* full = s.full + warp * D;
    unsigned char* ring = s.ring + (size_t)warp * D * kTileBytes;

    for (int i = threadIdx.x; i < CH * kWarps * RV; i += kStreamThreads) s.red[i] = 0.f;
    __syncthreads();
    auto issue = [&](int i, int slot) { stream_issue<WT>(Wt, K, g0, nks, n0, items0, i, slot, full, ring); };

    float acc[kGroupRows][BT];
#pragma unroll
    for (int r = 0; r < kGroupRows; ++r)
#pragma unroll
        for (int b = 0; b < BT; ++b) acc[r][b] = 0.f;
    int cur_g = -1;
    int chunk_end = g0 + CH;
    for (int j = 0;; ++j) {
        const int i = warp + kWarps * j;
        int g = g1, ks = 0;
        if (i < total) stream_item(i, g0, nks, n0, items0, g, ks);
        if (g != cur_g && cur_g >= 0) {  // leaving a group: fold this warp's partials into the chunk buffer
            R::run(&acc[0][0], lane);
            if (R::owner(lane)) s.red[((size_t)(cur_g - chunk_end + CH) * kWarps + warp) * RV + R::index(lane)] += acc[0][0];
#pragma unroll
            for (int r = 0; r < kGroupRows; ++r)
#pragma unroll
                for (int b = 0; b < BT; ++b) acc[r][b] = 0.f;
        }
        // every warp crosses into pass 1 once (before any chunk boundary: all groups are
        // in one chunk then)
        if (!crossed && i >= items0) {
            crossed = true;
            __syncthreads();  // no warp reads pass-0 columns any more
            ProParams p1 = *pass1;
            p1.x = (const unsigned char*)p1.x + (size_t)kx0 * (p1.pro == PRO_F32 ? sizeof(float) : (size_t)G::kES);
            stage_activations<WT>(p1, K - kx0, s.X, Kpad, b0, nb, status, nullptr);
            __syncthreads();
        }
        // every warp passes every chunk boundary once: when its next group lies beyond the
        // chunk, or (for the last, possibly partial, chunks) when its items are exhausted
        while ((g >= chunk_end || i >= total) && chunk_end - CH < g1) {
            __syncthreads();
            epi.chunk(chunk_end - CH, min(chunk_end, g1), s.red);
            __syncthreads();
            for (int q = threadIdx.x; q < CH * kWarps * RV; q += kStreamThreads) s.red[q] = 0.f;
            __syncthreads();
            chunk_end += CH;
        }
        if (i >= total) break;
        cur_g = g;
        const int slot = j % D;
        if (mbar_wait_abortable(&full[slot], (uint32_t)(j / D) & 1u, status, s.abort)) {
            const int kc = ks * G::kKS;
            tile_compute<WT, BT>(ring + (size_t)slot * kTileBytes, s.X, Kpad, ks < n0 ? kc : kc - kx0,
                                 min(G::kKS, K - kc), nb, lane, acc);
        }
        __syncwarp();
        if (lane == 0 && i + kWarps * D < total && !*(volatile int*)s.abort) {
            issue(i + kWarps * D, slot);
            ++issued;
        }
        __syncwarp();
    }
    // Never leave with copies in flight (only possible after an abort): wait for them.
    if (lane == 0 && *(volatile int*)s.abort) {
        for (int jj = 0; jj < issued; ++jj) mbar_wait(&full[jj % D], (uint32_t)(jj / D) & 1u, status, 100000000LL);
    }
}


// Slots per warp that fit next to `fixed` bytes of other shared memory (0 if none fits).
inline int stream_slots(size_t smem_budget, size_t fixed) {
    if (fixed >= smem_budget) return 0;
    int d = (int)((smem_budget - fixed) / ((size_t)kWarps * (kTileBytes + sizeof(uint64_t))));
    return d > kMaxSlots ? kMaxSlots : d;
}

}  // namespace fe

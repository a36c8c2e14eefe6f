// Weight-streaming core shared by every matrix-vector phase of the drafter.
//
// At batch 1 each phase of the cascade (Eq. 1 FCs, the QKV / O / gate-up / down
// projections of every layer L_i in Eq. 2, the LM head of Sec. 2.1) reads a weight
// matrix once and does 2 flops per weight: the phases are bound by HBM bandwidth, not
// by arithmetic. So the CTA is built around keeping HBM busy:
//
//   - Weights are tile-packed at init (fe_pack.cu): each matrix is cut into groups of 4
//     rows, and each group into K-slices of kKS columns; the 4 x width block of one
//     (group, slice) is stored contiguously, so one stage of the stream is ONE
//     contiguous bulk copy of up to 16 KB. (Row-major stages made of 4 row pieces at the
//     row stride measured at ~3.7 TB/s on GB300; contiguous 4-16 KB copies at ~6.4 TB/s.)
//   - Warp 8 (one elected thread) is the producer: it walks the CTA's contiguous range of
//     row groups and issues cp.async.bulk (TMA) copies into a ring of n_stages stages,
//     each completing on its own mbarrier, running as far ahead as the ring allows.
//   - Warps 0..7 are consumers: thread t handles 16-byte column vectors t, t+256, ... of
//     all 4 rows of a stage and multiplies them by the activations X (float32 in shared
//     memory for the whole phase, staged once with a fused prologue), so each X vector is
//     reused for 4 weight rows. Per row group the 4 x BT partial sums are reduced across
//     each warp with a transposing shuffle reduction, then across the 8 warps through
//     shared memory, and handed to the phase's epilogue.
//
// Accumulation is float32 FMA on CUDA cores: at 1..8 activation rows the tensor pipe
// would idle, and this keeps fp32 weights (the small parity workload) on exact fp32
// arithmetic, never TF32.
#pragma once

#include "fe_common.cuh"

namespace fe {

constexpr int kConsumerWarps = 8;
constexpr int kConsumers = kConsumerWarps * 32;  // 256 threads
constexpr int kStreamThreads = kConsumers + 32;  // + the producer warp
constexpr int kGroupRows = 4;                    // weight rows per group
constexpr int kStageBytes = 16384;               // 4 rows x 4 KB
constexpr int kMaxStages = 13;

template <typename WT>
struct StreamGeom {
    static constexpr int kES = Storage<WT>::kBytes;
    static constexpr int kVec = Vec16<WT>::kN;                    // elements per 16 B
    static constexpr int kKS = kStageBytes / (kGroupRows * kES);  // columns per full slice
};

// Element offset of tile (group g, slice s) in a tile-packed [ceil(M/4)*4, K] matrix.
template <typename WT>
__host__ __device__ __forceinline__ int64_t tile_offset(int g, int s, int K) {
    return (int64_t)g * kGroupRows * K + (int64_t)s * kGroupRows * StreamGeom<WT>::kKS;
}

struct StreamSmem {
    unsigned char* ring;  // n_stages x kStageBytes (128-byte aligned)
    float* X;             // [xrows][Kpad] activations
    float* red;           // [2][kConsumerWarps][4 * BT] per-warp partial sums (double-buffered)
    uint64_t* full;       // [n_stages]
    uint64_t* empty;      // [n_stages]
    int* abort;           // set when any wait of this CTA gave up
};

// Bytes of dynamic shared memory a streaming CTA needs (before any epilogue extras).
__host__ __device__ inline size_t stream_smem_bytes(int n_stages, int xrows, int Kpad, int BT) {
    size_t b = (size_t)n_stages * kStageBytes;
    b += (size_t)xrows * Kpad * sizeof(float);
    b += (size_t)2 * kConsumerWarps * kGroupRows * BT * sizeof(float);
    b = (b + 15) & ~(size_t)15;
    b += (size_t)2 * n_stages * sizeof(uint64_t) + 16;
    return b;
}

__device__ inline StreamSmem carve_stream_smem(unsigned char* smem, int n_stages, int xrows, int Kpad, int BT) {
    StreamSmem s;
    s.ring = smem;
    s.X = (float*)(smem + (size_t)n_stages * kStageBytes);
    s.red = s.X + (size_t)xrows * Kpad;
    size_t off = (size_t)n_stages * kStageBytes +
                 ((size_t)xrows * Kpad + 2 * kConsumerWarps * kGroupRows * BT) * sizeof(float);
    off = (off + 15) & ~(size_t)15;
    s.full = (uint64_t*)(smem + off);
    s.empty = s.full + n_stages;
    s.abort = (int*)(s.empty + n_stages);
    return s;
}

// Wait on a phase of `bar`; gives up when the CTA's abort flag is raised or after the
// wall-clock budget (then raises the flag and records ST_TIMEOUT).
__device__ __forceinline__ bool mbar_wait_abortable(uint64_t* bar, uint32_t parity, int* status, int* abort) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*(volatile int*)abort) return false;
        if ((int64_t)(globaltimer_ns() - t0) > kWaitBudgetNs) {
            atomicOr(status, ST_TIMEOUT);
            *(volatile int*)abort = 1;
            return false;
        }
    }
}

__device__ inline void stream_init_barriers(StreamSmem& s, int n_stages) {
    if (threadIdx.x == 0) {
        for (int i = 0; i < n_stages; ++i) {
            mbar_init(&s.full[i], 1);
            mbar_init(&s.empty[i], kConsumerWarps);
        }
        *s.abort = 0;
        mbar_fence_init();
    }
    __syncthreads();
}

// Producer: one thread streams the row groups [g0, g1) of the tile-packed W through the ring.
template <typename WT>
__device__ void stream_produce(const unsigned char* Wt, int K, int g0, int g1, StreamSmem& s, int ns, int* status) {
    using G = StreamGeom<WT>;
    const int nks = (K + G::kKS - 1) / G::kKS;
    const int total = (g1 - g0) * nks;
    int it = 0;
    for (; it < total; ++it) {
        const int slot = it % ns;
        const uint32_t u = (uint32_t)(it / ns);
        if (!mbar_wait_abortable(&s.empty[slot], (u & 1u) ^ 1u, status, s.abort)) break;
        const int g = g0 + it / nks, ks = it % nks;
        const uint32_t bytes = (uint32_t)kGroupRows * (uint32_t)min(G::kKS, K - ks * G::kKS) * G::kES;
        mbar_arrive_expect_tx(&s.full[slot], bytes);
        bulk_g2s(s.ring + (size_t)slot * kStageBytes, Wt + tile_offset<WT>(g, ks, K) * G::kES, bytes, &s.full[slot]);
    }
    // Do not leave the CTA with copies in flight: wait for the last issued stages to land.
    for (int j = max(0, it - ns); j < it; ++j) mbar_wait(&s.full[j % ns], (uint32_t)(j / ns) & 1u, status);
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

// Sum over the 8 consumer warps of partial (row r, batch column b) from one red buffer.
template <int BT>
__device__ __forceinline__ float group_sum(const float* red, int r, int b) {
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < kConsumerWarps; ++w) v += red[w * kGroupRows * BT + r * BT + b];
    return v;
}

// One stage: 4 weight rows x `width` columns (rows at stride `width`) starting at column kc.
template <typename WT, int BT>
__device__ __forceinline__ void stage_compute(const unsigned char* st, const float* X, int Kpad, int kc, int width,
                                              int nb, int t, float (&acc)[kGroupRows][BT]) {
    using G = StreamGeom<WT>;
    constexpr int V = G::kVec;
    const size_t rs = (size_t)width * G::kES;
    const int nv = width / V;
    for (int v = t; v < nv; v += kConsumers) {
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

// Consumers: compute every row group of [g0, g1); after each group call epi(g, red) on
// all 256 consumer threads (the epilogue reads group_sum<BT>(red, r, b)).
template <typename WT, int BT, typename Epi>
__device__ void stream_consume(int K, int g0, int g1, StreamSmem& s, int ns, int Kpad, int nb, int* status, Epi& epi) {
    using G = StreamGeom<WT>;
    using R = WarpMultiSum<kGroupRows * BT>;
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int nks = (K + G::kKS - 1) / G::kKS;
    int it = 0;
    for (int g = g0; g < g1; ++g) {
        float acc[kGroupRows][BT];
#pragma unroll
        for (int r = 0; r < kGroupRows; ++r)
#pragma unroll
            for (int b = 0; b < BT; ++b) acc[r][b] = 0.f;
        for (int ks = 0; ks < nks; ++ks, ++it) {
            const int slot = it % ns;
            const uint32_t u = (uint32_t)(it / ns);
            if (mbar_wait_abortable(&s.full[slot], u & 1u, status, s.abort)) {
                const int kc = ks * G::kKS;
                stage_compute<WT, BT>(s.ring + (size_t)slot * kStageBytes, s.X, Kpad, kc, min(G::kKS, K - kc), nb,
                                      t, acc);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&s.empty[slot]);
        }
        float* red = s.red + (size_t)((g - g0) & 1) * kConsumerWarps * kGroupRows * BT;
        R::run(&acc[0][0], lane);
        if (R::owner(lane)) red[warp * kGroupRows * BT + R::index(lane)] = acc[0][0];
        named_sync(1, kConsumers);
        epi(g, red);
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

template <typename WT>
__device__ void stage_activations(const ProParams& p, int K, float* X, int Kpad, int b0, int nb, int* status,
                                  float* scratch /* >= kConsumerWarps floats */) {
    using S = Storage<WT>;
    const int t = threadIdx.x;
    for (int b = 0; b < nb; ++b) {
        const int row = b0 + b;
        float* Xb = X + (size_t)b * Kpad;
        if (p.pro == PRO_F32) {
            const float* xr = (const float*)p.x + (size_t)row * p.ldx;
            for (int k = t; k < K; k += kConsumers) Xb[k] = xr[k];
        } else if (p.pro == PRO_STORAGE) {
            const WT* xr = (const WT*)p.x + (size_t)row * p.ldx;
            for (int k = t; k < K; k += kConsumers) Xb[k] = S::load(xr, k);
        } else if (p.pro == PRO_CONCAT_EMB) {
            const float* xr = (const float*)p.x + (size_t)row * p.ldx;
            int tok = p.tok[row];
            if (tok < 0 || tok >= p.vocab) {
                if (t == 0) atomicOr(status, ST_DEVICE);
                tok = -1;
            }
            const int de = K - p.d_split;
            const WT* er = (const WT*)p.embed + (size_t)(tok < 0 ? 0 : tok) * de;
            for (int k = t; k < K; k += kConsumers)
                Xb[k] = k < p.d_split ? xr[k] : (tok < 0 ? 0.f : S::load(er, k - p.d_split));
        } else {  // PRO_RMSNORM
            const float* xr = (const float*)p.x + (size_t)row * p.ldx;
            float ss = 0.f;
            for (int k = t; k < K; k += kConsumers) {
                const float v = xr[k];
                Xb[k] = v;
                ss = fmaf(v, v, ss);
            }
            ss = warp_sum(ss);
            if ((t & 31) == 0) scratch[t >> 5] = ss;
            named_sync(1, kConsumers);
            float tot = 0.f;
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w) tot += scratch[w];
            const float rs = 1.0f / sqrtf(tot / (float)K + p.eps);
            const WT* gm = (const WT*)p.gamma;
            for (int k = t; k < K; k += kConsumers) Xb[k] = Xb[k] * rs * S::load(gm, k);
            named_sync(1, kConsumers);  // scratch reuse by the next row
        }
    }
    // zero the padding columns so vector loads past K read zeros
    for (int b = 0; b < nb; ++b)
        for (int k = K + t; k < Kpad; k += kConsumers) X[(size_t)b * Kpad + k] = 0.f;
}

}  // namespace fe

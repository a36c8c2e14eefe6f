// Weight-streaming core shared by every matrix-vector phase of the drafter.
//
// At batch 1 each phase of the cascade (Eq. 1 FCs, the QKV / O / gate-up / down
// projections of every layer L_i in Eq. 2, the LM head of Sec. 2.1) reads a weight
// matrix once and does 2 flops per weight: the phases are bound by HBM bandwidth, not
// by arithmetic. So the CTA is built around keeping HBM busy:
//
//   - warp 8 (one elected thread) is the producer: it walks the CTA's contiguous range
//     of 4-row groups of W and issues bulk TMA copies (cp.async.bulk, global -> shared)
//     of up to 16 KB per stage into a ring of n_stages stages, each stage completing on
//     its own mbarrier; it runs as far ahead as the ring allows;
//   - warps 0..7 are consumers: stage t holds 4 rows x KS columns; thread t handles rows
//     {2h, 2h+1} (h = t / 128) at 16-byte column vectors t % 128, t % 128 + 128, ... and
//     multiplies them by the activations X, which sit in shared memory as float32 for
//     the whole phase. Each X vector is reused for two weight rows. Partial sums are
//     reduced across the 128 threads of a half once per row group (warp shuffles, then
//     4 warps through shared memory) and handed to the phase's epilogue.
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
constexpr int kMaxStages = 8;

template <typename WT>
struct StreamGeom {
    static constexpr int kES = Storage<WT>::kBytes;
    static constexpr int kVec = Vec16<WT>::kN;                       // elements per 16 B
    static constexpr int kKS = kStageBytes / (kGroupRows * kES);     // columns per stage
};

struct StreamSmem {
    unsigned char* ring;  // n_stages x kStageBytes (128-byte aligned)
    float* X;             // [nb][Kpad] activations
    float* red;           // [2][kConsumerWarps][2][BT] partial sums (double-buffered)
    uint64_t* full;       // [n_stages]
    uint64_t* empty;      // [n_stages]
    int* abort;           // set when any wait of this CTA gave up
};

// Bytes of dynamic shared memory a streaming CTA needs (before epilogue extras).
__host__ __device__ inline size_t stream_smem_bytes(int n_stages, int nb, int Kpad, int BT) {
    size_t b = (size_t)n_stages * kStageBytes;
    b += (size_t)nb * Kpad * sizeof(float);
    b += (size_t)2 * kConsumerWarps * 2 * BT * sizeof(float);
    b = (b + 15) & ~(size_t)15;
    b += (size_t)2 * n_stages * sizeof(uint64_t) + 16;
    return b;
}

__device__ inline StreamSmem carve_stream_smem(unsigned char* smem, int n_stages, int nb, int Kpad, int BT) {
    StreamSmem s;
    s.ring = smem;
    s.X = (float*)(smem + (size_t)n_stages * kStageBytes);
    s.red = s.X + (size_t)nb * Kpad;
    size_t off = (size_t)n_stages * kStageBytes + ((size_t)nb * Kpad + 2 * kConsumerWarps * 2 * BT) * sizeof(float);
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

// Producer: one thread streams the row groups [g0, g1) of W [M, K] through the ring.
template <typename WT>
__device__ void stream_produce(const unsigned char* W, int M, int K, int g0, int g1, StreamSmem& s, int ns,
                               int* status) {
    using G = StreamGeom<WT>;
    const int nks = (K + G::kKS - 1) / G::kKS;
    const int total = (g1 - g0) * nks;
    int it = 0;
    for (; it < total; ++it) {
        const int slot = it % ns;
        const uint32_t u = (uint32_t)(it / ns);
        if (!mbar_wait_abortable(&s.empty[slot], (u & 1u) ^ 1u, status, s.abort)) break;
        const int g = g0 + it / nks;
        const int kc = (it % nks) * G::kKS;
        const int width = min(G::kKS, K - kc);
        const uint32_t rowbytes = (uint32_t)width * G::kES;
        const int rows = min(kGroupRows, M - g * kGroupRows);
        mbar_arrive_expect_tx(&s.full[slot], (uint32_t)rows * rowbytes);
        unsigned char* dst = s.ring + (size_t)slot * kStageBytes;
        for (int r = 0; r < rows; ++r)
            bulk_g2s(dst + (size_t)r * G::kKS * G::kES,
                     W + ((int64_t)(g * kGroupRows + r) * K + kc) * G::kES, rowbytes, &s.full[slot]);
    }
    // Do not leave the CTA with copies in flight: wait for the last issued stages to land.
    for (int j = max(0, it - ns); j < it; ++j) mbar_wait(&s.full[j % ns], (uint32_t)(j / ns) & 1u, status);
}

// Sum of row r (0..3) of the group, batch column b, from one red buffer.
template <int BT>
__device__ __forceinline__ float group_sum(const float* red, int r, int b) {
    const int h = r >> 1, j = r & 1;
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) v += red[((h * 4 + w) * 2 + j) * BT + b];
    return v;
}

// One stage: 4 weight rows x `width` columns starting at column kc.
template <typename WT, int BT>
__device__ __forceinline__ void stage_compute(const unsigned char* st, const float* X, int Kpad, int kc, int width,
                                              int nb, int t, float (&acc0)[BT], float (&acc1)[BT]) {
    using G = StreamGeom<WT>;
    constexpr int V = G::kVec;
    const int half = t >> 7, cv = t & 127;
    const unsigned char* r0 = st + (size_t)(2 * half) * G::kKS * G::kES;
    const unsigned char* r1 = r0 + (size_t)G::kKS * G::kES;
    const int nv = width / V;
    for (int v = cv; v < nv; v += 128) {
        const uint4 a = *reinterpret_cast<const uint4*>(r0 + (size_t)v * 16);
        const uint4 c = *reinterpret_cast<const uint4*>(r1 + (size_t)v * 16);
        float fa[V], fc[V];
        Vec16<WT>::widen(a, fa);
        Vec16<WT>::widen(c, fc);
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
                for (int j = 0; j < V; ++j) {
                    acc0[b] = fmaf(fa[j], xv[j], acc0[b]);
                    acc1[b] = fmaf(fc[j], xv[j], acc1[b]);
                }
            }
        }
    }
}

// Consumers: compute every row group of [g0, g1); after each group call
// epi(g, red_buffer) on all 256 consumer threads (the epilogue reads group_sum()).
template <typename WT, int BT, typename Epi>
__device__ void stream_consume(int K, int g0, int g1, StreamSmem& s, int ns, int Kpad, int nb, int* status, Epi& epi) {
    using G = StreamGeom<WT>;
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int nks = (K + G::kKS - 1) / G::kKS;
    int it = 0;
    for (int g = g0; g < g1; ++g) {
        float acc0[BT], acc1[BT];
#pragma unroll
        for (int b = 0; b < BT; ++b) { acc0[b] = 0.f; acc1[b] = 0.f; }
        for (int ks = 0; ks < nks; ++ks, ++it) {
            const int slot = it % ns;
            const uint32_t u = (uint32_t)(it / ns);
            const bool ok = mbar_wait_abortable(&s.full[slot], u & 1u, status, s.abort);
            if (ok) {
                const int kc = ks * G::kKS;
                stage_compute<WT, BT>(s.ring + (size_t)slot * kStageBytes, s.X, Kpad, kc, min(G::kKS, K - kc), nb, t,
                                      acc0, acc1);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&s.empty[slot]);
        }
        float* red = s.red + (size_t)((g - g0) & 1) * kConsumerWarps * 2 * BT;
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            const float v0 = warp_sum(acc0[b]);
            const float v1 = warp_sum(acc1[b]);
            if (lane == 0) {
                red[(warp * 2 + 0) * BT + b] = v0;
                red[(warp * 2 + 1) * BT + b] = v1;
            }
        }
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

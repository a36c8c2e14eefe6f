// Linear phases of the cascade (Eq. 1 FCs; QKV, O-proj, gate/up and down projections
// of each layer L_i, Eq. 2) as weight-streaming CTAs (fe_stream.cuh) with a fused
// prologue (RMSNorm / concat with the token embedding) and epilogue (store, residual
// add, SwiGLU).
#include "fe_kernels.h"
#include "fe_stream.cuh"

namespace fe {

template <int BT>
struct LinearEpi {
    const LinearArgs* a;
    int b0, nb;
    __device__ __forceinline__ void chunk(int cg0, int cg1, const float* red) const {
        const int ng = cg1 - cg0;
        if (a->epi == EPI_SWIGLU) {  // rows (2j, 2j+1) of the packed [gate; up] matrix
            for (int q = threadIdx.x; q < ng * 2 * BT; q += kStreamThreads) {
                const int gl = q / (2 * BT), pr = (q / BT) % 2, b = q % BT;
                const int m = (cg0 + gl) * kGroupRows + 2 * pr;
                if (b < nb && m + 1 < a->M) {
                    const float gate = chunk_value<BT>(red, gl, 2 * pr, b);
                    const float up = chunk_value<BT>(red, gl, 2 * pr + 1, b);
                    a->y[(size_t)(b0 + b) * a->ldy + (m >> 1)] = silu(gate) * up;
                }
            }
            return;
        }
        for (int q = threadIdx.x; q < ng * kGroupRows * BT; q += kStreamThreads) {
            const int gl = q / (kGroupRows * BT), r = (q / BT) % kGroupRows, b = q % BT;
            const int m = (cg0 + gl) * kGroupRows + r;
            if (b < nb && m < a->M) {
                const float v = chunk_value<BT>(red, gl, r, b);
                float* yp = a->y + (size_t)(b0 + b) * a->ldy + m;
                if (a->epi == EPI_RESID) {
                    // (read through L2: another CTA may have written it in a persistent kernel)
                    const float nv = __ldcg(a->ybase ? a->ybase + (size_t)(b0 + b) * a->ldy + m : yp) + v;
                    *yp = nv;
                    if (a->y2) a->y2[(size_t)(b0 + b) * a->ldy2 + m] = nv;
                } else {
                    *yp = v;
                }
            }
        }
    }
};

// n0 > 0: the activations are staged in two passes of n0 and the remaining slices' columns
// (X holds Kx columns per row), so that a long row leaves room for more pipeline slots
template <typename WT, int BT>
__global__ void __launch_bounds__(kStreamThreads, 1) linear_kernel(const LinearArgs a, int D, int n0) {
    const LaunchStamp stamp(a.stamp);
    extern __shared__ __align__(128) unsigned char smem[];
    const int Kx = n0 > 0 ? n0 * StreamGeom<WT>::kKS : (a.K + 3) & ~3;
    const int b0 = blockIdx.y * BT;
    const int nb = min(BT, a.B - b0);
    StreamSmem s = carve_stream_smem(smem, D, min(BT, a.B), Kx, BT);
    const int GM = (a.M + kGroupRows - 1) / kGroupRows;
    const int g0 = (int)(((int64_t)blockIdx.x * GM) / gridDim.x);
    const int g1 = (int)(((int64_t)(blockIdx.x + 1) * GM) / gridDim.x);
    // weights do not depend on the previous kernel: start streaming them first
    const int issued = stream_begin<WT>((const unsigned char*)a.W, a.K, g0, g1, s, D, false, n0);
    griddep_launch_dependents();
    // gains and embedding rows do not depend on the previous kernel either
    ProParams pp{a.pro, a.x, a.ldx, a.gamma, a.eps, a.embed, a.tok, a.d_split, a.vocab};
    const bool pre = n0 > 0 ? false : stage_pre<WT>(pp, a.K, s.X, Kx, b0, nb, a.status);
    griddep_wait();
    stage_activations<WT>(pp, n0 > 0 ? Kx : a.K, s.X, Kx, b0, nb, a.status, s.red, pre);
    __syncthreads();
    LinearEpi<BT> e{&a, b0, nb};
    stream_run<WT, BT>((const unsigned char*)a.W, a.K, g0, g1, s, D, Kx, nb, a.status, e, issued, n0, &pp, b0);
}

// ---- persistent stack of linear phases --------------------------------------------------------
// Runs sa.nph consecutive linear phases (e.g. W_o, W_gate/up, W_down and the next layer's
// W_qkv) in one launch of one CTA per SM: between phases every CTA issues its first copies
// of the next phase's weights (they do not depend on the phase in flight) and then meets the
// others at a grid-wide barrier, after which the next phase's activations — written by all
// CTAs — are complete. This removes the per-launch pipeline fill and tail of separate
// launches. Each phase computes exactly what linear_kernel computes for it (same row
// partition, same order of operations).
template <typename WT, int BT>
__global__ void __launch_bounds__(kStreamThreads, 1) stack_kernel(const StackArgs sa, int D, int Kpad_max) {
    const LaunchStamp stamp(sa.ph[0].stamp);
    extern __shared__ __align__(128) unsigned char smem[];
    StreamSmem s = carve_stream_smem(smem, D, 1, Kpad_max, BT);
    int issued = 0;
    for (int p = 0; p < sa.nph; ++p) {
        const LinearArgs& a = sa.ph[p];
        const int Kpad = (a.K + 3) & ~3;
        const int GM = (a.M + kGroupRows - 1) / kGroupRows;
        const int g0 = (int)(((int64_t)blockIdx.x * GM) / gridDim.x);
        const int g1 = (int)(((int64_t)(blockIdx.x + 1) * GM) / gridDim.x);
        if (p == 0) {
            issued = stream_begin<WT>((const unsigned char*)a.W, a.K, g0, g1, s, D);
            griddep_launch_dependents();
            griddep_wait();
        }
        ProParams pp{a.pro, a.x, a.ldx, a.gamma, a.eps, a.embed, a.tok, a.d_split, a.vocab};
        stage_activations<WT>(pp, a.K, s.X, Kpad, 0, a.B, a.status, s.red);
        __syncthreads();
        LinearEpi<BT> e{&a, 0, a.B};
        stream_run<WT, BT>((const unsigned char*)a.W, a.K, g0, g1, s, D, Kpad, a.B, a.status, e, issued);
        if (p + 1 == sa.nph || *(volatile int*)s.abort) break;
        const LinearArgs& nx = sa.ph[p + 1];
        const int GMn = (nx.M + kGroupRows - 1) / kGroupRows;
        const int h0 = (int)(((int64_t)blockIdx.x * GMn) / gridDim.x);
        const int h1 = (int)(((int64_t)(blockIdx.x + 1) * GMn) / gridDim.x);
        grid_arrive(sa.barrier);  // (its __syncthreads: every warp is done with the ring and its barriers)
        issued = stream_begin<WT>((const unsigned char*)nx.W, nx.K, h0, h1, s, D, true);
        if (!grid_wait(sa.barrier, (uint32_t)(p + 1), a.status, s.abort)) {
            // never leave with copies in flight: wait (bounded) for this warp's first copies
            const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
            if (lane == 0)
                for (int j = 0; j < issued; ++j) mbar_wait(&s.full[warp * D + j], 0u, a.status, 100000000LL);
            break;
        }
    }
}

// ---- host side ----------------------------------------------------------------------------
namespace {

constexpr size_t kXBudget = 128 * 1024;  // activations held in shared memory per CTA
// Per-warp pipeline depth: three 8 KB slots where shared memory allows (more bytes in flight
// per SM), two next to attention (its CTAs start early on the same SMs and need the room).
constexpr int kPreferredSlots = 3;

template <typename WT, int BT>
cudaError_t set_attr(const DeviceInfo& dev) {
    return cudaFuncSetAttribute(linear_kernel<WT, BT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                dev.max_smem_optin);
}

int pick_bt(int B, int K) {
    const size_t row = (size_t)((K + 3) & ~3) * sizeof(float);
    int bt = 8;
    while (bt > 1 && ((size_t)(bt < B ? bt : B) * row > kXBudget || bt / 2 >= B)) bt >>= 1;
    return bt;
}

template <typename WT, int BT>
cudaError_t launch_bt(const LinearArgs& a, const DeviceInfo& dev, cudaStream_t st) {
    const int Kpad = (a.K + 3) & ~3;
    const int xrows = BT < a.B ? BT : a.B;
    const int pref = a.slots > 0 ? a.slots : kPreferredSlots;
    auto slots_for = [&](int kx) {
        const int d = stream_slots((size_t)dev.max_smem_optin, stream_smem_bytes(0, xrows, kx, BT));
        return d > pref ? pref : d;
    };
    int D = slots_for(Kpad);
    const int GM = (a.M + kGroupRows - 1) / kGroupRows;
    dim3 grid(GM < dev.num_sms ? GM : dev.num_sms, (a.B + BT - 1) / BT);
    // A row too long for two slots per warp next to it (the FC over the concatenated target
    // features, the down projection of a wide MLP) is staged in two passes when that buys a
    // deeper pipeline and the CTA's row groups fit one epilogue chunk. Plain float32 or
    // storage-type inputs only (no row-wide RMSNorm, no concatenation).
    int n0 = 0, Kx = Kpad;
    constexpr int KS = StreamGeom<WT>::kKS;
    const int nks = (a.K + KS - 1) / KS;
    if (D < 2 && nks >= 2 && (a.pro == PRO_F32 || a.pro == PRO_STORAGE) &&
        (GM + (int)grid.x - 1) / (int)grid.x <= chunk_groups(BT)) {
        const int h = (nks + 1) / 2;
        const int d2 = slots_for(h * KS);
        if (d2 > D) {
            D = d2;
            n0 = h;
            Kx = h * KS;
        }
    }
    if (D < 1) return cudaErrorInvalidValue;
    const size_t smem = stream_smem_bytes(D, xrows, Kx, BT);
    return launch_k(linear_kernel<WT, BT>, grid, dim3(kStreamThreads), smem, st, a.pdl, a, D, n0);
}

template <typename WT>
cudaError_t launch_t(const LinearArgs& a, const DeviceInfo& dev, cudaStream_t st) {
    switch (pick_bt(a.B, a.K)) {
        case 1: return launch_bt<WT, 1>(a, dev, st);
        case 2: return launch_bt<WT, 2>(a, dev, st);
        case 4: return launch_bt<WT, 4>(a, dev, st);
        default: return launch_bt<WT, 8>(a, dev, st);
    }
}

}  // namespace

template <typename WT, int BT>
cudaError_t set_stack_attr(const DeviceInfo& dev) {
    return cudaFuncSetAttribute(stack_kernel<WT, BT>, cudaFuncAttributeMaxDynamicSharedMemorySize, dev.max_smem_optin);
}

cudaError_t linear_prepare(const DeviceInfo& dev) {
    cudaError_t e;
    if ((e = set_stack_attr<float, 1>(dev)) != cudaSuccess) return e;
    if ((e = set_stack_attr<bf16_t, 1>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<float, 1>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<float, 2>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<float, 4>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<float, 8>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<bf16_t, 1>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<bf16_t, 2>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<bf16_t, 4>(dev)) != cudaSuccess) return e;
    return set_attr<bf16_t, 8>(dev);
}

// pipeline slots per warp for a stack whose largest K is k_max (B = 1); 0 if it does not fit
int stack_slots(int k_max, const DeviceInfo& dev) {
    const int Kpad = (k_max + 3) & ~3;
    int D = stream_slots((size_t)dev.max_smem_optin, stream_smem_bytes(0, 1, Kpad, 1));
    return D > kPreferredSlots ? kPreferredSlots : D;
}

cudaError_t launch_stack(fe_dtype dt, const StackArgs& sa, const DeviceInfo& dev, cudaStream_t st) {
    if (sa.nph < 1 || sa.nph > kMaxStackPhases || !sa.barrier) return cudaErrorInvalidValue;
    int kmax = 0;
    for (int p = 0; p < sa.nph; ++p) {
        if (sa.ph[p].B != 1 || sa.ph[p].M <= 0) return cudaErrorInvalidValue;
        kmax = sa.ph[p].K > kmax ? sa.ph[p].K : kmax;
    }
    const int D = stack_slots(kmax, dev);
    if (D < 1) return cudaErrorInvalidValue;
    const int Kpad = (kmax + 3) & ~3;
    const size_t smem = stream_smem_bytes(D, 1, Kpad, 1);
    // one CTA per SM, all resident at once (the grid barrier needs them all)
    const int grid = dev.num_sms;
    return dt == FE_F32 ? launch_k(stack_kernel<float, 1>, dim3(grid), dim3(kStreamThreads), smem, st, sa.ph[0].pdl, sa, D, Kpad)
                        : launch_k(stack_kernel<bf16_t, 1>, dim3(grid), dim3(kStreamThreads), smem, st, sa.ph[0].pdl, sa, D,
                                   Kpad);
}

cudaError_t launch_linear(fe_dtype dt, const LinearArgs& a, const DeviceInfo& dev, cudaStream_t st) {
    if (a.M <= 0 || a.B <= 0) return cudaSuccess;
    return dt == FE_F32 ? launch_t<float>(a, dev, st) : launch_t<bf16_t>(a, dev, st);
}

}  // namespace fe

// Device-side helpers shared by the drafter's kernels (sm_103a).
//
// - storage conversion (bfloat16 bits <-> float32) for weights, features and caches
// - mbarrier and bulk-copy (TMA, cp.async.bulk) wrappers in inline PTX
// - bounded waits: every spin on a barrier gives up after a wall-clock budget, records
//   FE_ERR_TIMEOUT in the handle's status word and lets the kernel return, so no wait
//   can hang the GPU
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "fe_kernels.h"

namespace fe {

constexpr int64_t kWaitBudgetNs = 2000000000LL;  // 2 s: far above any legitimate wait

// ---- storage types ----------------------------------------------------------------
struct bf16_t { uint16_t bits; };

__device__ __forceinline__ float bf16_to_f32(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }

// round-to-nearest-even float -> bfloat16 bits (finite inputs)
__device__ __forceinline__ uint16_t f32_to_bf16(float f) {
    uint32_t u = __float_as_uint(f);
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

template <typename T> struct Storage;
template <> struct Storage<float> {
    static constexpr int kBytes = 4;
    __device__ __forceinline__ static float load(const float* p, int64_t i) { return p[i]; }
    __device__ __forceinline__ static void store(float* p, int64_t i, float v) { p[i] = v; }
};
template <> struct Storage<bf16_t> {
    static constexpr int kBytes = 2;
    __device__ __forceinline__ static float load(const bf16_t* p, int64_t i) { return bf16_to_f32(p[i].bits); }
    __device__ __forceinline__ static void store(bf16_t* p, int64_t i, float v) { p[i].bits = f32_to_bf16(v); }
};

// 16 bytes of storage widened to floats: 4 floats or 8 bfloat16 values
template <typename T> struct Vec16;
template <> struct Vec16<float> {
    static constexpr int kN = 4;
    __device__ __forceinline__ static void widen(const uint4& v, float* f) {
        f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
        f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
    }
};
template <> struct Vec16<bf16_t> {
    static constexpr int kN = 8;
    __device__ __forceinline__ static void widen(const uint4& v, float* f) {
        f[0] = __uint_as_float(v.x << 16); f[1] = __uint_as_float(v.x & 0xFFFF0000u);
        f[2] = __uint_as_float(v.y << 16); f[3] = __uint_as_float(v.y & 0xFFFF0000u);
        f[4] = __uint_as_float(v.z << 16); f[5] = __uint_as_float(v.z & 0xFFFF0000u);
        f[6] = __uint_as_float(v.w << 16); f[7] = __uint_as_float(v.w & 0xFFFF0000u);
    }
};

// ---- time ---------------------------------------------------------------------------
__device__ __forceinline__ uint64_t globaltimer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// ---- in-graph launch timing ------------------------------------------------------------
// When a launch is given a stamp pair p (both words zero before the graph runs), the CTA's
// thread 0 records its start and each warp's first active lane its exit, as %globaltimer
// nanoseconds: p[0] = max over CTAs of ~start (so ~p[0] is the earliest start and zero
// means "never stamped"), p[1] = max over warps of the exit time. Declared first in a
// kernel, the object's destructor runs on every return path.
struct LaunchStamp {
    unsigned long long* p;
    __device__ __forceinline__ explicit LaunchStamp(unsigned long long* s) : p(s) {
        if (p && threadIdx.x == 0) atomicMax(p, ~(unsigned long long)globaltimer_ns());
    }
    __device__ __forceinline__ ~LaunchStamp() {
        if (p) {
            const unsigned m = __activemask();
            if ((int)(threadIdx.x & 31) == __ffs(m) - 1) atomicMax(p + 1, (unsigned long long)globaltimer_ns());
        }
    }
};

// ---- mbarrier -------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

// retire an mbarrier (no pending arrivals or copies) before its memory is initialised again
__device__ __forceinline__ void mbar_inval(uint64_t* bar) {
    asm volatile("mbarrier.inval.shared::cta.b64 [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_fence_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// As mbar_try_wait, but the thread may sleep up to `hint_ns` for the phase to complete
// (for waits that are expected to be long: no busy spinning).
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t* bar, uint32_t parity, uint32_t hint_ns) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "r"(hint_ns)
        : "memory");
    return ok != 0;
}

// ---- programmatic dependent launch --------------------------------------------------------
// Kernels after the first of a draft are launched with programmatic stream serialization:
// they may start while the previous kernel finishes. Each one issues only work that does
// not depend on earlier kernels (weight and cached-prefix copies) before griddep_wait(),
// which blocks until every earlier kernel has completed and its writes are visible.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Wait for the phase of `bar` with the given parity to complete. Returns false (and sets
// ST_TIMEOUT in *status) if it has not completed within `budget_ns`.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, int* status,
                                          int64_t budget_ns = kWaitBudgetNs) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((int64_t)(globaltimer_ns() - t0) > budget_ns) {
            if (status) atomicOr(status, ST_TIMEOUT);
            return false;
        }
    }
}

// ---- bulk copy (TMA, non-tensor) -------------------------------------------------------
// global -> shared, completion counted on `bar` in bytes. dst, src 16-byte aligned,
// bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

// An L2 policy for data read once per draft (weights, cached K/V): evict first, so the
// streams do not push out what the next kernels read back (partials, activations, operands).
__device__ __forceinline__ uint64_t l2_evict_first() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

// bulk_g2s with an L2 cache policy (l2_evict_first() for streamed data)
__device__ __forceinline__ void bulk_g2s_hint(void* dst, const void* src, uint32_t bytes, uint64_t* bar, uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(pol)
        : "memory");
}

// global -> L2 prefetch of `bytes` (16-byte aligned address, multiple of 16); no completion
__device__ __forceinline__ void bulk_prefetch_l2(const void* src, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

// atomic add at GPU scope with acquire-release semantics; returns the old value
__device__ __forceinline__ int atom_add_acq_rel_gpu(int* p, int v) {
    int old;
    asm volatile("atom.add.acq_rel.gpu.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

// ---- grid-wide barrier of a persistent kernel ----------------------------------------------
__device__ __forceinline__ uint32_t ld_acquire_gpu(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Grid-wide barrier of a persistent kernel, split in two so that work that does not
// depend on the other CTAs (issuing weight copies) can go between arrive and wait. Every
// CTA arrives once on *count (zero at launch) per barrier; the k-th barrier (k = 1, 2, ...)
// completes when *count reaches k * gridDim.x. All CTAs must be resident at once (grid <=
// SMs, one CTA per SM). Writes made before grid_arrive are visible to L2-coherent reads
// (ld.global.cg, TMA) after grid_wait. The arriving / polling thread is lane 1 of warp 0,
// which issues no asynchronous copies, so its fence does not wait for any. Both are called
// by every thread of the CTA.
constexpr int kGridBarrierThread = 1;

__device__ __forceinline__ void grid_arrive(uint32_t* count) {
    __syncthreads();
    if (threadIdx.x == kGridBarrierThread) {
        __threadfence();
        atomicAdd(count, 1u);
    }
}

// Bounded: after kWaitBudgetNs it records ST_TIMEOUT, raises *abort and returns false.
__device__ __forceinline__ bool grid_wait(uint32_t* count, uint32_t k, int* status, int* abort) {
    if (threadIdx.x == kGridBarrierThread) {
        const uint32_t target = k * gridDim.x;
        if (ld_acquire_gpu(count) < target) {
            const uint64_t t0 = globaltimer_ns();
            while (ld_acquire_gpu(count) < target) {
                if ((int64_t)(globaltimer_ns() - t0) > kWaitBudgetNs) {
                    atomicOr(status, ST_TIMEOUT);
                    *(volatile int*)abort = 1;
                    break;
                }
            }
        }
        __threadfence();
    }
    __syncthreads();
    return !*(volatile int*)abort;
}

// ---- named barriers (a subset of the CTA's warps) ---------------------------------------
__device__ __forceinline__ void named_sync(int id, int nthreads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// ---- reductions ----------------------------------------------------------------------------
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// SiLU(a) = a / (1 + e^-a)
__device__ __forceinline__ float silu(float a) { return a / (1.0f + expf(-a)); }

// 2^x by the hardware approximation (relative error about 2^-22; 2^-inf = 0)
__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

constexpr float kLog2e = 1.4426950408889634f;  // log2(e)

}  // namespace fe

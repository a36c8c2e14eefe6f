// Linear phases of the cascade on the tensor cores (tcgen05 + TMEM), for batches of
// sequences: Y[b, m] = epilogue(sum_k W[m, k] X[b, k]) for b < B (Eq. 1 FCs; QKV, O-proj,
// gate/up and down projections of every layer L_i, Eq. 2).
//
// At batch 1 a linear phase is a matrix-vector product and the CUDA-core streaming kernel
// (fe_linear.cu) is the right tool. With many sequences it re-reads the weights once per
// batch tile; here every weight is read once for the whole batch and the products run on
// the tensor cores:
//   - xprep_kernel applies the phase's prologue (RMSNorm, concat with the token embedding,
//     storage or float32 input) and writes the activations as a bf16 B operand split into
//     hi and lo parts (x = hi + lo to ~16 significant bits, so the products keep float32
//     accuracy): rows [0, B_pad) hold hi, [B_pad, 2 B_pad) hold lo, in the 128-byte-
//     swizzled K-major layout of fe_tc.cuh, one 2 B_pad x 64 block per 64 columns.
//   - linear_mma_kernel: the weights are packed at init in 128 x 64 swizzled blocks
//     (fe_pack.cu), so one TMA bulk copy lands one A operand. The (tile of 128 output rows,
//     64-column block) units are split evenly over the CTAs in tile-major order (stream-K),
//     so every SM streams the same number of bytes whatever the matrix shape. Warp 4 issues
//     the copies (weights block + activation block per stage, a ring of S stages), warp 5
//     issues tcgen05.mma (M = 128, N = 2 B_pad, K = 16; float32 accumulators in TMEM, two
//     buffers), warps 0-3 read TMEM (thread = output row) and add hi + lo.
//   - A tile whose units all fall in one CTA is finished there. A tile split between CTAs
//     leaves one float32 partial per CTA in global scratch; the last CTA to finish its
//     share of the tile (an atomic counter) sums the partials in CTA order (so results do
//     not depend on timing) and applies the epilogue: store, residual add (+ copy into the
//     hidden-state buffer), or SwiGLU over the interleaved gate/up rows (the partner row
//     sits in the neighbouring lane).
#include "fe_kernels.h"
#include "fe_stream.cuh"
#include "fe_tc.cuh"
#include "fe_splitk.cuh"

namespace fe {

namespace {

constexpr int kLmThreads = 192;  // 4 epilogue warps, 1 producer warp, 1 MMA warp
constexpr size_t kXprepRowSmem = 16384 * sizeof(float);  // a finished row of up to 16384 columns
constexpr int kLinMaxStages = 8;


struct LinMmaState {
    uint64_t full[kLinMaxStages], empty[kLinMaxStages], tfull[2], tempty[2];
    uint32_t tmem_base;
    int abort;
};

__device__ __forceinline__ void split_bf16(float z, uint16_t& hi, uint16_t& lo) {
    hi = f32_to_bf16(z);
    lo = f32_to_bf16(z - bf16_to_f32(hi));
}

}  // namespace

// ---- activation operand ------------------------------------------------------------------
// Grid (B_pad, ceil(K / 2048)): CTA (b, y) writes row b's 16-byte chunks [256 y, 256 y + 256)
// (rows b >= B are zero); with RMSNorm every CTA of the row reads the whole row for its sum
// of squares (an L2 read of 4 d bytes). Reads what the previous kernel wrote only after
// griddep_wait(), through L2, and never through a __restrict__ pointer.
// When the previous tensor-core phase deferred its split tiles (a.prev.active), the input
// columns of those tiles are finished here first (prev_finish); with RMSNorm, one CTA per
// row (grid (B_pad, 1)) finishes the whole row into shared memory before normalising it.
constexpr int kXprepChunks = 256;  // 16-byte chunks per CTA (one per thread)

// sum of squares of 8 values, in one fixed order
__device__ __forceinline__ float sumsq8(const float (&v)[8]) {
    float s = v[0] * v[0];
#pragma unroll
    for (int e = 1; e < 8; ++e) s = fmaf(v[e], v[e], s);
    return s;
}

// the bf16 hi / lo operand chunk c of row b from 8 values
__device__ __forceinline__ void put_operand(uint16_t* xb, int N, int B_pad, int b, int c, const float (&v)[8]) {
    uint32_t hi[4], lo[4];
#pragma unroll
    for (int e = 0; e < 8; e += 2) {
        uint16_t h0, l0, h1, l1;
        split_bf16(v[e], h0, l0);
        split_bf16(v[e + 1], h1, l1);
        hi[e / 2] = (uint32_t)h0 | ((uint32_t)h1 << 16);
        lo[e / 2] = (uint32_t)l0 | ((uint32_t)l1 << 16);
    }
    unsigned char* blk = (unsigned char*)xb + (size_t)(c / 8) * N * 128;
    *reinterpret_cast<uint4*>(blk + sw128_offset(b, c % 8)) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
    *reinterpret_cast<uint4*>(blk + sw128_offset(B_pad + b, c % 8)) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
}

__global__ void __launch_bounds__(256) xprep_kernel(const LinearArgs a, int B_pad, uint16_t* xb, float* sq) {
    const LaunchStamp stamp(a.stamp);
    const int b = blockIdx.x, t = threadIdx.x;
    const int N = 2 * B_pad, K = a.K, nc = K / 8;
    const int c = blockIdx.y * kXprepChunks + t;  // this thread's 16-byte chunk of row b
    const int k0 = 8 * c;
    __shared__ float red[8];
    griddep_launch_dependents();
    // weights do not depend on the previous kernel: the RMSNorm gains are loaded, and the
    // embedding row's line is prefetched into L2 (from a token id read early: a stale id
    // only warms a wrong line), before the wait
    uint4 gq = make_uint4(0, 0, 0, 0);
    if (b < a.B && c < nc) {
        if (a.pro == PRO_RMSNORM) gq = *reinterpret_cast<const uint4*>((const bf16_t*)a.gamma + k0);
        if (a.pro == PRO_CONCAT_EMB && k0 >= a.d_split) {
            const int tk = a.tok[b];
            if (tk >= 0 && tk < a.vocab)
                asm volatile("prefetch.global.L2 [%0];" ::"l"((const bf16_t*)a.embed + (size_t)tk * (K - a.d_split) +
                                                               (k0 - a.d_split)));
        }
    }
    griddep_wait();
    const bool live = b < a.B;
    const bool fin = live && a.prev.active;  // (without norm_post, RMSNorm inputs take xprep_row_kernel)
    const bool post = a.norm_post && a.pro == PRO_RMSNORM;  // the scale goes on the products
    int tok = 0;
    if (live && a.pro == PRO_CONCAT_EMB) {
        tok = a.tok[b];
        if (tok < 0 || tok >= a.vocab) {
            if (t == 0) atomicOr(a.status, ST_DEVICE);
            tok = -1;
        }
    }
    const float* xf = (const float*)a.x + (size_t)b * a.ldx;
    // the CTA's sum of per-thread partials in a fixed order
    auto cta_sum = [&](float ss) {
        ss = warp_sum(ss);
        if ((t & 31) == 0) red[t >> 5] = ss;
        __syncthreads();
        float tot = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) tot += red[w];
        return tot;
    };
    float rs = 1.f;
    if (live && a.pro == PRO_RMSNORM && !post) {  // 1 / sqrt(mean of squares + eps) over the whole row
        float ss = 0.f;
#pragma unroll 4
        for (int cc = t; cc < nc; cc += 256) {
            const float4 p = __ldcg(reinterpret_cast<const float4*>(xf) + 2 * cc);
            const float4 q = __ldcg(reinterpret_cast<const float4*>(xf) + 2 * cc + 1);
            const float v[8] = {p.x, p.y, p.z, p.w, q.x, q.y, q.z, q.w};
            ss += sumsq8(v);
        }
        rs = 1.0f / sqrtf(cta_sum(ss) / (float)K + a.eps);
    }
    float v[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = 0.f;
    if (live && c < nc) {
        if (a.pro == PRO_STORAGE) {
            Vec16<bf16_t>::widen(*reinterpret_cast<const uint4*>((const bf16_t*)a.x + (size_t)b * a.ldx + k0), v);
        } else if (a.pro == PRO_CONCAT_EMB && k0 >= a.d_split) {
            if (tok >= 0)
                Vec16<bf16_t>::widen(*reinterpret_cast<const uint4*>((const bf16_t*)a.embed +
                                                                     (size_t)tok * (K - a.d_split) + (k0 - a.d_split)),
                                     v);
        } else if (fin) {  // the previous phase's output, its split tiles finished here
            prev_finish(a.prev, B_pad, b, k0, v);
        } else {  // float32 input (PRO_F32, PRO_RMSNORM, or the float part of PRO_CONCAT_EMB)
            const float4 p = __ldcg(reinterpret_cast<const float4*>(xf + k0));
            const float4 q = __ldcg(reinterpret_cast<const float4*>(xf + k0) + 1);
            v[0] = p.x; v[1] = p.y; v[2] = p.z; v[3] = p.w; v[4] = q.x; v[5] = q.y; v[6] = q.z; v[7] = q.w;
        }
    }
    if (a.pro == PRO_RMSNORM) {
        float g[8];
        Vec16<bf16_t>::widen(gq, g);
        if (post) {  // gamma * x here; this CTA's sum of squares of x for the product kernel
            const float tot = cta_sum(sumsq8(v));
            if (t == 0) sq[blockIdx.y * B_pad + b] = tot;
#pragma unroll
            for (int e = 0; e < 8; ++e) v[e] *= g[e];
        } else {
#pragma unroll
            for (int e = 0; e < 8; ++e) v[e] = v[e] * rs * g[e];
        }
    }
    if (c < nc) put_operand(xb, N, B_pad, b, c, v);
}

// The deferred-input prep of an RMSNorm phase: one CTA of kRowThreads per row b finishes the
// previous phase's output over the whole row into shared memory (its split tiles, as
// prev_finish), sums its squares and writes the normalised row's operand. Thread t owns
// chunks t, t + kRowThreads, ... (the same per-thread order of the sum as xprep_kernel).
constexpr int kRowThreads = 512;

__global__ void __launch_bounds__(kRowThreads) xprep_row_kernel(const LinearArgs a, int B_pad, uint16_t* xb) {
    const LaunchStamp stamp(a.stamp);
    extern __shared__ __align__(16) float xrow[];  // the finished row [K]
    const int b = blockIdx.x, t = threadIdx.x;
    const int N = 2 * B_pad, K = a.K, nc = K / 8;
    __shared__ float red[kRowThreads / 32];
    griddep_launch_dependents();
    // the RMSNorm gains of this thread's first kPreChunks chunks (weights: loaded before the
    // wait; d <= 8192 needs no more)
    constexpr int kRowChunks = kXprepRowSmem / sizeof(float) / 8 / kRowThreads;
    constexpr int kPreChunks = 2;
    uint4 gq[kPreChunks];
#pragma unroll
    for (int j = 0; j < kPreChunks; ++j) {
        const int c = t + j * kRowThreads;
        gq[j] = b < a.B && c < nc ? *reinterpret_cast<const uint4*>((const bf16_t*)a.gamma + 8 * c) : make_uint4(0, 0, 0, 0);
    }
    griddep_wait();
    if (b >= a.B) {  // a padding row of the operand is zero
        const float z[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        for (int c = t; c < nc; c += kRowThreads) put_operand(xb, N, B_pad, b, c, z);
        return;
    }
    float ss = 0.f;
    for (int c = t; c < nc; c += kRowThreads) {
        float v[8];
        prev_finish_t<false>(a.prev, B_pad, b, 8 * c, v);  // (an RMSNorm input is never SwiGLU's output)
        ss += sumsq8(v);
        reinterpret_cast<float4*>(xrow)[2 * c] = make_float4(v[0], v[1], v[2], v[3]);
        reinterpret_cast<float4*>(xrow)[2 * c + 1] = make_float4(v[4], v[5], v[6], v[7]);
    }
    ss = warp_sum(ss);
    if ((t & 31) == 0) red[t >> 5] = ss;
    __syncthreads();  // (also publishes xrow)
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < kRowThreads / 32; ++w) tot += red[w];
    const float rs = 1.0f / sqrtf(tot / (float)K + a.eps);
#pragma unroll
    for (int j = 0; j < kRowChunks; ++j) {
        const int c = t + j * kRowThreads;
        if (c >= nc) break;
        float v[8], g[8];
        const float4 p = reinterpret_cast<const float4*>(xrow)[2 * c];
        const float4 q = reinterpret_cast<const float4*>(xrow)[2 * c + 1];
        v[0] = p.x; v[1] = p.y; v[2] = p.z; v[3] = p.w; v[4] = q.x; v[5] = q.y; v[6] = q.z; v[7] = q.w;
        Vec16<bf16_t>::widen(j < kPreChunks ? gq[j < kPreChunks ? j : 0]
                                            : *reinterpret_cast<const uint4*>((const bf16_t*)a.gamma + 8 * c),
                             g);
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = v[e] * rs * g[e];
        put_operand(xb, N, B_pad, b, c, v);
    }
}

// ---- the RMSNorm scale after the product (LinearArgs::norm_post) ---------------------------
// The operand prep of an RMSNorm phase writes gamma * x and, per CTA (row b, column range
// y), the sum of squares of x over its columns in sq[y * B_pad + b]; the product kernel sums
// them (fixed order) to 1 / sqrt(mean(x^2) + eps) and multiplies its products by it. So
// the prep needs no whole-row pass and runs column-parallel like any other.
constexpr int kAuxRs = 0;      // bytes into the counter buffer: the last normalised phase's scales
constexpr int kAuxSq = 256;    // the prep's sums of squares [ny][kLinMmaMaxBatch]
constexpr int kAuxEnd = 1280;  // (ny <= 8: K <= 16384)

// ---- the product ---------------------------------------------------------------------------
// Epilogue for output row m of all B sequences; v[b] is the finished dot product.
// SwiGLU pairs rows (2j, 2j + 1) held by neighbouring lanes of one warp.
template <int BP>
__device__ __forceinline__ void lin_epilogue(const LinearArgs& a, int m, const float (&v)[BP]) {
    const int lane = threadIdx.x & 31;
    // Every operand is read before any result is written: a load after a store to the same
    // buffer would wait for it, making the 32 rows one chain of L2 round trips.
    if (a.epi == EPI_SWIGLU) {
        float o[BP];
#pragma unroll
        for (int b = 0; b < BP; ++b) o[b] = silu(v[b]) * __shfl_xor_sync(0xffffffffu, v[b], 1);
        if ((lane & 1) || m + 1 >= a.M) return;
        float* y = a.y + (m >> 1);
#pragma unroll
        for (int b = 0; b < BP; ++b)
            if (b < a.B) y[(size_t)b * a.ldy] = o[b];
        return;
    }
    if (m >= a.M) return;
    float* y = a.y + m;
    if (a.epi == EPI_RESID) {
        const float* base = a.ybase ? a.ybase + m : y;
        float r[BP];
#pragma unroll
        for (int b = 0; b < BP; ++b) r[b] = b < a.B ? __ldcg(base + (size_t)b * a.ldy) : 0.f;
#pragma unroll
        for (int b = 0; b < BP; ++b) {
            if (b >= a.B) break;
            const float nv = r[b] + v[b];
            y[(size_t)b * a.ldy] = nv;
            if (a.y2) a.y2[(size_t)b * a.ldy2 + m] = nv;
        }
        return;
    }
#pragma unroll
    for (int b = 0; b < BP; ++b)
        if (b < a.B) y[(size_t)b * a.ldy] = v[b];
}

template <int BP>  // B_pad: 8, 16, 24 or 32
__global__ void __launch_bounds__(kLmThreads, 1) linear_mma_kernel(const LinearArgs a, uint16_t* xb, int S,
                                                                   int stage_bytes, uint32_t tmem_cols, float* part,
                                                                   int* counters, unsigned char* aux) {
    const LaunchStamp stamp(a.stamp ? a.stamp + (a.prepped ? 0 : 2) : nullptr);
    constexpr int N = 2 * BP;
    extern __shared__ unsigned char dsm_raw[];
    __shared__ LinMmaState st;
    __shared__ float rs_s[BP];  // norm_post: the rows' RMSNorm scales
    unsigned char* ring = (unsigned char*)(((uintptr_t)dsm_raw + 1023) & ~(uintptr_t)1023);
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int G = gridDim.x, cta = blockIdx.x;
    const int nkb = a.K / 64;
    const int ntiles = (a.M + 127) / 128;
    const int64_t U = (int64_t)ntiles * nkb;
    const int64_t u0 = unit_begin(cta, U, G), u1 = unit_begin(cta + 1, U, G);
    const int tile0 = (int)(u0 / nkb), tile1 = (int)((u1 - 1) / nkb);  // tiles this CTA touches

    if (t == 0) {
        for (int i = 0; i < S; ++i) {
            mbar_init(&st.full[i], 1);
            mbar_init(&st.empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&st.tfull[i], 1);
            mbar_init(&st.tempty[i], 4);
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
    if (warp == 4) {  // ---- TMA producer
        if (lane == 0) {
            const int total = (int)(u1 - u0);
            const int pre = min(S, total);
            const uint32_t xbytes = (uint32_t)N * 128u;
            const unsigned char* Wsrc = (const unsigned char*)a.W + (size_t)u0 * 16384;
            const uint64_t wpol = l2_evict_first();  // weights are read once per draft
            // the weights do not depend on earlier kernels: the first stages go out at once
            for (int it = 0; it < pre; ++it) {
                mbar_arrive_expect_tx(&st.full[it], 16384u + xbytes);
                bulk_g2s_hint(ring + (size_t)it * stage_bytes, Wsrc + (size_t)it * 16384, 16384, &st.full[it], wpol);
            }
            griddep_wait();
            int kx = (int)(u0 % nkb);  // activation block of the next copy: (u0 + it) % nkb
            for (int it = 0; it < pre; ++it) {
                bulk_g2s(ring + (size_t)it * stage_bytes + 16384, (const unsigned char*)xb + (size_t)kx * xbytes, xbytes,
                         &st.full[it]);
                if (++kx == nkb) kx = 0;
            }
            // iteration it >= S reuses slot it % S after the MMAs of iteration it - S: completion
            // (it - S) / S of empty[slot]
            int slot = 0;
            uint32_t pe = 0;
            for (int it = pre; it < total; ++it) {
                if (!mbar_wait_abortable(&st.empty[slot], pe, a.status, &st.abort)) break;
                unsigned char* dst = ring + (size_t)slot * stage_bytes;
                mbar_arrive_expect_tx(&st.full[slot], 16384u + xbytes);
                bulk_g2s_hint(dst, Wsrc + (size_t)it * 16384, 16384, &st.full[slot], wpol);
                bulk_g2s(dst + 16384, (const unsigned char*)xb + (size_t)kx * xbytes, xbytes, &st.full[slot]);
                if (++kx == nkb) kx = 0;
                if (++slot == S) { slot = 0; pe ^= 1u; }
            }
        }
    } else if (warp == 5) {  // ---- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, N);
            int64_t u = u0;
            int slot = 0;
            uint32_t pf = 0;  // phase bit of full[slot]
            for (int tile = tile0, j = 0; tile <= tile1; ++tile, ++j) {
                const int buf = j & 1;
                const int64_t ue = min(u1, (int64_t)(tile + 1) * nkb);
                if (!mbar_wait_abortable(&st.tempty[buf], ((uint32_t)(j >> 1) & 1u) ^ 1u, a.status, &st.abort)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem + (uint32_t)(buf * N);
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
                    for (int kk = 0; kk < 4; ++kk)
                        tc_mma(d_tmem, adesc + 2 * kk, bdesc + 2 * kk, idesc, (!first || kk) ? 1u : 0u);
                    tc_commit(&st.empty[slot]);
                    if (++slot == S) { slot = 0; pf ^= 1u; }
                }
                if (!ok) break;
                tc_commit(&st.tfull[buf]);
            }
        }
    } else {  // ---- epilogue warps 0..3: TMEM lane 32 w + l = output row of the tile
        float rsv[BP];  // per-row factor of the products (norm_post: the RMSNorm scales, else 1)
#pragma unroll
        for (int b = 0; b < BP; ++b) rsv[b] = 1.f;
        griddep_wait();  // the epilogue reads and writes activations of earlier kernels
        if (a.norm_post && a.pro == PRO_RMSNORM) {  // the rows' scales from the prep's sums of squares
            const float* sq = (const float*)(aux + kAuxSq);
            const int ny = (a.K / 8 + kXprepChunks - 1) / kXprepChunks;
            // row b = t / 4 sums column ranges y = t % 4, t % 4 + 4 (loads first, then in
            // order), then the four lanes combine in a fixed pattern
            const int b = t >> 2, p0 = t & 3;
            float q0 = 0.f, q1 = 0.f;
            if (b < BP) {
                if (p0 < ny) q0 = __ldcg(sq + (size_t)p0 * BP + b);
                if (p0 + 4 < ny) q1 = __ldcg(sq + (size_t)(p0 + 4) * BP + b);
            }
            float acc4 = q0 + q1;
            acc4 += __shfl_xor_sync(0xffffffffu, acc4, 1);
            acc4 += __shfl_xor_sync(0xffffffffu, acc4, 2);
            if (b < BP && p0 == 0) rs_s[b] = 1.0f / sqrtf(acc4 / (float)a.K + a.eps);
            named_sync(1, 128);  // (the four epilogue warps)
#pragma unroll
            for (int bb = 0; bb < BP; ++bb) rsv[bb] = rs_s[bb];
            // a deferred split tile of this phase is finished by the next phase's prep, which
            // reads these (the previous phase's scales were read by this phase's prep,
            // complete before this kernel's griddep_wait returned)
            if (cta == 0 && t < BP) ((float*)(aux + kAuxRs))[t] = rs_s[t];
        }
        const int r = warp * 32 + lane;
        for (int tile = tile0, j = 0; tile <= tile1; ++tile, ++j) {
            const int buf = j & 1;
            if (!mbar_wait_abortable(&st.tfull[buf], (uint32_t)(j >> 1) & 1u, a.status, &st.abort)) break;
            tc_fence_after();
            float acc[N];
            const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)(buf * N);
#pragma unroll
            for (int c = 0; c < N; c += 16) tc_ld16(taddr + c, acc + c);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&st.tempty[buf]);
            float v[BP];  // this CTA's products (a split tile's share stays unscaled)
#pragma unroll
            for (int b = 0; b < BP; ++b) v[b] = acc[b] + acc[BP + b];
            const int m = tile * 128 + r;
            const int c_first = unit_owner((int64_t)tile * nkb, U, G);
            const int c_last = unit_owner((int64_t)(tile + 1) * nkb - 1, U, G);
            if (c_first == c_last) {  // the whole tile was ours
#pragma unroll
                for (int b = 0; b < BP; ++b) v[b] *= rsv[b];
                lin_epilogue<BP>(a, m, v);
                continue;
            }
            // leave this CTA's share: slot 0 for its first tile, 1 for its last. Rows are
            // independent, so each warp finishes its own 32 rows (its own counter): no wait
            // on another warp.
            const int slot = tile == tile0 ? 0 : 1;
            float* pp = part + ((size_t)(cta * 2 + slot) * BP) * 128 + r;
#pragma unroll
            for (int b = 0; b < BP; ++b) pp[(size_t)b * 128] = v[b];
            if (a.defer) continue;  // the next phase's operand prep finishes this tile
            // lane 0's acquire-release add publishes the warp's shares (ordered before it by
            // the warp barrier) and, in the last warp to arrive, orders the reads below
            __syncwarp();
            int last = 0;
            if (lane == 0) last = atom_add_acq_rel_gpu(&counters[tile * 4 + warp], 1) == c_last - c_first;
            last = __shfl_sync(0xffffffffu, last, 0);
            if (!last) continue;
            float s[BP];
#pragma unroll
            for (int b = 0; b < BP; ++b) s[b] = 0.f;
            // (slot 1 only for c_first, when the tile is not its first: see prev_finish_t)
            const int cs_first = unit_begin(c_first, U, G) < (int64_t)tile * nkb ? 1 : 0;
            for (int c = c_first; c <= c_last; ++c) {
                const int cs = c == c_first ? cs_first : 0;
                const float* q = part + ((size_t)(c * 2 + cs) * BP) * 128 + r;
                float x[BP];
#pragma unroll
                for (int b = 0; b < BP; ++b) x[b] = __ldcg(q + (size_t)b * 128);
#pragma unroll
                for (int b = 0; b < BP; ++b) s[b] += x[b];
            }
#pragma unroll
            for (int b = 0; b < BP; ++b) s[b] *= rsv[b];
            lin_epilogue<BP>(a, m, s);
            if (lane == 0) counters[tile * 4 + warp] = 0;
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tc_dealloc(tmem, tmem_cols);
}

// ---- host side -----------------------------------------------------------------------------
namespace {

template <int BP>
cudaError_t set_attr(const DeviceInfo& dev) {
    return cudaFuncSetAttribute(linear_mma_kernel<BP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                dev.max_smem_optin - (int)sizeof(LinMmaState) - 256);
}

template <int BP>
cudaError_t launch_bp(const LinearArgs& a, uint16_t* xb, float* part, int* counters, unsigned char* aux,
                      const DeviceInfo& dev, cudaStream_t st, int grid) {
    constexpr int N = 2 * BP;
    const int stage_bytes = 16384 + N * 128;
    const size_t budget = (size_t)dev.max_smem_optin - sizeof(LinMmaState) - 256 - 1024;
    int S = (int)(budget / stage_bytes);
    S = S > kLinMaxStages ? kLinMaxStages : S;
    if (S < 2) return cudaErrorInvalidValue;
    const size_t smem = 1024 + (size_t)S * stage_bytes;
    uint32_t cols = 32;
    while (cols < (uint32_t)(2 * N)) cols <<= 1;
    return launch_k(linear_mma_kernel<BP>, dim3(grid), dim3(kLmThreads), smem, st, a.pdl, a, xb, S, stage_bytes, cols,
                    part, counters, aux);
}

}  // namespace

int linear_mma_bpad(int B) { return (B + 7) / 8 * 8; }

bool linear_mma_ok(int M, int K, int B) { return M > 0 && K % 64 == 0 && B >= 1 && B <= kLinMmaMaxBatch; }

size_t linear_mma_xb_bytes(int K, int B) { return (size_t)2 * linear_mma_bpad(B) * K * 2; }

int linear_mma_grid(int M, int K, const DeviceInfo& dev) {
    const int64_t U = (int64_t)((M + 127) / 128) * (K / 64);
    return (int)(U < dev.num_sms ? U : dev.num_sms);
}

size_t linear_mma_part_bytes(int B, const DeviceInfo& dev) {
    return (size_t)dev.num_sms * 2 * linear_mma_bpad(B) * 128 * sizeof(float);
}

namespace {
// the split-tile counters' offset in the counter buffer (after the RMSNorm scales and sums)
size_t tile_counter_offset(const DeviceInfo&) { return kAuxEnd; }
}  // namespace

size_t linear_mma_counter_bytes(int M_max, const DeviceInfo& dev) {
    return tile_counter_offset(dev) + 4 * (size_t)((M_max + 127) / 128) * sizeof(int);
}

float* linear_mma_rs(int* counters) { return (float*)((unsigned char*)counters + kAuxRs); }

cudaError_t linear_mma_prepare(const DeviceInfo& dev) {
    cudaError_t e = cudaFuncSetAttribute(xprep_row_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kXprepRowSmem);
    if (e != cudaSuccess) return e;
    if ((e = set_attr<8>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<16>(dev)) != cudaSuccess) return e;
    if ((e = set_attr<24>(dev)) != cudaSuccess) return e;
    return set_attr<32>(dev);
}

cudaError_t launch_linear_mma(const LinearArgs& a, uint16_t* xb, float* part, int* counters, const DeviceInfo& dev,
                              cudaStream_t st, cudaEvent_t after_prep) {
    if (!linear_mma_ok(a.M, a.K, a.B)) return cudaErrorInvalidValue;
    const int BP = linear_mma_bpad(a.B);
    unsigned char* aux = (unsigned char*)counters;
    int* tctr = (int*)(aux + tile_counter_offset(dev));
    const int grid = linear_mma_grid(a.M, a.K, dev);
    // finish + normalise a row per CTA (only when the scale goes on the operand)
    const bool row_cta = !a.norm_post && a.prev.active && a.pro == PRO_RMSNORM;
    if (row_cta && ((size_t)a.K * sizeof(float) > kXprepRowSmem || a.prev.epi == EPI_SWIGLU)) return cudaErrorInvalidValue;
    const int ny = (a.K / 8 + kXprepChunks - 1) / kXprepChunks;
    if (a.norm_post && a.pro == PRO_RMSNORM && (size_t)ny * kLinMmaMaxBatch * sizeof(float) > kAuxEnd - kAuxSq)
        return cudaErrorInvalidValue;
    if (a.prepped) {  // the operand is in place (the attention kernel wrote it)
        if (a.prev.active) return cudaErrorInvalidValue;
        switch (BP) {
            case 8: return launch_bp<8>(a, xb, part, tctr, aux, dev, st, grid);
            case 16: return launch_bp<16>(a, xb, part, tctr, aux, dev, st, grid);
            case 24: return launch_bp<24>(a, xb, part, tctr, aux, dev, st, grid);
            default: return launch_bp<32>(a, xb, part, tctr, aux, dev, st, grid);
        }
    }
    cudaError_t e = row_cta ? launch_k(xprep_row_kernel, dim3(BP), dim3(kRowThreads), (size_t)a.K * sizeof(float), st,
                                       a.pdl, a, BP, xb)
                            : launch_k(xprep_kernel, dim3(BP, ny), dim3(256), 0, st, a.pdl, a, BP, xb,
                                       (float*)(aux + kAuxSq));
    if (e != cudaSuccess) return e;
    if (after_prep && (e = cudaEventRecord(after_prep, st)) != cudaSuccess) return e;
    switch (BP) {
        case 8: return launch_bp<8>(a, xb, part, tctr, aux, dev, st, grid);
        case 16: return launch_bp<16>(a, xb, part, tctr, aux, dev, st, grid);
        case 24: return launch_bp<24>(a, xb, part, tctr, aux, dev, st, grid);
        default: return launch_bp<32>(a, xb, part, tctr, aux, dev, st, grid);
    }
}

}  // namespace fe

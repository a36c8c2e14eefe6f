// Split tiles of the tensor-core linear phases (fe_linear_mma.cu): the stream-K partition of
// a phase's (128-row tile, 64-column block) units over its CTAs, and the fix-up of a tile
// whose units fell to several CTAs, run by the reader of the phase's output when the phase
// deferred it: the next phase's operand prep, or the attention kernel after the QKV phase.
// Each CTA c leaves its share of such a tile in slot 0 (its first tile) or 1 (its last) of
// part[c] ([2][B_pad][128] floats).
#pragma once

#include "fe_kernels.h"
#include "fe_common.cuh"

namespace fe {

// ---- stream-K partition ---------------------------------------------------------------------
// first unit of CTA c when U units are split over G CTAs (32-bit division whenever U * G
// fits, as it does for every drafter shape: a 64-bit division is a long software sequence)
__device__ __forceinline__ int64_t unit_begin(int c, int64_t U, int G) {
    if (U * G <= 0xFFFFFFFFll) return (int64_t)((uint32_t)c * (uint32_t)U / (uint32_t)G);
    return (int64_t)c * U / G;
}

// the CTA whose range holds unit u: the largest c with floor(c U / G) <= u, i.e. with
// c U / G < u + 1, which is floor(((u + 1) G - 1) / U)
__device__ __forceinline__ int unit_owner(int64_t u, int64_t U, int G) {
    if (U * G <= 0xFFFFFFFFll) return (int)(((uint32_t)u * (uint32_t)G + (uint32_t)G - 1u) / (uint32_t)U);
    return (int)(((u + 1) * G - 1) / U);
}

// The previous phase's finished output at columns k0 .. k0 + 7 of row b (this phase's
// input). Columns of a tile the previous phase finished itself are read from where its
// epilogue stored them; a split tile's shares are summed in CTA order, its epilogue applied
// (residual add with the copy into y2, SwiGLU over the interleaved gate/up rows, or a plain
// store) and (STORE) the result stored, exactly as the phase's own fix-up would have.
// GLU: the previous phase is the SwiGLU one (16 rows per 8 columns); otherwise 8 rows.
template <bool GLU, bool STORE = true>
__device__ __forceinline__ void prev_finish_t(const LinearArgs::Prev& p, int BP, int b, int k0, float (&v)[8]) {
    constexpr int NR = GLU ? 16 : 8;  // the previous phase's rows behind these 8 columns
    constexpr bool glu = GLU;
    const int nkb = p.K / 64;
    const int64_t U = (int64_t)((p.M + 127) / 128) * nkb;
    const int row0 = glu ? 2 * k0 : k0;  // the previous phase's first output row of these columns
    const int tile = row0 / 128, r0 = row0 % 128;
    const int c_first = unit_owner((int64_t)tile * nkb, U, p.G);
    const int c_last = unit_owner((int64_t)(tile + 1) * nkb - 1, U, p.G);
    float* y = p.y + (size_t)b * p.ldy + k0;
    if (c_first == c_last) {  // a whole tile: the phase stored it
        const float4 q0 = __ldcg(reinterpret_cast<const float4*>(y)), q1 = __ldcg(reinterpret_cast<const float4*>(y) + 1);
        v[0] = q0.x; v[1] = q0.y; v[2] = q0.z; v[3] = q0.w; v[4] = q1.x; v[5] = q1.y; v[6] = q1.z; v[7] = q1.w;
        return;
    }
    // the residual (EPI_RESID) and the previous phase's RMSNorm scale are loaded before the
    // shares, so the round trips overlap
    const float prs = p.rs ? __ldcg(p.rs + b) : 1.f;
    float4 rb0 = make_float4(0.f, 0.f, 0.f, 0.f), rb1 = rb0;
    if (!GLU && p.epi == EPI_RESID) {
        const float* base = p.ybase ? p.ybase + (size_t)b * p.ldy + k0 : y;
        rb0 = __ldcg(reinterpret_cast<const float4*>(base));
        rb1 = __ldcg(reinterpret_cast<const float4*>(base) + 1);
    }
    float sm[NR];
#pragma unroll
    for (int i = 0; i < NR; ++i) sm[i] = 0.f;
    // the shares in batches of kPrevBatch CTAs: every load of a batch is issued before any
    // is summed (one L2 round trip per batch), the sums still in CTA order
    constexpr int kPrevBatch = GLU ? 4 : 8;  // (register budget: NR floats per share)
    // a tile is the first of every CTA after c_first that shares it (their shares sit in slot
    // 0); it is c_first's first tile only if c_first's range starts at the tile's first unit
    const int cs_first = unit_begin(c_first, U, p.G) < (int64_t)tile * nkb ? 1 : 0;
    for (int c0 = c_first; c0 <= c_last; c0 += kPrevBatch) {
        float x[kPrevBatch][NR];
#pragma unroll
        for (int j = 0; j < kPrevBatch; ++j) {
            const int c = c0 + j;
            if (c > c_last) break;
            const int cs = c == c_first ? cs_first : 0;
            const float4* q = reinterpret_cast<const float4*>(p.part + ((size_t)(c * 2 + cs) * BP + b) * 128 + r0);
#pragma unroll
            for (int i = 0; i < NR / 4; ++i) {
                const float4 w = __ldcg(q + i);
                x[j][4 * i] = w.x; x[j][4 * i + 1] = w.y; x[j][4 * i + 2] = w.z; x[j][4 * i + 3] = w.w;
            }
        }
#pragma unroll
        for (int j = 0; j < kPrevBatch; ++j) {
            if (c0 + j > c_last) break;
#pragma unroll
            for (int i = 0; i < NR; ++i) sm[i] += x[j][i];
        }
    }
    if (p.rs) {
#pragma unroll
        for (int i = 0; i < NR; ++i) sm[i] *= prs;
    }
    if constexpr (GLU) {
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = silu(sm[2 * e]) * sm[2 * e + 1];
    } else if (p.epi == EPI_RESID) {
        const float r[8] = {rb0.x, rb0.y, rb0.z, rb0.w, rb1.x, rb1.y, rb1.z, rb1.w};
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = r[e] + sm[e];
        if (STORE && p.y2) {
            float* y2 = p.y2 + (size_t)b * p.ldy2 + k0;
            reinterpret_cast<float4*>(y2)[0] = make_float4(v[0], v[1], v[2], v[3]);
            reinterpret_cast<float4*>(y2)[1] = make_float4(v[4], v[5], v[6], v[7]);
        }
    } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = sm[e];
    }
    if (STORE) {
        reinterpret_cast<float4*>(y)[0] = make_float4(v[0], v[1], v[2], v[3]);
        reinterpret_cast<float4*>(y)[1] = make_float4(v[4], v[5], v[6], v[7]);
    }
}

__device__ __forceinline__ void prev_finish(const LinearArgs::Prev& p, int BP, int b, int k0, float (&v)[8]) {
    if (p.epi == EPI_SWIGLU) prev_finish_t<true>(p, BP, b, k0, v);
    else prev_finish_t<false>(p, BP, b, k0, v);
}

}  // namespace fe

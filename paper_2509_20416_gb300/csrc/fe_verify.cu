// Lossless verification of a sampled draft tree (Sec. 2.4: the target scores the tree with
// tree attention and speculative sampling finds the longest accepted path; the paper names
// no variant). Read as recursive rejection sampling over each node's children in draw order
// (the multi-candidate form of speculative sampling: Leviathan et al. and Chen et al. 2023;
// Jeon et al. 2024), matching candidates drawn without replacement (Sec. 2.2):
//
//   at the current node, with r = the target's next-token distribution there and s = the
//   drafter's proposal of the next depth, the children are tested in draw order; child c
//   with token x is accepted iff u_acc[c] * s(x) <= r(x) (probability min(1, r(x) / s(x)));
//   on rejection r <- max(r - s, 0) renormalised and x leaves s (s renormalised over the
//   tokens not yet drawn: the law of the next draw). An accepted child becomes the current
//   node and r its own target distribution. When all children are rejected, or the node has
//   none, or N tokens were accepted, the bonus token is drawn from r by inverse CDF: the
//   smallest x with u_bonus[current] < r(0) + ... + r(x) (the last token with r > 0 when
//   rounding leaves the total below u).
//
// One CTA of 512 threads per sequence. s needs no buffer: after the draws X so far it is
// q / (1 - q(X)) off X and 0 on X. r is kept as an unnormalised residual w in a per-sequence
// buffer with its sum Z (r = w / Z), so a rejection is one pass over the vocabulary (read w
// or p and q, write the new w, sum it); the up to k - 1 tokens already drawn, whose s is 0,
// are put back after the pass from values saved before it. Every thread walks the tree with
// the same values (broadcast loads, a deterministic block sum), so the decisions agree.
// Precision: the elementwise residual is float32 (one rounding per operation); the sums
// that set the scale of everything after them -- each thread's share of Z (compensated),
// the block total and q's drawn mass, the CDF of the bonus draw -- are carried in double,
// so that their error does not grow with V.
#include <float.h>
#include <limits.h>

#include "fe_common.cuh"
#include "fe_kernels.h"

namespace fe {

namespace {

constexpr int kVsThreads = 512;
constexpr int kVsWarps = kVsThreads / 32;
constexpr int kVsMaxKids = 32;

// sum of one value per thread in double, the same bits in every thread (fixed order)
__device__ __forceinline__ double block_sum(double v, double* red) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    double s = 0.0;
#pragma unroll
    for (int w = 0; w < kVsWarps; ++w) s += red[w];
    __syncthreads();
    return s;
}

// compensated (Kahan) float accumulation: the sum's error stays near one rounding
struct KahanF {
    float s = 0.f, c = 0.f;
    __device__ __forceinline__ void add(float x) {
        const float y = x - c;
        const float t = s + y;
        c = (t - s) - y;
        s = t;
    }
    __device__ __forceinline__ double value() const { return (double)s - (double)c; }
};

__global__ void __launch_bounds__(kVsThreads) verify_sampled_kernel(const VerifySampledArgs a) {
    const int b = blockIdx.x, t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int T = a.T, N = a.N, V = a.V;
    __shared__ int kids[kVsMaxKids];
    __shared__ int nkids;
    __shared__ double red[kVsWarps];
    __shared__ int rem_tok[kVsMaxKids];   // tokens drawn (and rejected) at this node so far
    __shared__ float saved[kVsMaxKids];   // their r before a pass
    __shared__ double chunk_sum[kVsThreads];
    __shared__ int pick_s, last_s;
    const int* tk = a.tok + (size_t)b * T;
    const int* pr = a.parent + (size_t)b * T;
    const int* dp = a.depth + (size_t)b * T;
    const int* rk = a.rank + (size_t)b * (T - 1);  // node c >= 1 -> rk[c - 1]
    float* w = a.rbuf + (size_t)b * V;
    int cur = 0, n = 0;
    bool from_p = true;  // r is p[b][cur] itself; else r = w / Z
    double Z = 1.0;
    const float* pcur = a.p + (size_t)b * T * V;
    bool bad = false;

    for (;;) {
        // ---- the children of cur, in draw order (warp 0)
        if (warp == 0) {
            int m = 0;
            for (int c0 = 1; c0 < T; c0 += 32) {
                const int c = c0 + lane;
                const bool is = c < T && pr[c] == cur;
                const unsigned bal = __ballot_sync(0xffffffffu, is);
                const int pos = m + __popc(bal & ((1u << lane) - 1u));
                if (is && pos < kVsMaxKids) kids[pos] = c;
                m += __popc(bal);
            }
            m = min(m, kVsMaxKids);
            __syncwarp();
            const int c = lane < m ? kids[lane] : -1;
            const int rc = lane < m ? rk[c - 1] : INT_MAX;
            int place = 0;
            for (int j = 0; j < m; ++j) {
                const int rj = __shfl_sync(0xffffffffu, rc, j), cj = __shfl_sync(0xffffffffu, c, j);
                if (j != lane && (rj < rc || (rj == rc && cj < c))) ++place;
            }
            __syncwarp();
            if (lane < m) kids[place] = c;
            if (lane == 0) nkids = m;
        }
        __syncthreads();
        const int m = nkids;
        if (m == 0 || n >= N) break;
        const int dcur = dp[cur];
        if (dcur < 0 || dcur >= N) {
            bad = true;
            break;
        }
        const float* qs = a.q + ((size_t)b * N + dcur) * V;
        double removed = 0.0;  // q mass of the tokens drawn so far at this node
        int nrem = 0;
        int next = -1;
        for (int i = 0; i < m; ++i) {
            const int c = kids[i], x = tk[c];
            if (x < 0 || x >= V) {
                bad = true;
                break;
            }
            const float inv = removed < 1.0 ? (float)(1.0 / (1.0 - removed)) : 0.f;
            const float invZ = Z > 0.0 ? (float)(1.0 / Z) : 0.f;
            const float sx = qs[x] * inv;
            const float rx = from_p ? pcur[x] : w[x] * invZ;
            if (a.u_acc[(size_t)b * T + c] * sx <= rx) {
                next = c;
                break;
            }
            // rejected: r <- max(r - s, 0) (renormalised through Z); x leaves s
            if (t < nrem) {
                const int v = rem_tok[t];
                saved[t] = from_p ? pcur[v] : w[v] * invZ;
            }
            __syncthreads();
            KahanF part;
            for (int v = t; v < V; v += kVsThreads) {
                const float rv = from_p ? pcur[v] : w[v] * invZ;
                const float nv = fmaxf(rv - qs[v] * inv, 0.f);
                w[v] = nv;
                part.add(nv);
            }
            double sum = block_sum(part.value(), red);
            // the tokens drawn before x have s = 0: their r stays
            for (int j = 0; j < nrem; ++j) {
                const float sj = saved[j];
                sum += (double)sj - (double)fmaxf(sj - qs[rem_tok[j]] * inv, 0.f);
            }
            if (t < nrem) w[rem_tok[t]] = saved[t];
            Z = sum;
            from_p = false;
            __syncthreads();  // everyone has read rem_tok / saved; the fix-ups are written
            if (t == 0) rem_tok[nrem] = x;
            removed += (double)qs[x];
            ++nrem;
            __syncthreads();
        }
        if (next < 0) break;  // every child rejected (or a malformed node)
        if (t == 0) a.path[(size_t)b * N + n] = next;
        ++n;
        cur = next;
        from_p = true;
        Z = 1.0;
        pcur = a.p + ((size_t)b * T + cur) * V;
        __syncthreads();  // kids[] is rebuilt for the new node
    }
    if (bad && t == 0) atomicOr(a.status, ST_DEVICE);

    // ---- the bonus token: inverse CDF of r. Thread t sums a contiguous chunk; the chunks'
    // prefix gives each its start; the first chunk whose running sum passes u holds it.
    const double u = a.u_bonus[(size_t)b * T + cur];
    const float invZ = Z > 0.0 ? (float)(1.0 / Z) : 0.f;
    const int chunk = (V + kVsThreads - 1) / kVsThreads;
    const int v0 = min(V, t * chunk), v1 = min(V, v0 + chunk);
    double cs = 0.0;
    int last = -1;
    for (int v = v0; v < v1; ++v) {
        const float rv = from_p ? pcur[v] : w[v] * invZ;
        cs += (double)rv;
        if (rv > 0.f) last = v;
    }
    chunk_sum[t] = cs;
    if (t == 0) {
        pick_s = INT_MAX;
        last_s = -1;
    }
    __syncthreads();
    if (t == 0) {  // exclusive prefix of the chunk sums, in chunk order
        double run = 0.0;
        for (int j = 0; j < kVsThreads; ++j) {
            const double cj = chunk_sum[j];
            chunk_sum[j] = run;
            run += cj;
        }
    }
    if (last >= 0) atomicMax(&last_s, last);
    __syncthreads();
    double run = chunk_sum[t];
    for (int v = v0; v < v1; ++v) {
        run += (double)(from_p ? pcur[v] : w[v] * invZ);
        if (u < run) {
            atomicMin(&pick_s, v);
            break;
        }
    }
    __syncthreads();
    for (int i = n + t; i < N; i += kVsThreads) a.path[(size_t)b * N + i] = -1;
    if (t == 0) {
        a.n_accept[b] = n;
        a.bonus[b] = pick_s != INT_MAX ? pick_s : max(last_s, 0);
    }
}

}  // namespace

cudaError_t launch_verify_sampled(const VerifySampledArgs& a, int B, cudaStream_t st) {
    verify_sampled_kernel<<<B, kVsThreads, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace fe

// Backbone Expansion draft tree (Sec. 2.2) and its tree-attention mask (Sec. 2.4).
//
// Level-major node order with T = 1 + N k nodes: node 0 is the root (the last verified
// token, whose embedding fed the cascade); level i = 1..N holds the k candidates of
// depth i in rank order at nodes 1 + (i-1) k + r. Level 1 hangs under the root and
// level i >= 2 under node 1 + (i-2) k, the previous level's rank-0 (backbone) node, so
// the backbone is the chain of rank-0 nodes and every other node is a leaf. The
// ancestors of a node at depth i are the root and the backbone nodes of depths < i,
// which gives every mask entry in O(1): the kernel writes tokens, parents, depths and
// the T x T mask with one thread per element (one CTA per sequence).
#include "fe_kernels.h"
#include "fe_common.cuh"

namespace fe {

__global__ void tree_kernel(int N, int k, int V, const int* __restrict__ next_tok, const int* __restrict__ topk_id,
                            int* tok, int* parent, int* depth, uint8_t* mask, int* status,
                            unsigned long long* stamp_pair) {
    const LaunchStamp stamp(stamp_pair);
    const int b = blockIdx.x;
    const int T = 1 + N * k;
    bool bad = false;
    for (int n = threadIdx.x; n < T; n += blockDim.x) {
        int tk, dp, pr;
        if (n == 0) {
            tk = next_tok[b];
            dp = 0;
            pr = -1;
        } else {
            const int i = (n - 1) / k + 1, r = (n - 1) % k;
            tk = topk_id[((size_t)b * N + (i - 1)) * k + r];
            dp = i;
            pr = i == 1 ? 0 : 1 + (i - 2) * k;
        }
        if (tk < 0 || tk >= V) bad = true;
        tok[(size_t)b * T + n] = tk;
        parent[(size_t)b * T + n] = pr;
        depth[(size_t)b * T + n] = dp;
    }
    if (bad) atomicOr(status, ST_DEVICE);
    uint8_t* mb = mask + (size_t)b * T * T;
    for (int idx = threadIdx.x; idx < T * T; idx += blockDim.x) {
        const int a = idx / T, c = idx % T;
        const int da = a == 0 ? 0 : (a - 1) / k + 1;
        const int dc = c == 0 ? 0 : (c - 1) / k + 1;
        const bool backbone = c == 0 || (c - 1) % k == 0;
        mb[idx] = (uint8_t)(c == a || (backbone && dc < da));
    }
}

cudaError_t launch_tree(int B, int N, int k, int V, const int* next_tok, const int* topk_id, int* tok, int* parent,
                        int* depth, uint8_t* mask, int* status, cudaStream_t st, unsigned long long* stamp) {
    tree_kernel<<<B, 256, 0, st>>>(N, k, V, next_tok, topk_id, tok, parent, depth, mask, status, stamp);
    return cudaGetLastError();
}

// ---- verification side (Sec. 2.4, "Parallel Verification") --------------------------------
// One warp per sequence: the tree positions pos[a] = P_b + depth[a], then the greedy
// acceptance walk — from the root, the child (first in node order) whose token equals the
// target's greedy token after the current node is accepted and becomes current, until no
// child matches; the children of a node are found with one ballot per 32 nodes. Every
// index the walk follows comes from the node range, so malformed parents or tokens can
// only end the walk early.
__global__ void verify_kernel(int T, int max_path, const int* prefix_len, const int* tok, const int* parent,
                              const int* depth, const int* target_next, int* pos, int* path, int* n_accept,
                              int* bonus) {
    const int b = blockIdx.x, lane = threadIdx.x;
    const int* tk = tok + (size_t)b * T;
    const int* pr = parent + (size_t)b * T;
    const int* tn = target_next + (size_t)b * T;
    const int P = prefix_len[b];
    for (int a = lane; a < T; a += 32) pos[(size_t)b * T + a] = P + depth[(size_t)b * T + a];
    int cur = 0, n = 0;
    while (n < max_path) {
        const int want = tn[cur];
        int next = -1;
        for (int c0 = 1; c0 < T; c0 += 32) {
            const int c = c0 + lane;
            const unsigned m = __ballot_sync(0xffffffffu, c < T && pr[c] == cur && tk[c] == want);
            if (m) {
                next = c0 + __ffs(m) - 1;
                break;
            }
        }
        if (next < 0) break;
        if (lane == 0) path[(size_t)b * max_path + n] = next;
        ++n;
        cur = next;
    }
    for (int i = n + lane; i < max_path; i += 32) path[(size_t)b * max_path + i] = -1;
    if (lane == 0) {
        n_accept[b] = n;
        bonus[b] = tn[cur];
    }
}

cudaError_t launch_verify(int B, int T, int max_path, const int* prefix_len, const int* tok, const int* parent,
                          const int* depth, const int* target_next, int* pos, int* path, int* n_accept, int* bonus,
                          cudaStream_t st) {
    verify_kernel<<<B, 32, 0, st>>>(T, max_path, prefix_len, tok, parent, depth, target_next, pos, path, n_accept,
                                    bonus);
    return cudaGetLastError();
}

// One thread waits on an mbarrier that nothing will complete; the bounded wait gives up
// after timeout_ns and records ST_TIMEOUT. Exercises the failure path of every ring and
// grid wait without hanging the GPU.
__global__ void timeout_probe_kernel(int64_t timeout_ns, int* status) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        mbar_fence_init();
        mbar_wait(&bar, 0, status, timeout_ns);
    }
}

cudaError_t launch_timeout_probe(int64_t timeout_ns, int* status, cudaStream_t st) {
    timeout_probe_kernel<<<1, 32, 0, st>>>(timeout_ns, status);
    return cudaGetLastError();
}

}  // namespace fe

// Internal launch interface of the drafter's kernels (host side). Not part of the ABI.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "fe_draft.h"

namespace fe {

// Launch `kern` on `st`; with pdl the launch may overlap the previous kernel of the stream
// (programmatic stream serialization; the kernel calls griddepcontrol.wait before it
// touches anything an earlier kernel wrote).
template <typename... P, typename... A>
inline cudaError_t launch_k(void (*kern)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, bool pdl,
                            A&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kern, std::forward<A>(args)...);
}

// status-word bits (combined with atomicOr; the host maps them back to fe_status)
enum : int {
    ST_CAPACITY = 1,  // prefix_len[b] + 1 > max_seq or negative
    ST_DEVICE = 2,    // a token id or page id out of range
    ST_TIMEOUT = 4,   // a bounded wait ran out
};

// how a weight-streaming phase stages its activations X[b][k]
enum Prologue : int {
    PRO_F32 = 0,         // x is float32 [B, ldx]
    PRO_STORAGE = 1,     // x is in the storage type [B, ldx]
    PRO_RMSNORM = 2,     // x float32; X = gamma * x / sqrt(mean(x^2) + eps)
    PRO_CONCAT_EMB = 3,  // X = concat(x[b][0:d_split] (float32), embed[tok[b]] (storage))
};

// ---- weight-streaming linear phase: Y = epilogue(W . prologue(X)) ---------------------
enum Epilogue : int {
    EPI_STORE = 0,   // y[b, m] = acc
    EPI_RESID = 1,   // y[b, m] += acc; y2[b, m] = the new y (if y2)
    EPI_SWIGLU = 2,  // rows (2j, 2j+1) are (gate_j, up_j): y[b, j] = silu(gate) * up
};

// tile-packed weight layout (fe_pack.cu / fe_stream.cuh)
size_t packed_bytes(int M, int K, int es);
cudaError_t launch_pack_tiles(const void* src, void* dst, int M, int K, int es, cudaStream_t st);

struct LinearArgs {
    const void* W;  // tile-packed [ceil(M/4)*4, K] storage type, 16-byte aligned, K % 8 == 0
    int M, K;
    int B;  // activation rows
    // prologue
    int pro;
    const void* x;
    int ldx;
    const void* gamma;
    float eps;
    const void* embed;
    const int* tok;
    int d_split;
    int vocab;
    // epilogue
    int epi;
    float* y;
    int ldy;
    float* y2;
    int ldy2;
    const float* ybase;  // EPI_RESID: y = ybase + acc (same layout as y) when set, else y += acc
    int slots;           // streaming kernel: pipeline slots per warp (0: the default)
    int* status;
    bool pdl;  // launch overlapping the previous kernel (programmatic dependent launch)
    // in-graph timing (fe_profile_graph): the (start, end) stamp pair of this phase's
    // first kernel, the next kernel of the phase at stamp + 2; null when not profiling
    unsigned long long* stamp = nullptr;
    // tensor-core path: whether another tensor-core phase follows (next_W non-null) and
    // reads this phase's output, which lets this phase defer its split tiles to it
    const void* next_W = nullptr;
    // tensor-core path, deferred split-tile reduction. With defer, a tile whose units are
    // split between CTAs leaves each CTA's share in the partial buffer and nothing else; the
    // next tensor-core phase's operand prep, given this phase as `prev`, sums the shares in
    // CTA order, applies this phase's epilogue and stores the result before using it (the
    // same operations, in the same order, as the in-kernel reduction).
    int defer = 0;
    // tensor-core path: the operand is already in place (written by the attention kernel)
    int prepped = 0;
    struct Prev {
        int active = 0;
        const float* part = nullptr;  // the partial buffer the phase wrote
        int M = 0, K = 0, G = 0;      // its shape and grid
        int epi = 0;
        float* y = nullptr;
        int ldy = 0;
        float* y2 = nullptr;
        int ldy2 = 0;
        const float* ybase = nullptr;
        // the phase normalised its input after the product (norm_post): its per-row RMSNorm
        // scales, which multiply the summed shares before its epilogue
        const float* rs = nullptr;
    } prev;
    // tensor-core path, RMSNorm input: the operand is gamma * x (the prep runs column-parallel
    // and leaves per-CTA sums of squares) and the per-row scale 1 / sqrt(mean(x^2) + eps)
    // multiplies the products; otherwise the prep scales the operand itself (a whole-row pass)
    int norm_post = 0;
};

struct DeviceInfo {
    int num_sms;
    int max_smem_optin;
};

cudaError_t linear_prepare(const DeviceInfo& dev);
cudaError_t launch_linear(fe_dtype dt, const LinearArgs& a, const DeviceInfo& dev, cudaStream_t st);
// number of kernels launch_linear() issues for these shapes (always 1)
inline int linear_launches() { return 1; }

// A persistent stack of consecutive linear phases at B = 1 (one launch; grid-wide barriers
// between phases on *barrier, which must be zero at launch). ph[0].pdl decides the launch's
// programmatic dependence; the others' pdl is ignored.
constexpr int kMaxStackPhases = 4;
struct StackArgs {
    LinearArgs ph[kMaxStackPhases];
    int nph;
    uint32_t* barrier;
};
int stack_slots(int k_max, const DeviceInfo& dev);
cudaError_t launch_stack(fe_dtype dt, const StackArgs& sa, const DeviceInfo& dev, cudaStream_t st);

// ---- tensor-core linear phase (bf16 weights, batches of 1..kLinMmaMaxBatch) -------------
// W packed by launch_pack_mma (interleaved gate/up rows for EPI_SWIGLU); xb scratch of
// linear_mma_xb_bytes(K_max, max_batch); part of linear_mma_part_bytes(); counters:
// 4 * ceil(M_max / 128) ints, zero between calls. Two kernels: operand prep + product.
constexpr int kLinMmaMaxBatch = 32;
int linear_mma_bpad(int B);
bool linear_mma_ok(int M, int K, int B);
size_t linear_mma_xb_bytes(int K, int B);
size_t linear_mma_part_bytes(int B, const DeviceInfo& dev);
int linear_mma_grid(int M, int K, const DeviceInfo& dev);
cudaError_t linear_mma_prepare(const DeviceInfo& dev);
// the completion-counter buffer: the last norm_post phase's per-row scales and its prep's
// sums of squares, then 4 * ceil(M_max / 128) ints of split-tile counters; zero at init
size_t linear_mma_counter_bytes(int M_max, const DeviceInfo& dev);
// where a norm_post phase leaves its per-row scales (inside the counter buffer)
float* linear_mma_rs(int* counters);
// after_prep (optional): an event recorded on st between the two kernels it launches
cudaError_t launch_linear_mma(const LinearArgs& a, uint16_t* xb, float* part, int* counters, const DeviceInfo& dev,
                              cudaStream_t st, cudaEvent_t after_prep = nullptr);

// ---- LM head + fused softmax statistics + per-slab top-k ------------------------------
struct LmHeadArgs {
    const void* W;  // lm_head, tile-packed [ceil(V/4)*4, d]
    const void* gamma;  // final_norm [d]
    int V, d;
    int R;  // rows of hidden states (N * B), row r = i * B + b
    int B, N;
    const float* hid;  // [R, d] float32
    float eps;
    float inv_temp;
    int top_k;
    int n_slabs;  // filled by lmhead_plan()
    int* part_id;      // [R, n_slabs, top_k]
    float* part_val;   // [R, n_slabs, top_k]
    float* part_ms;    // [R, n_slabs, 2] (max, sum of exp) of logit * inv_temp
    int* counters;     // [ceil(R / 8)] slab-completion counters, zero between calls
    // tensor-core LM head (N * B <= 16): with these, (vocabulary tile, 64-column block) units
    // are split evenly over the CTAs; a tile split between CTAs c and c + 1 is finished by c
    // from c + 1's partial. split_part [n_slabs][128][R_pad] floats; split_flag [n_slabs]
    // ints, zero between calls. Without them each CTA takes whole tiles.
    float* split_part;
    int* split_flag;
    float* dbg_logits; // [B, N, V] or null
    int* topk_id;       // [B, N, k]
    float* topk_logit;  // [B, N, k]
    float* topk_prob;   // [B, N, k]
    float* lse;         // [B, N]
    int* status;
    bool pdl;
    // stochastic drafting (Sec. 2.2): with sample, each row's candidates are the top_k keys
    // logit * inv_temp + G (fe_sample.cuh) instead of the top_k logits; the partials then
    // hold keys in part_val and the candidates' logits in part_lg [R, n_slabs, top_k]; the
    // merge orders the drawn set by logit and writes each one's draw position to topk_rank
    int sample = 0;
    unsigned long long seed = 0;
    float* part_lg = nullptr;
    int* topk_rank = nullptr;  // [B, N, k] or null
    // in-graph timing: stamp pairs of the head's kernels (operand prep, product, merge in
    // that order; the CUDA-core head uses the first); null when not profiling
    unsigned long long* stamp = nullptr;
};
cudaError_t lmhead_prepare(const DeviceInfo& dev);
int lmhead_slabs(int V, const DeviceInfo& dev);
int lmhead_launches(int R, int d, const DeviceInfo& dev);
cudaError_t launch_lmhead(fe_dtype dt, const LmHeadArgs& a, const DeviceInfo& dev, cudaStream_t st);

// tensor-core LM head (bf16 storage, N*B <= 16 rows, d % 64 == 0): W in the swizzled MMA
// layout (launch_pack_mma), zb scratch of lmhead_mma_zb_bytes(); n_slabs = CTAs
bool lmhead_mma_ok(const LmHeadArgs& a);
size_t lmhead_mma_zb_bytes(int R, int d);
size_t lmhead_mma_split_bytes(int R, const DeviceInfo& dev);  // split_part
size_t mma_packed_bytes(int M, int K);
cudaError_t launch_pack_mma(const void* src, void* dst, int M, int K, cudaStream_t st);
cudaError_t lmhead_mma_prepare(const DeviceInfo& dev);
// Three kernels: operand prep, the product with per-slab statistics and top-k, the per-row
// merge; after_prep / after_main (optional): events recorded on st after the first two
cudaError_t launch_lmhead_mma(const LmHeadArgs& a, uint16_t* zb, const DeviceInfo& dev, cudaStream_t st,
                              cudaEvent_t after_prep = nullptr, cudaEvent_t after_main = nullptr);

// wide tensor-core LM head (bf16, 16 < R <= 256 rows, top_k <= 16, d % 64 == 0): the same
// packed W, z rounded to bf16 (zb of lmhead_wide_zb_bytes()), n_slabs = lmhead_wide_slabs()
// CTAs; three kernels (operand prep, product + per-slab top-k, per-row merge)
bool lmhead_wide_ok(const LmHeadArgs& a);
size_t lmhead_wide_zb_bytes(int R, int d);
int lmhead_wide_slabs(int V, const DeviceInfo& dev);
cudaError_t lmhead_wide_prepare(const DeviceInfo& dev);
cudaError_t launch_lmhead_wide(const LmHeadArgs& a, uint16_t* zb, const DeviceInfo& dev, cudaStream_t st,
                               cudaEvent_t after_prep = nullptr, cudaEvent_t after_main = nullptr);

// Read-only view of what a handle holds for its LM head (for entry points outside
// fe_runtime.cu). Returns false for a null handle.
struct LmHeadView {
    const void* lm_head;     // packed for the tensor cores (mma) or tile-packed
    const void* final_norm;  // [d]
    bool mma;
    fe_dtype dtype;
    int d, V, N, max_batch, top_k_max, n_slabs;
    float eps;
    int* status;
    DeviceInfo dev;
    int device;  // the CUDA device the handle's memory lives on
};
bool handle_lmhead_view(const fe_handle* h, LmHeadView* v);
// record a message for fe_last_error_detail() (calling thread)
void set_error_detail(const char* msg);
// fe_noalloc.cu: look up the allocation-free LM head's scratch array on the current device
// (once per device; called by fe_draft_init with the handle's device current)
cudaError_t noalloc_resolve_scratch(int device);

// ---- decode attention ----------------------------------------------------------------
struct AttnArgs {
    const float* qkv;  // [B, (H + 2 Hkv) hd] float32, before RoPE
    void* kc;          // layer cache (storage type)
    void* vc;
    const int* prefix_len;  // [B]
    const int* page_table;  // [B, max_pages] or null
    int max_pages, n_pages, page_size, max_seq;
    const float* rope_cs;   // [max_seq, hd/2, 2] (cos, sin)
    int B, H, Hkv, hd;
    int split, n_split;     // keys per work item, work items per (sequence, KV head)
    float* part;            // [B, H, n_split, hd + 4]: value sum [hd], max, sum of weights, padding
    int* counters;          // [B, Hkv] split-completion counters, zero between calls
    float* out;             // [B, H * hd]
    int* status;
    bool pdl;
    // rows of qkv / out: sequence b's is row b * row_stride + row_off (a draft: 1, 0); the
    // row sits at position prefix_len[b] + pos_add; with n_rows, sequences with
    // n_rows[b] <= pos_add are skipped (a commit of accepted rows)
    int row_stride = 1, row_off = 0, pos_add = 0;
    const int* n_rows = nullptr;
    unsigned long long* stamp = nullptr;  // in-graph timing stamp pair, or null
    // bytes at the start of dynamic shared memory the last split's combine may use (set by
    // launch_attention: the K/V slots, or more when every split's partials then fit at once)
    int combine_smem = 0;
    // batched drafts: the outputs go straight into the O projection's tensor-core operand (bf16
    // hi/lo, the 128-byte-swizzled layout of fe_tc.cuh, rows [0, xb_bpad) hi and [xb_bpad,
    // 2 xb_bpad) lo per 64-column block) instead of `out`, so that phase needs no prep kernel
    uint16_t* xb = nullptr;
    int xb_bpad = 0;
    // batched drafts: the QKV phase left the tiles it split between CTAs to this kernel, which
    // sums their shares for the columns it reads (fe_splitk.cuh); qprev_bpad is that phase's
    // operand row padding (its shares' row stride)
    LinearArgs::Prev qprev{};
    int qprev_bpad = 0;
};
int attn_split(int B, int Hkv, int max_seq, const DeviceInfo& dev);
cudaError_t attention_prepare();
cudaError_t launch_attention(fe_dtype dt, const AttnArgs& a, cudaStream_t st);
inline int attention_launches() { return 1; }

// ---- draft tree + failure-detection probe ------------------------------------------------
cudaError_t launch_tree(int B, int N, int k, int V, const int* next_tok, const int* topk_id, int* tok, int* parent,
                        int* depth, uint8_t* mask, int* status, cudaStream_t st, unsigned long long* stamp = nullptr);
cudaError_t launch_timeout_probe(int64_t timeout_ns, int* status, cudaStream_t st);
// commit (fe_commit.cu): gather rows i0 .. i0 + nb - 1 of every sequence into a dense block
cudaError_t launch_commit_gather(const void* feat, const int* tok, const int* n_rows, int B, int L, int i0, int nb,
                                 int row_bytes, void* cfeat, int* ctok, cudaStream_t st);
// training-objective forward (fe_loss.cu): ce, fl [B, N]; total [B]
cudaError_t launch_loss(int N, int B, int V, int d, const float* logits, const float* teacher, const float* hidden,
                        const float* feat, float alpha, float beta, float decay, float* ce, float* fl, float* total,
                        cudaStream_t st);
cudaError_t launch_verify(int B, int T, int max_path, const int* prefix_len, const int* tok, const int* parent,
                          const int* depth, const int* target_next, int* pos, int* path, int* n_accept, int* bonus,
                          cudaStream_t st);
// lossless verification of a sampled tree (fe_verify.cu): one CTA per sequence
struct VerifySampledArgs {
    int T, N, V;
    const int *tok, *parent, *depth;  // [B, T] trees in fe_build_tree's layout
    const int* rank;                  // [B, T - 1]: node c >= 1's draw position at rank[c - 1]
    const float* q;                   // [B, N, V] the drafter's proposal per depth
    const float* p;                   // [B, T, V] the target's distribution after each node
    const float *u_acc, *u_bonus;     // [B, T]
    float* rbuf;                      // [B, V] scratch: each sequence's residual
    int *path, *n_accept, *bonus;     // [B, N], [B], [B]
    int* status;
};
cudaError_t launch_verify_sampled(const VerifySampledArgs& a, int B, cudaStream_t st);

}  // namespace fe

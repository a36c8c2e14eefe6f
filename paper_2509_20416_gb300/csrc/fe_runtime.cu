// C ABI of the drafter (include/fe_draft.h): handle, weight packing, RoPE table, scratch
// buffers, the launch sequence of one draft, and its CUDA-graph replay.
//
// One draft (Eq. 1, Eq. 2, Sec. 2.1) is this stream-ordered sequence:
//   g  = W_fuse concat(l, m, h)                 linear, prologue: storage -> float
//   x  = W_in concat(g, Embed[next_tok])        linear, prologue: concat with the embedding
//   for each layer L_i:
//     qkv = W_qkv RMSNorm(x; gamma_1)            linear, prologue: RMSNorm
//     o   = attention(RoPE(q), cache_i + own row) split-KV attention + combine (writes slot P_b)
//     x  += W_o o                                linear, epilogue: residual add
//     a   = silu(W_gate u) * (W_up u), u = RMSNorm(x; gamma_2)   linear over the interleaved
//                                                [gate; up] rows, epilogue: SwiGLU
//     x  += W_down a;  h_i = x                   linear, epilogue: residual add + copy to h_i
//   logits of all N*B rows h_i through RMSNorm(gamma_out) and the LM head, fused with the
//   softmax statistics and a per-slab top-k; then a merge per row.
// The sequence is captured once per distinct argument set into a CUDA graph on an
// internal stream and replayed on the caller's stream.
#include <math.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <cstdlib>
#include <new>
#include <vector>

#include "fe_kernels.h"

using namespace fe;

namespace {

struct LayerPacked {
    const void *attn_norm, *w_qkv, *w_o, *mlp_norm, *w_gu, *w_down;
};

struct GraphKey {
    fe_forward_args args;
    std::vector<void*> kc, vc;
    bool operator==(const GraphKey& o) const {
        const fe_forward_args &x = args, &y = o.args;
        return x.B == y.B && x.top_k == y.top_k && x.temperature == y.temperature && x.feat == y.feat &&
               x.next_tok == y.next_tok && x.prefix_len == y.prefix_len && x.page_table == y.page_table &&
               x.n_pages == y.n_pages && x.topk_id == y.topk_id && x.topk_logit == y.topk_logit &&
               x.topk_prob == y.topk_prob && x.lse == y.lse && x.dbg_logits == y.dbg_logits &&
               x.dbg_hidden == y.dbg_hidden && x.sample == y.sample && x.seed == y.seed &&
               x.topk_rank == y.topk_rank && kc == o.kc && vc == o.vc;
    }
};

// what a fe_draft_step_host graph was captured for
struct HostKey {
    int B = 0, top_k = 0;
    float temperature = 0.f;
    int sample = 0;
    uint64_t seed = 0;
    const void* feat_direct = nullptr;  // the caller's pinned features, copied from directly
    const int32_t* page_table = nullptr;
    int n_pages = 0;
    std::vector<void*> kc, vc;
    bool operator==(const HostKey& o) const {
        return B == o.B && top_k == o.top_k && temperature == o.temperature && sample == o.sample &&
               seed == o.seed && feat_direct == o.feat_direct &&
               page_table == o.page_table &&
               n_pages == o.n_pages && kc == o.kc && vc == o.vc;
    }
};

// fe_draft_step_host's packing of one step's inputs and outputs (16-byte aligned pieces),
// the same in the pinned staging buffers and in their device copies
struct StepLayout {
    size_t feat, tok, plen, in_bytes;
    size_t id, logit, prob, lse, rank, ttok, tpar, tdep, tmask, out_bytes;
};

StepLayout step_layout(const fe_config& c, size_t es, int B, int k) {
    auto al = [](size_t x) { return (x + 15) & ~(size_t)15; };
    const size_t b = (size_t)B, N = (size_t)c.n_layers, T = 1 + N * (size_t)k;
    StepLayout L{};
    size_t o = 0;
    L.feat = o; o = al(o + b * 3 * (size_t)c.d * es);
    L.tok = o; o = al(o + b * 4);
    L.plen = o; o = al(o + b * 4);
    L.in_bytes = o;
    o = 0;
    L.id = o; o = al(o + b * N * k * 4);
    L.logit = o; o = al(o + b * N * k * 4);
    L.prob = o; o = al(o + b * N * k * 4);
    L.lse = o; o = al(o + b * N * 4);
    L.rank = o; o = al(o + b * N * k * 4);
    L.ttok = o; o = al(o + b * T * 4);
    L.tpar = o; o = al(o + b * T * 4);
    L.tdep = o; o = al(o + b * T * 4);
    L.tmask = o; o = al(o + b * T * T);
    L.out_bytes = o;
    return L;
}

}  // namespace

struct fe_handle {
    fe_config cfg;
    int device = 0;
    DeviceInfo dev{};
    size_t es = 2;
    void* wbuf = nullptr;
    const void *w_fuse = nullptr, *w_in = nullptr, *embed = nullptr, *lm_head = nullptr, *final_norm = nullptr;
    std::vector<LayerPacked> layers;
    float* rope_cs = nullptr;
    void* cfeat = nullptr;  // commit: one block's gathered feature rows [<= 32, 3d]
    int* ctok = nullptr;    // commit: their tokens
    void* sbuf = nullptr;
    float *g = nullptr, *x = nullptr, *qkv = nullptr, *o = nullptr, *act = nullptr, *hid = nullptr;
    float* x0 = nullptr;  // the cascade input x0 (Eq. 1), kept for layer 1 and the parallel ablation
    float* attn_part = nullptr;
    int* lm_part_id = nullptr;
    float *lm_part_val = nullptr, *lm_part_ms = nullptr;
    float* lm_part_lg = nullptr;  // sampling: the logits of the partials' candidates
    float* vs_rbuf = nullptr;     // fe_verify_sampled: each sequence's residual distribution [max_batch, V]
    int* status = nullptr;
    int* attn_counters = nullptr;
    int* lm_counters = nullptr;
    bool lm_mma = false;      // LM head packed for (and run on) the tensor cores
    bool lin_mma = false;     // linear phases packed for (and run on) the tensor cores
    bool lin_defer = true;    // tensor-core phases leave split tiles to the next phase's prep
    bool lin_normpost = true; // tensor-core RMSNorm phases: the scale on the products (column-parallel prep)
    bool attn_operand = true; // tensor-core O projection: its operand written by the attention kernel
    int lm_16row = -1;        // up to 16 hidden rows: 1 the 16-row tensor-core LM head, 0 the wide one where it fits, -1 by vocabulary size
    uint16_t* lin_xb = nullptr;  // tensor-core linear: bf16 hi/lo activation operand
    float* lin_part = nullptr;   // tensor-core linear: per-CTA partials of split tiles
    int* lin_counters = nullptr; // tensor-core linear: per (tile, warp) completion counters
    bool use_stack = false;      // B = 1 drafts run their linear phases as persistent stacks
    uint32_t* stack_bar = nullptr;  // grid-barrier counters, one per stack of a draft
    uint16_t* lm_zb = nullptr;  // tensor-core LM head: bf16 hi/lo operand of the hidden rows
    float* lm_split_part = nullptr;  // tensor-core LM head: parts of tiles split between CTAs
    int* lm_split_flag = nullptr;    // ... and their hand-off flags (zero between calls)
    int attn_split_rows = 0, attn_nsplit = 0, lm_slabs = 0;
    cudaStream_t cap = nullptr;
    cudaGraphExec_t gexec = nullptr;
    GraphKey gkey;
    bool use_graph = true;
    bool use_pdl = true;
    std::vector<cudaEvent_t> prof_ev;  // fe_profile_forward's events (created on first use)
    // fe_profile_graph: the stamp pairs (device, allocated on first use), the stamped
    // graph and what it was captured for
    unsigned long long* prof_stamps = nullptr;
    int prof_stamp_cap = 0;
    cudaGraphExec_t pexec = nullptr;
    GraphKey pkey;
    fe_tree ptree{};
    std::vector<int32_t> pkinds;
    // fe_draft_step_host: pinned staging of a step's inputs and outputs, their device
    // copies (sized for max_batch and top_k_max) and the step's graph
    unsigned char *hs_in = nullptr, *hs_out = nullptr, *ds_in = nullptr, *ds_out = nullptr;
    cudaGraphExec_t hexec = nullptr;
    HostKey hkey;
};

namespace {

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

thread_local char g_detail[256] = "";

fe_status fail(cudaError_t e, const char* what, int line) {
    snprintf(g_detail, sizeof(g_detail), "%s (fe_runtime.cu:%d): %s", what, line, cudaGetErrorString(e));
    if (e == cudaErrorMemoryAllocation) return FE_ERR_OOM;
    return FE_ERR_CUDA;
}

#define from_cuda(call) (((_fe_e = (call)) == cudaSuccess) ? FE_OK : fail(_fe_e, #call, __LINE__))

#define FE_TRY(call)                                       \
    do {                                                   \
        cudaError_t _e = (call);                           \
        if (_e != cudaSuccess) return fail(_e, #call, __LINE__); \
    } while (0)

// Every call that enqueues work requires the handle's device to be the calling thread's
// current device: the handle's weights, scratch and status word live there, and a launch
// on another device would reach them across devices (or fault).
fe_status check_device(const fe_handle* h) {
    int dev = -1;
    const cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(e, "cudaGetDevice", __LINE__);
    if (dev != h->device) {
        snprintf(g_detail, sizeof(g_detail), "the current CUDA device (%d) is not the handle's device (%d)", dev,
                 h->device);
        return FE_ERR_INVALID_ARG;
    }
    return FE_OK;
}

bool valid_config(const fe_config* c) {
    if (!c) return false;
    if (c->d <= 0 || c->n_heads <= 0 || c->n_kv_heads <= 0 || c->ffn <= 0 || c->vocab <= 0) return false;
    if (c->n_heads % c->n_kv_heads) return false;
    if (c->n_layers < 1 || c->n_layers > 16) return false;
    if (c->top_k_max < 1 || c->top_k_max > 32 || c->top_k_max > c->vocab) return false;
    if (c->max_batch < 1 || c->max_seq < 1 || c->page_size < 0) return false;
    if (!(c->rope_theta > 0.f) || !(c->rms_eps >= 0.f)) return false;
    if (c->dtype != FE_F32 && c->dtype != FE_BF16) return false;
    if (c->head_dim <= 0 || c->head_dim % 2) return false;
    if (c->parallel_layers != 0 && c->parallel_layers != 1) return false;
    return true;
}

// legal shapes the library's kernels cover
bool supported_config(const fe_config* c) {
    const int G = c->n_heads / c->n_kv_heads;
    if (c->head_dim != 64 && c->head_dim != 128) return false;
    if (G != 1 && G != 2 && G != 4 && G != 8) return false;
    // every matrix row must be a whole number of 16-byte vectors
    if (c->d % 8 || c->ffn % 8 || (c->n_heads * c->head_dim) % 8) return false;
    return true;
}

struct Sizes {
    size_t w_fuse, w_in, embed, lm_head, norm, qkv, wo, gu, down;
};

// The profilers' recorder. Event mode (fe_profile_forward, ev set): ev[0] is recorded
// before the first launch and ev[j + 1] after launch j. Stamp mode (fe_profile_graph,
// stamps set): launch j gets the stamp pair stamps + 2 j. Either way launch j's family is
// kinds[j].
struct Prof {
    cudaEvent_t* ev;
    unsigned long long* stamps;
    int32_t* kinds;
    int cap, n;
};

inline cudaError_t mark(Prof* pf, int kind, cudaStream_t st) {
    if (!pf) return cudaSuccess;
    if (pf->n >= pf->cap) return cudaErrorInvalidValue;
    pf->kinds[pf->n] = kind;
    ++pf->n;
    return pf->ev ? cudaEventRecord(pf->ev[pf->n], st) : cudaSuccess;
}

// the stamp pair of the next launch (stamp mode), else null
inline unsigned long long* next_stamp(const Prof* pf) {
    return pf && pf->stamps && pf->n < pf->cap ? pf->stamps + 2 * (size_t)pf->n : nullptr;
}

// bytes of each matrix in the tile-packed layout (rows padded to a multiple of 4); the
// embedding and the norm gains stay in their canonical layout
Sizes weight_sizes(const fe_config& c, size_t es, bool mma) {
    const int d = c.d, H = c.n_heads, Hkv = c.n_kv_heads, hd = c.head_dim, F = c.ffn, V = c.vocab;
    const int e = (int)es;
    auto pk = [&](int M, int K) { return mma ? mma_packed_bytes(M, K) : packed_bytes(M, K, e); };
    Sizes s;
    s.w_fuse = pk(d, 3 * d);
    s.w_in = pk(d, 2 * d);
    s.embed = (size_t)V * d * es;
    s.lm_head = packed_bytes(V, d, e);
    s.norm = (size_t)d * es;
    s.qkv = pk((H + 2 * Hkv) * hd, d);
    s.wo = pk(d, H * hd);
    s.gu = pk(2 * F, d);
    s.down = pk(d, F);
    return s;
}

// Pipeline slots of a streaming linear phase next to attention: 3 (the default) for a matrix
// of 64 MB or more, whose stream outlasts attention's early start; 2 for a smaller one, so
// that attention's CTAs fit beside it on the SMs (measured on the LLaMA-3.1-8B and
// Vicuna-13B shapes).
int near_attention_slots(int M, int K, int es) { return (size_t)M * K * es >= ((size_t)64 << 20) ? 0 : 2; }

fe_status enqueue_forward(fe_handle* h, const fe_forward_args* a, cudaStream_t st, Prof* pf = nullptr) {
    const fe_config& c = h->cfg;
    const int B = a->B, d = c.d, H = c.n_heads, Hkv = c.n_kv_heads, hd = c.head_dim, F = c.ffn, V = c.vocab;
    const int N = c.n_layers, nqkv = (H + 2 * Hkv) * hd;
    const fe_dtype dt = c.dtype;
    const bool pdl = h->use_pdl && !(pf && pf->ev);  // event-profiled launches do not overlap
    const bool stacked = h->use_stack && B == 1;
    if (stacked) {
        // the stacks' barrier counters start at zero in every draft
        FE_TRY(cudaMemsetAsync(h->stack_bar, 0, (size_t)(N + 1) * sizeof(uint32_t), st));
    }
    if (pf && pf->ev) FE_TRY(cudaEventRecord(pf->ev[0], st));
    // one linear phase: the CUDA-core streaming kernel, or operand prep + tensor-core product
    // persistent stacks: linear phases are queued and launched together at the next
    // attention (or at the LM head)
    StackArgs sq{};
    sq.nph = 0;
    int nstack = 0;
    auto flush_stack = [&]() -> fe_status {
        if (sq.nph == 0) return FE_OK;
        sq.barrier = h->stack_bar + nstack;
        sq.ph[0].stamp = next_stamp(pf);
        cudaError_t e = launch_stack(dt, sq, h->dev, st);
        if (e != cudaSuccess) return fail(e, "linear stack launch", __LINE__);
        if ((e = mark(pf, FE_KERNEL_LINEAR, st)) != cudaSuccess) return fail(e, "profiling event", __LINE__);
        sq.nph = 0;
        ++nstack;
        return FE_OK;
    };
    // a tensor-core phase followed by another defers its split tiles to that phase's operand
    // prep (LinearArgs::defer / prev): `pending` carries the deferring phase to the next one
    LinearArgs::Prev pending{};
    const void* next_in = nullptr;  // the buffer the next tensor-core phase reads (set by next_is below)
    auto linear = [&](const LinearArgs& L0) -> fe_status {
        cudaError_t e;
        LinearArgs L = L0;
        L.stamp = stacked ? nullptr : next_stamp(pf);
        if (h->lin_mma) {
            if (pending.active && pending.y != L.x) {  // a deferred phase must be finished by its reader
                set_error_detail("internal: a deferred linear phase is not followed by its reader");
                return FE_ERR_CUDA;
            }
            L.prev = pending;
            pending = LinearArgs::Prev{};
            L.norm_post = h->lin_normpost ? 1 : 0;
            L.defer = h->lin_defer && L.next_W && next_in == L.y ? 1 : 0;
            if (L.defer) {
                pending.active = 1;
                pending.part = h->lin_part;
                pending.M = L.M;
                pending.K = L.K;
                pending.G = linear_mma_grid(L.M, L.K, h->dev);
                pending.epi = L.epi;
                pending.y = L.y;
                pending.ldy = L.ldy;
                pending.y2 = L.y2;
                pending.ldy2 = L.ldy2;
                pending.ybase = L.ybase;
                pending.rs = L.norm_post && L.pro == PRO_RMSNORM ? linear_mma_rs(h->lin_counters) : nullptr;
            }
        }
        if (stacked) {
            if (sq.nph == kMaxStackPhases) {
                const fe_status r = flush_stack();
                if (r != FE_OK) return r;
            }
            sq.ph[sq.nph++] = L;
            return FE_OK;
        }
        if (h->lin_mma) {
            if (pf && !L.prepped) {
                if (pf->n + 2 > pf->cap) return FE_ERR_INVALID_ARG;
                pf->kinds[pf->n++] = FE_KERNEL_LINEAR_PREP;
            }
            e = launch_linear_mma(L, h->lin_xb, h->lin_part, h->lin_counters, h->dev, st,
                                  pf && pf->ev && !L.prepped ? pf->ev[pf->n] : nullptr);
        } else {
            e = launch_linear(dt, L, h->dev, st);
        }
        if (e != cudaSuccess) return fail(e, "linear phase launch", __LINE__);
        if ((e = mark(pf, FE_KERNEL_LINEAR, st)) != cudaSuccess) return fail(e, "profiling event", __LINE__);
        return FE_OK;
    };
    fe_status lrc;
#define FE_LINEAR(L)                                \
    do {                                            \
        if ((lrc = linear(L)) != FE_OK) return lrc; \
    } while (0)


    LinearArgs la{};
    la.status = h->status;
    la.eps = c.rms_eps;
    la.B = B;
    // tensor-core phases: the phase that follows and the buffer it reads (a phase defers its
    // split tiles only to a tensor-core successor that reads its output)
    auto next_is = [&](const void* W, int, int, const void* in) {
        la.next_W = h->lin_mma ? W : nullptr;
        next_in = W ? in : nullptr;
    };
    // g = W_fuse concat(l, m, h). The first kernel of a draft waits for everything before it
    // on the stream (it is launched without programmatic dependence); later kernels may
    // overlap their predecessor's tail (see griddep_wait()).
    la.pdl = false;
    la.W = h->w_fuse; la.M = d; la.K = 3 * d;
    la.pro = PRO_STORAGE; la.x = a->feat; la.ldx = 3 * d;
    la.epi = EPI_STORE; la.y = h->g; la.ldy = d; la.y2 = nullptr;
    next_is(h->w_in, d, 2 * d, h->g);
    FE_LINEAR(la);
    la.pdl = pdl;
    // x0 = W_in concat(g, e)
    la.W = h->w_in; la.M = d; la.K = 2 * d;
    la.pro = PRO_CONCAT_EMB; la.x = h->g; la.ldx = d; la.embed = h->embed; la.tok = a->next_tok;
    la.d_split = d; la.vocab = V;
    la.epi = EPI_STORE; la.y = h->x0; la.ldy = d;
    next_is(h->layers[0].w_qkv, nqkv, d, h->x0);
    FE_LINEAR(la);

    AttnArgs aa{};
    aa.qkv = h->qkv; aa.prefix_len = a->prefix_len; aa.page_table = a->page_table;
    aa.page_size = c.page_size; aa.max_seq = c.max_seq; aa.n_pages = a->n_pages;
    aa.max_pages = c.page_size > 0 ? (c.max_seq + c.page_size - 1) / c.page_size : 0;
    aa.rope_cs = h->rope_cs; aa.B = B; aa.H = H; aa.Hkv = Hkv; aa.hd = hd;
    aa.split = h->attn_split_rows; aa.n_split = h->attn_nsplit;
    aa.part = h->attn_part; aa.counters = h->attn_counters; aa.out = h->o; aa.status = h->status;
    aa.pdl = pdl;
    // batched handles: attention writes the O projection's tensor-core operand itself
    const bool o_direct = h->lin_mma && h->attn_operand && !stacked;
    if (o_direct) {
        aa.xb = h->lin_xb;
        aa.xb_bpad = linear_mma_bpad(B);
    }

    for (int i = 0; i < N; ++i) {
        const LayerPacked& L = h->layers[i];
        // qkv = W_qkv RMSNorm(x)
        la.W = L.w_qkv; la.M = nqkv; la.K = d;
        // the phases next to attention leave room for its CTAs unless they are large
        la.slots = near_attention_slots(nqkv, d, (int)h->es);
        // L_1 (and every L_i of the parallel ablation) reads x0; the cascade's L_i reads h_{i-1}
        const bool from_x0 = i == 0 || c.parallel_layers;
        la.pro = PRO_RMSNORM; la.x = from_x0 ? h->x0 : h->x; la.ldx = d; la.gamma = L.attn_norm;
        la.epi = EPI_STORE; la.y = h->qkv; la.ldy = nqkv; la.y2 = nullptr;
        // attention follows; on batched handles it finishes this phase's split tiles itself
        next_is(h->lin_mma ? L.w_qkv : nullptr, 0, 0, h->qkv);
        FE_LINEAR(la);
        aa.qprev = pending;
        aa.qprev_bpad = pending.active ? linear_mma_bpad(B) : 0;
        pending = LinearArgs::Prev{};
        // attention over the layer's cache (+ own row), appends slot P_b
        aa.kc = a->k_cache[i]; aa.vc = a->v_cache[i];
        if ((lrc = flush_stack()) != FE_OK) return lrc;
        aa.stamp = next_stamp(pf);
        FE_TRY(launch_attention(dt, aa, st));
        FE_TRY(mark(pf, FE_KERNEL_ATTENTION, st));
        // x += W_o o
        la.slots = near_attention_slots(d, H * hd, (int)h->es);
        la.W = L.w_o; la.M = d; la.K = H * hd;
        la.pro = PRO_F32; la.x = h->o; la.ldx = H * hd;
        la.epi = EPI_RESID; la.y = h->x; la.ldy = d; la.y2 = nullptr; la.ybase = from_x0 ? h->x0 : nullptr;
        next_is(L.w_gu, 2 * F, d, h->x);
        la.prepped = o_direct ? 1 : 0;
        FE_LINEAR(la);
        la.prepped = 0;
        // a = silu(W_gate u) * (W_up u), u = RMSNorm(x)
        la.slots = 0;
        la.W = L.w_gu; la.M = 2 * F; la.K = d;
        la.pro = PRO_RMSNORM; la.x = h->x; la.ldx = d; la.gamma = L.mlp_norm; la.ybase = nullptr;
        la.epi = EPI_SWIGLU; la.y = h->act; la.ldy = F;
        next_is(L.w_down, d, F, h->act);
        FE_LINEAR(la);
        // x += W_down a; h_i = x
        la.W = L.w_down; la.M = d; la.K = F;
        la.pro = PRO_F32; la.x = h->act; la.ldx = F;
        la.epi = EPI_RESID; la.y = h->x; la.ldy = d; la.y2 = h->hid + (size_t)i * B * d; la.ldy2 = d;
        if (i + 1 < N) next_is(h->layers[i + 1].w_qkv, nqkv, d, c.parallel_layers ? h->x0 : h->x);
        else next_is(nullptr, 0, 0, nullptr);  // the LM head follows
        FE_LINEAR(la);
    }

    if ((lrc = flush_stack()) != FE_OK) return lrc;
    const float inv_temp = a->temperature > 0.f ? 1.0f / a->temperature : 1.0f;
    LmHeadArgs lm{};
    lm.W = h->lm_head; lm.gamma = h->final_norm; lm.V = V; lm.d = d; lm.R = N * B; lm.B = B; lm.N = N;
    lm.hid = h->hid; lm.eps = c.rms_eps; lm.inv_temp = inv_temp; lm.top_k = a->top_k; lm.n_slabs = h->lm_slabs;
    lm.part_id = h->lm_part_id; lm.part_val = h->lm_part_val; lm.part_ms = h->lm_part_ms;
    lm.counters = h->lm_counters; lm.dbg_logits = a->dbg_logits; lm.status = h->status;
    lm.topk_id = a->topk_id; lm.topk_logit = a->topk_logit; lm.topk_prob = a->topk_prob; lm.lse = a->lse;
    lm.sample = a->sample ? 1 : 0; lm.seed = a->seed; lm.part_lg = h->lm_part_lg; lm.topk_rank = a->topk_rank;
    lm.pdl = pdl;
    lm.stamp = next_stamp(pf);
    // Up to 16 rows the wide kernel (z as bf16 hi + lo) takes greedy calls on vocabularies of
    // at least four 128-entry tiles per CTA (it hands out whole tiles, so fewer leave CTAs
    // idle at the end): it streams the 1-2 GB heads of 128256 entries 10-11 % faster than the
    // 16-row kernel (stream-K units), which keeps the smaller vocabularies, top_k > 16 and
    // sampled calls (the wide kernel draws a row's deviates on one thread: 532 vs 388 us per
    // 70B-shaped draft)
    const bool wide_small = h->lm_16row == 0 ||
                            (h->lm_16row < 0 && !a->sample && (V + 127) / 128 >= 4 * h->dev.num_sms);
    if (h->lm_mma && N * B <= 16 && !(wide_small && lmhead_wide_ok(lm))) {
        lm.n_slabs = std::min(h->dev.num_sms, (V + 127) / 128);  // one CTA per SM, at least one 128-row tile each
        lm.split_part = h->lm_split_part;  // (tile, column block) units split evenly over the CTAs
        lm.split_flag = h->lm_split_flag;
        if (pf) {
            if (pf->n + 3 > pf->cap) return FE_ERR_INVALID_ARG;
            pf->kinds[pf->n] = FE_KERNEL_LM_PREP;
            pf->kinds[pf->n + 1] = FE_KERNEL_LM_HEAD;
            pf->n += 2;
        }
        FE_TRY(launch_lmhead_mma(lm, h->lm_zb, h->dev, st, pf && pf->ev ? pf->ev[pf->n - 1] : nullptr,
                                 pf && pf->ev ? pf->ev[pf->n] : nullptr));
        FE_TRY(mark(pf, FE_KERNEL_LM_HEAD, st));
    } else if (h->lm_mma) {
        lm.n_slabs = lmhead_wide_slabs(V, h->dev);
        if (pf) {
            if (pf->n + 3 > pf->cap) return FE_ERR_INVALID_ARG;
            pf->kinds[pf->n] = FE_KERNEL_LM_PREP;
            pf->kinds[pf->n + 1] = FE_KERNEL_LM_HEAD;
            pf->n += 2;
        }
        FE_TRY(launch_lmhead_wide(lm, h->lm_zb, h->dev, st, pf && pf->ev ? pf->ev[pf->n - 1] : nullptr,
                                  pf && pf->ev ? pf->ev[pf->n] : nullptr));
        FE_TRY(mark(pf, FE_KERNEL_LM_HEAD, st));
    } else {
        FE_TRY(launch_lmhead(dt, lm, h->dev, st));
        FE_TRY(mark(pf, FE_KERNEL_LM_HEAD, st));
    }
    if (a->dbg_hidden) {
        FE_TRY(cudaMemcpyAsync(a->dbg_hidden, h->hid, (size_t)N * B * d * sizeof(float), cudaMemcpyDeviceToDevice,
                               st));
        FE_TRY(mark(pf, FE_KERNEL_COPY, st));
    }
    return FE_OK;
#undef FE_LINEAR
}

// The commit of accepted rows (include/fe_draft.h): blocks of up to 32 rows (whole row
// indices of every sequence); per block the rows are gathered, then Eq. 1 and the cascade
// run over them like a draft's rows, with one attention launch per row index (row i of a
// sequence reads the rows before it from the cache, so they must be stored first).
fe_status enqueue_commit(fe_handle* h, const fe_commit_args* a, cudaStream_t st) {
    const fe_config& c = h->cfg;
    const int B = a->B, d = c.d, H = c.n_heads, Hkv = c.n_kv_heads, hd = c.head_dim, F = c.ffn, V = c.vocab;
    const int N = c.n_layers, nqkv = (H + 2 * Hkv) * hd;
    const fe_dtype dt = c.dtype;
    const bool pdl = h->use_pdl;
    const int nb_max = std::max(1, std::min(a->L, 32 / B));
    auto linear = [&](const LinearArgs& L) -> fe_status {
        const cudaError_t e = h->lin_mma ? launch_linear_mma(L, h->lin_xb, h->lin_part, h->lin_counters, h->dev, st, nullptr)
                                         : launch_linear(dt, L, h->dev, st);
        return e == cudaSuccess ? FE_OK : fail(e, "commit linear phase launch", __LINE__);
    };
    fe_status rc;
    for (int i0 = 0; i0 < a->L; i0 += nb_max) {
        const int nb = std::min(nb_max, a->L - i0), R = B * nb;
        FE_TRY(launch_commit_gather(a->feat, a->tok, a->n_rows, B, a->L, i0, nb, 3 * d * (int)h->es, h->cfeat, h->ctok,
                                    st));
        LinearArgs la{};
        la.status = h->status;
        la.eps = c.rms_eps;
        la.B = R;
        la.pdl = false;  // the gather kernel does not trigger programmatic launch
        la.W = h->w_fuse; la.M = d; la.K = 3 * d;
        la.pro = PRO_STORAGE; la.x = h->cfeat; la.ldx = 3 * d;
        la.epi = EPI_STORE; la.y = h->g; la.ldy = d;
        if ((rc = linear(la)) != FE_OK) return rc;
        la.pdl = pdl;
        la.W = h->w_in; la.M = d; la.K = 2 * d;
        la.pro = PRO_CONCAT_EMB; la.x = h->g; la.ldx = d; la.embed = h->embed; la.tok = h->ctok;
        la.d_split = d; la.vocab = V;
        la.epi = EPI_STORE; la.y = h->x0; la.ldy = d;
        if ((rc = linear(la)) != FE_OK) return rc;

        AttnArgs aa{};
        aa.qkv = h->qkv; aa.prefix_len = a->prefix_len; aa.page_table = a->page_table;
        aa.page_size = c.page_size; aa.max_seq = c.max_seq; aa.n_pages = a->n_pages;
        aa.max_pages = c.page_size > 0 ? (c.max_seq + c.page_size - 1) / c.page_size : 0;
        aa.rope_cs = h->rope_cs; aa.B = B; aa.H = H; aa.Hkv = Hkv; aa.hd = hd;
        aa.split = h->attn_split_rows; aa.n_split = h->attn_nsplit;
        aa.part = h->attn_part; aa.counters = h->attn_counters; aa.out = h->o; aa.status = h->status;
        aa.pdl = pdl;
        aa.row_stride = nb; aa.n_rows = a->n_rows;
        for (int l = 0; l < N; ++l) {
            const LayerPacked& Lw = h->layers[l];
            const bool from_x0 = l == 0 || c.parallel_layers;
            la.W = Lw.w_qkv; la.M = nqkv; la.K = d;
            la.pro = PRO_RMSNORM; la.x = from_x0 ? h->x0 : h->x; la.ldx = d; la.gamma = Lw.attn_norm;
            la.epi = EPI_STORE; la.y = h->qkv; la.ldy = nqkv; la.y2 = nullptr; la.ybase = nullptr;
            if ((rc = linear(la)) != FE_OK) return rc;
            aa.kc = a->k_cache[l]; aa.vc = a->v_cache[l];
            for (int j = 0; j < nb; ++j) {
                aa.row_off = j;
                aa.pos_add = i0 + j;
                // row j reads the rows the launches before it appended: it must not start
                // (and copy cache rows) before they finish
                aa.pdl = j == 0 && pdl;
                FE_TRY(launch_attention(dt, aa, st));
            }
            aa.pdl = pdl;
            la.W = Lw.w_o; la.M = d; la.K = H * hd;
            la.pro = PRO_F32; la.x = h->o; la.ldx = H * hd;
            la.epi = EPI_RESID; la.y = h->x; la.ldy = d; la.ybase = from_x0 ? h->x0 : nullptr;
            if ((rc = linear(la)) != FE_OK) return rc;
            la.W = Lw.w_gu; la.M = 2 * F; la.K = d;
            la.pro = PRO_RMSNORM; la.x = h->x; la.ldx = d; la.gamma = Lw.mlp_norm; la.ybase = nullptr;
            la.epi = EPI_SWIGLU; la.y = h->act; la.ldy = F;
            if ((rc = linear(la)) != FE_OK) return rc;
            la.W = Lw.w_down; la.M = d; la.K = F;
            la.pro = PRO_F32; la.x = h->act; la.ldx = F;
            la.epi = EPI_RESID; la.y = h->x; la.ldy = d;
            if ((rc = linear(la)) != FE_OK) return rc;
        }
    }
    return FE_OK;
}

bool forward_args_ok(const fe_handle* h, const fe_forward_args* a) {
    if (!h || !a) return false;
    const fe_config& c = h->cfg;
    if (a->B < 1 || a->B > c.max_batch) return false;
    if (a->top_k < 1 || a->top_k > c.top_k_max) return false;
    if (!a->feat || !a->next_tok || !a->prefix_len || !a->k_cache || !a->v_cache) return false;
    if (!a->topk_id || !a->topk_logit || !a->topk_prob || !a->lse) return false;
    for (int i = 0; i < c.n_layers; ++i)
        if (!a->k_cache[i] || !a->v_cache[i]) return false;
    if (c.page_size > 0 && (!a->page_table || a->n_pages < 1)) return false;
    if (!(a->temperature == a->temperature)) return false;  // NaN
    if (a->sample && !(a->temperature > 0.f)) return false;  // draws need a temperature
    if (h->lin_mma && (reinterpret_cast<uintptr_t>(a->feat) & 15)) return false;  // read as 16-byte vectors
    return true;
}

void release(fe_handle* h) {
    if (!h) return;
    for (cudaEvent_t e : h->prof_ev) cudaEventDestroy(e);
    if (h->gexec) cudaGraphExecDestroy(h->gexec);
    if (h->pexec) cudaGraphExecDestroy(h->pexec);
    if (h->prof_stamps) cudaFree(h->prof_stamps);
    if (h->hexec) cudaGraphExecDestroy(h->hexec);
    if (h->hs_in) cudaFreeHost(h->hs_in);
    if (h->hs_out) cudaFreeHost(h->hs_out);
    if (h->ds_in) cudaFree(h->ds_in);
    if (h->ds_out) cudaFree(h->ds_out);
    if (h->cap) cudaStreamDestroy(h->cap);
    if (h->wbuf) cudaFree(h->wbuf);
    if (h->sbuf) cudaFree(h->sbuf);
    delete h;
}

}  // namespace

void fe::set_error_detail(const char* msg) { snprintf(g_detail, sizeof(g_detail), "%s", msg); }

bool fe::handle_lmhead_view(const fe_handle* h, LmHeadView* v) {
    if (!h || !v) return false;
    v->lm_head = h->lm_head;
    v->final_norm = h->final_norm;
    v->mma = h->lm_mma;
    v->dtype = h->cfg.dtype;
    v->d = h->cfg.d;
    v->V = h->cfg.vocab;
    v->N = h->cfg.n_layers;
    v->max_batch = h->cfg.max_batch;
    v->top_k_max = h->cfg.top_k_max;
    v->n_slabs = h->lm_mma ? std::min(h->dev.num_sms, (h->cfg.vocab + 127) / 128) : h->lm_slabs;
    v->eps = h->cfg.rms_eps;
    v->status = h->status;
    v->dev = h->dev;
    v->device = h->device;
    return true;
}

extern "C" {

const char* fe_status_str(fe_status s) {
    switch (s) {
        case FE_OK: return "ok";
        case FE_ERR_INVALID_ARG: return "invalid argument";
        case FE_ERR_UNSUPPORTED: return "unsupported shape";
        case FE_ERR_CUDA: return "CUDA error";
        case FE_ERR_OOM: return "out of device memory";
        case FE_ERR_CAPACITY: return "prefix does not fit the cache";
        case FE_ERR_TIMEOUT: return "device wait timed out";
        case FE_ERR_DEVICE: return "device-side range check failed";
    }
    return "unknown status";
}

fe_status fe_draft_init(const fe_config* cfg, const fe_weights* w, void* stream, fe_handle** out) {
    if (!out) return FE_ERR_INVALID_ARG;
    *out = nullptr;
    if (!valid_config(cfg) || !w) return FE_ERR_INVALID_ARG;
    if (!w->w_fuse || !w->w_in || !w->embed || !w->lm_head || !w->final_norm || !w->layers) return FE_ERR_INVALID_ARG;
    for (int i = 0; i < cfg->n_layers; ++i) {
        const fe_layer_weights& L = w->layers[i];
        if (!L.attn_norm || !L.w_qkv || !L.w_o || !L.mlp_norm || !L.w_gate || !L.w_up || !L.w_down)
            return FE_ERR_INVALID_ARG;
    }
    if (!supported_config(cfg)) return FE_ERR_UNSUPPORTED;

    fe_handle* h = new (std::nothrow) fe_handle();
    if (!h) return FE_ERR_OOM;
    cudaError_t _fe_e = cudaSuccess;
    h->cfg = *cfg;
    const char* g = getenv("FE_DRAFT_GRAPH");
    h->use_graph = !(g && g[0] == '0');
    const char* pd = getenv("FE_DRAFT_PDL");
    h->use_pdl = !(pd && pd[0] == '0');
    cudaStream_t st = (cudaStream_t)stream;
    fe_status rc = FE_OK;
    do {
        const fe_config& c = h->cfg;
        h->es = c.dtype == FE_F32 ? 4 : 2;
        if ((rc = from_cuda(cudaGetDevice(&h->device))) != FE_OK) break;
        if ((rc = from_cuda(cudaDeviceGetAttribute(&h->dev.num_sms, cudaDevAttrMultiProcessorCount, h->device))) != FE_OK)
            break;
        if ((rc = from_cuda(cudaDeviceGetAttribute(&h->dev.max_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin,
                                                   h->device))) != FE_OK)
            break;
        if ((rc = from_cuda(linear_prepare(h->dev))) != FE_OK) break;
        if ((rc = from_cuda(lmhead_prepare(h->dev))) != FE_OK) break;
        if ((rc = from_cuda(attention_prepare())) != FE_OK) break;
        if ((rc = from_cuda(lmhead_mma_prepare(h->dev))) != FE_OK) break;
        if ((rc = from_cuda(linear_mma_prepare(h->dev))) != FE_OK) break;
        if ((rc = from_cuda(lmhead_wide_prepare(h->dev))) != FE_OK) break;
        // the allocation-free LM head's fixed scratch array: its address on this device is
        // looked up here, so that entry point itself never loads a module or allocates
        if ((rc = from_cuda(noalloc_resolve_scratch(h->device))) != FE_OK) break;
        // the linear phases run on the tensor cores for batched handles (bf16, every K a
        // multiple of 64, at most kLinMmaMaxBatch sequences); FE_DRAFT_LINEAR_MMA=1 / 0
        // forces the choice where the shapes allow it
        {
            const fe_config& c = h->cfg;
            const bool shapes = c.dtype == FE_BF16 && c.max_batch <= kLinMmaMaxBatch && c.d % 64 == 0 &&
                                c.ffn % 64 == 0 && (c.n_heads * c.head_dim) % 64 == 0;
            const char* lm = getenv("FE_DRAFT_LINEAR_MMA");
            h->lin_mma = shapes && (lm ? lm[0] == '1' : c.max_batch > 8);
            // FE_DRAFT_STACK=1: B = 1 drafts on the CUDA-core path run their linear phases as
            // persistent stacks (when one pipeline slot per warp fits next to the largest
            // activation row). Off by default: measured on GB300, the separate launches with
            // programmatic dependent launch inside the CUDA graph are faster (720 vs 762 us
            // per Vicuna-13B-shaped draft); the stacks win only without programmatic launch.
            const int kmax = std::max({3 * c.d, c.ffn, c.n_heads * c.head_dim});
            const char* df = getenv("FE_DRAFT_LIN_DEFER");
            h->lin_defer = !(df && df[0] == '0');
            // FE_DRAFT_LIN_NORMPOST=0: an RMSNorm phase's prep scales the operand itself (one
            // CTA per row when it also finishes the previous phase's split tiles; kept for
            // comparison)
            const char* np = getenv("FE_DRAFT_LIN_NORMPOST");
            h->lin_normpost = !(np && np[0] == '0');
            // FE_DRAFT_ATTN_OPERAND=0: the attention output goes through float32 and the O
            // projection's own prep (kept for comparison)
            const char* ao = getenv("FE_DRAFT_ATTN_OPERAND");
            h->attn_operand = !(ao && ao[0] == '0');
            const char* sk = getenv("FE_DRAFT_STACK");
            h->use_stack = !h->lin_mma && sk && sk[0] == '1' && stack_slots(kmax, h->dev) >= 1;
        }

        // ---- packed weights: one allocation, every matrix 256-byte aligned ----
        const Sizes sz = weight_sizes(c, h->es, h->lin_mma);
        size_t total = align256(sz.w_fuse) + align256(sz.w_in) + align256(sz.embed) +
                       std::max(align256(sz.lm_head), align256(mma_packed_bytes(c.vocab, c.d))) + align256(sz.norm);
        total += (size_t)c.n_layers *
                 (2 * align256(sz.norm) + align256(sz.qkv) + align256(sz.wo) + align256(sz.gu) + align256(sz.down));
        if ((rc = from_cuda(cudaMalloc(&h->wbuf, total))) != FE_OK) break;
        char* p = (char*)h->wbuf;
        const int es = (int)h->es;
        // staging buffer for one canonical [M, K] matrix before it is tile-packed
        const size_t stage_bytes = std::max({(size_t)c.vocab * c.d, (size_t)c.d * 3 * c.d,
                                             (size_t)2 * c.ffn * c.d,
                                             (size_t)(c.n_heads + 2 * c.n_kv_heads) * c.head_dim * c.d}) * h->es;
        void* staging = nullptr;
        if ((rc = from_cuda(cudaMalloc(&staging, stage_bytes))) != FE_OK) break;
        auto put = [&](const void* src, size_t bytes) -> const void* {
            void* dst = p;
            p += align256(bytes);
            if ((_fe_e = cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDefault, st)) != cudaSuccess)
                rc = fail(_fe_e, "copy of a weight", __LINE__);
            return dst;
        };
        // a layer matrix in the layout of the linear path in use; the LM head is packed below
        auto pack = [&](const void* staged, void* dst, int M, int K) -> cudaError_t {
            return h->lin_mma ? launch_pack_mma(staged, dst, M, K, st) : launch_pack_tiles(staged, dst, M, K, es, st);
        };
        auto packed_size = [&](int M, int K) {
            return h->lin_mma ? mma_packed_bytes(M, K) : packed_bytes(M, K, es);
        };
        auto put_packed = [&](const void* src, int M, int K) -> const void* {
            void* dst = p;
            p += align256(packed_size(M, K));
            if ((_fe_e = cudaMemcpyAsync(staging, src, (size_t)M * K * es, cudaMemcpyDefault, st)) != cudaSuccess ||
                (_fe_e = pack(staging, dst, M, K)) != cudaSuccess)
                rc = fail(_fe_e, "copy or packing of a weight matrix", __LINE__);
            return dst;
        };
        const int dm = c.d, nq = (c.n_heads + 2 * c.n_kv_heads) * c.head_dim, hq = c.n_heads * c.head_dim;
        h->w_fuse = put_packed(w->w_fuse, dm, 3 * dm);
        h->w_in = put_packed(w->w_in, dm, 2 * dm);
        h->embed = put(w->embed, sz.embed);
        // the LM head runs on the tensor cores when every call fits one of their two kernels
        // (bf16, d a multiple of 64, at most 16 hidden rows; or at most 256 rows with
        // top_k_max <= 16); it is then packed in the swizzled MMA layout
        {
            const int64_t rmax = (int64_t)c.n_layers * c.max_batch;
            h->lm_mma = c.dtype == FE_BF16 && c.d % 64 == 0 && c.d <= 16384 &&
                        (rmax <= 16 || (rmax <= 256 && c.top_k_max <= 16)) &&
                        !(getenv("FE_DRAFT_LMHEAD_CUDA_CORES") && getenv("FE_DRAFT_LMHEAD_CUDA_CORES")[0] == '1');
            // FE_DRAFT_LMHEAD_16ROW=1 / 0: up to 16 rows, the 16-row kernel / the wide one
            // wherever it fits, instead of the choice by vocabulary size (for comparison)
            const char* l16 = getenv("FE_DRAFT_LMHEAD_16ROW");
            h->lm_16row = l16 && l16[0] == '1' ? 1 : (l16 && l16[0] == '0' ? 0 : -1);
        }
        if (h->lm_mma) {
            void* dst = p;
            p += align256(mma_packed_bytes(c.vocab, dm));
            if ((_fe_e = cudaMemcpyAsync(staging, w->lm_head, (size_t)c.vocab * dm * es, cudaMemcpyDefault, st)) !=
                    cudaSuccess ||
                (_fe_e = launch_pack_mma(staging, dst, c.vocab, dm, st)) != cudaSuccess)
                rc = fail(_fe_e, "copy or packing of the LM head", __LINE__);
            h->lm_head = dst;
        } else {
            void* dst = p;
            p += align256(packed_bytes(c.vocab, dm, es));
            if ((_fe_e = cudaMemcpyAsync(staging, w->lm_head, (size_t)c.vocab * dm * es, cudaMemcpyDefault, st)) !=
                    cudaSuccess ||
                (_fe_e = launch_pack_tiles(staging, dst, c.vocab, dm, es, st)) != cudaSuccess)
                rc = fail(_fe_e, "copy or packing of the LM head", __LINE__);
            h->lm_head = dst;
        }
        h->final_norm = put(w->final_norm, sz.norm);
        h->layers.resize(c.n_layers);
        for (int i = 0; i < c.n_layers && rc == FE_OK; ++i) {
            const fe_layer_weights& L = w->layers[i];
            LayerPacked& P = h->layers[i];
            P.attn_norm = put(L.attn_norm, sz.norm);
            P.mlp_norm = put(L.mlp_norm, sz.norm);
            P.w_qkv = put_packed(L.w_qkv, nq, dm);
            P.w_o = put_packed(L.w_o, dm, hq);
            // [gate; up] interleaved by row (row 2j = gate_j, row 2j+1 = up_j), then packed
            void* gu = p;
            p += align256(sz.gu);
            const size_t rowb = (size_t)dm * h->es;
            if (cudaMemcpy2DAsync(staging, 2 * rowb, L.w_gate, rowb, rowb, c.ffn, cudaMemcpyDefault, st) !=
                    cudaSuccess ||
                cudaMemcpy2DAsync((char*)staging + rowb, 2 * rowb, L.w_up, rowb, rowb, c.ffn, cudaMemcpyDefault,
                                  st) != cudaSuccess ||
                pack(staging, gu, 2 * c.ffn, dm) != cudaSuccess)
                rc = fail(cudaGetLastError(), "interleave or packing of gate/up", __LINE__);
            P.w_gu = gu;
            P.w_down = put_packed(L.w_down, dm, c.ffn);
        }
        cudaStreamSynchronize(st);
        cudaFree(staging);
        if (rc != FE_OK) break;

        // ---- RoPE table (cos, sin) per position and pair, computed in double ----
        const int half = c.head_dim / 2;
        std::vector<float> cs((size_t)c.max_seq * half * 2);
        for (int pos = 0; pos < c.max_seq; ++pos)
            for (int i = 0; i < half; ++i) {
                const double ang = (double)pos * pow((double)c.rope_theta, -2.0 * i / (double)c.head_dim);
                cs[((size_t)pos * half + i) * 2] = (float)cos(ang);
                cs[((size_t)pos * half + i) * 2 + 1] = (float)sin(ang);
            }

        // ---- scratch ----
        const size_t B = c.max_batch, d = c.d, F = c.ffn, H = c.n_heads, hd = c.head_dim;
        // rows of the per-row work buffers: a draft's B, or a commit block's up to 32
        const size_t Rw = std::max<size_t>(B, std::min<size_t>(32, B * (size_t)std::max(1, c.n_layers)));
        const int Rmma = (int)std::min<size_t>(32, Rw);
        const size_t nqkv = (size_t)(c.n_heads + 2 * c.n_kv_heads) * hd;
        h->attn_split_rows = attn_split(c.max_batch, c.n_kv_heads, c.max_seq, h->dev);
        h->attn_nsplit = (c.max_seq + h->attn_split_rows - 1) / h->attn_split_rows;
        h->lm_slabs = lmhead_slabs(c.vocab, h->dev);
        const size_t R = (size_t)c.n_layers * B;
        const size_t k = c.top_k_max;
        const size_t kmax = std::max({(size_t)3 * c.d, (size_t)c.ffn, (size_t)c.n_heads * hd});
        const size_t mmax = std::max({(size_t)c.d, nqkv, (size_t)2 * c.ffn});
        size_t off[26], n = 0, tot = 0;
        const size_t bytes[26] = {
            cs.size() * sizeof(float),                             // rope
            Rw * d * 4, Rw * d * 4, Rw * nqkv * 4, Rw * H * hd * 4,   // g, x, qkv, o
            Rw * F * 4, R * d * 4,                                  // act, hid
            B * H * h->attn_nsplit * (hd + 4) * 4,                 // attention partials (rows of hd + 4)
            R * h->lm_slabs * k * 4, R * h->lm_slabs * k * 4,      // LM-head partial ids, values
            R * h->lm_slabs * 2 * 4,                               // LM-head partial (max, sum)
            256,                                                   // status
            B * c.n_kv_heads * 4,                                  // attention split counters
            R * 4,                                                 // LM-head slab counters
            h->lm_mma ? std::max(lmhead_mma_zb_bytes((int)std::min<size_t>(R, 16), c.d),
                                 lmhead_wide_zb_bytes((int)R, c.d)) : 0,  // tensor-core LM-head operand
            h->lin_mma ? linear_mma_xb_bytes((int)kmax, std::max(c.max_batch, Rmma)) : 0,  // tensor-core linear operand
            h->lin_mma ? linear_mma_part_bytes(std::max(c.max_batch, Rmma), h->dev) : 0,   // its split-tile partials
            h->lin_mma ? linear_mma_counter_bytes((int)mmax, h->dev) : 0,   // its counters and fused-prep sums
            h->use_stack ? (size_t)(c.n_layers + 1) * sizeof(uint32_t) : 0,  // stack barrier counters
            Rw * d * 4,                                                       // x0
            Rw * 3 * d * h->es,                                               // commit: gathered features
            Rw * sizeof(int),                                                 // commit: gathered tokens
            h->lm_mma ? lmhead_mma_split_bytes(16, h->dev) : 0,                // LM head: split-tile parts
            h->lm_mma ? (size_t)h->dev.num_sms * sizeof(int) : 0,             // ... and their flags
            R * h->lm_slabs * k * 4,                                          // LM-head partial logits (sampling)
            B * (size_t)c.vocab * 4};                                         // sampled verification's residuals
        for (n = 0; n < 26; ++n) { off[n] = tot; tot += align256(bytes[n]); }
        if ((rc = from_cuda(cudaMalloc(&h->sbuf, tot))) != FE_OK) break;
        char* s = (char*)h->sbuf;
        h->rope_cs = (float*)(s + off[0]);
        h->g = (float*)(s + off[1]);
        h->x = (float*)(s + off[2]);
        h->qkv = (float*)(s + off[3]);
        h->o = (float*)(s + off[4]);
        h->act = (float*)(s + off[5]);
        h->hid = (float*)(s + off[6]);
        h->attn_part = (float*)(s + off[7]);
        h->lm_part_id = (int*)(s + off[8]);
        h->lm_part_val = (float*)(s + off[9]);
        h->lm_part_ms = (float*)(s + off[10]);
        h->status = (int*)(s + off[11]);
        h->attn_counters = (int*)(s + off[12]);
        h->lm_counters = (int*)(s + off[13]);
        h->lm_zb = h->lm_mma ? (uint16_t*)(s + off[14]) : nullptr;
        h->lin_xb = h->lin_mma ? (uint16_t*)(s + off[15]) : nullptr;
        h->lin_part = h->lin_mma ? (float*)(s + off[16]) : nullptr;
        h->lin_counters = h->lin_mma ? (int*)(s + off[17]) : nullptr;
        h->stack_bar = h->use_stack ? (uint32_t*)(s + off[18]) : nullptr;
        h->x0 = (float*)(s + off[19]);
        h->cfeat = s + off[20];
        h->ctok = (int*)(s + off[21]);
        h->lm_split_part = h->lm_mma ? (float*)(s + off[22]) : nullptr;
        h->lm_split_flag = h->lm_mma ? (int*)(s + off[23]) : nullptr;
        h->lm_part_lg = (float*)(s + off[24]);
        h->vs_rbuf = (float*)(s + off[25]);
        if ((rc = from_cuda(cudaMemcpyAsync(h->rope_cs, cs.data(), bytes[0], cudaMemcpyHostToDevice, st))) != FE_OK)
            break;
        // status word and completion counters start (and stay, between calls) at zero
        if ((rc = from_cuda(cudaMemsetAsync(h->status, 0, off[13] + bytes[13] - off[11], st))) != FE_OK) break;
        if (h->lin_mma && (rc = from_cuda(cudaMemsetAsync(h->lin_counters, 0, bytes[17], st))) != FE_OK) break;
        if (h->lm_mma && (rc = from_cuda(cudaMemsetAsync(h->lm_split_flag, 0, bytes[23], st))) != FE_OK) break;
        if ((rc = from_cuda(cudaStreamCreateWithFlags(&h->cap, cudaStreamNonBlocking))) != FE_OK) break;
        {  // fe_draft_step_host's staging (pinned) and device buffers
            const StepLayout L = step_layout(c, h->es, c.max_batch, c.top_k_max);
            if ((rc = from_cuda(cudaMallocHost((void**)&h->hs_in, L.in_bytes))) != FE_OK) break;
            if ((rc = from_cuda(cudaMallocHost((void**)&h->hs_out, L.out_bytes))) != FE_OK) break;
            if ((rc = from_cuda(cudaMalloc((void**)&h->ds_in, L.in_bytes))) != FE_OK) break;
            if ((rc = from_cuda(cudaMalloc((void**)&h->ds_out, L.out_bytes))) != FE_OK) break;
        }
        if ((rc = from_cuda(cudaStreamSynchronize(st))) != FE_OK) break;
    } while (0);
    if (rc != FE_OK) {
        cudaStreamSynchronize(st);
        release(h);
        return rc;
    }
    *out = h;
    return FE_OK;
}

fe_status fe_draft_forward(fe_handle* h, const fe_forward_args* a, void* stream) {
    if (!forward_args_ok(h, a)) return FE_ERR_INVALID_ARG;
    const fe_status dv = check_device(h);
    if (dv != FE_OK) return dv;
    const fe_config& c = h->cfg;
    cudaStream_t st = (cudaStream_t)stream;
    try {
        if (!h->use_graph) return enqueue_forward(h, a, st);
        GraphKey key;
        key.args = *a;
        key.args.k_cache = nullptr;
        key.args.v_cache = nullptr;
        key.kc.assign(a->k_cache, a->k_cache + c.n_layers);
        key.vc.assign(a->v_cache, a->v_cache + c.n_layers);
        if (!h->gexec || !(key == h->gkey)) {
            cudaGraph_t graph = nullptr;
            FE_TRY(cudaStreamBeginCapture(h->cap, cudaStreamCaptureModeThreadLocal));
            fe_status rc = enqueue_forward(h, a, h->cap);
            cudaError_t e = cudaStreamEndCapture(h->cap, &graph);
            if (rc != FE_OK) {
                if (graph) cudaGraphDestroy(graph);
                return rc;
            }
            FE_TRY(e);
            cudaGraphExec_t ex = nullptr;
            e = cudaGraphInstantiate(&ex, graph, 0);
            cudaGraphDestroy(graph);
            FE_TRY(e);
            if (h->gexec) cudaGraphExecDestroy(h->gexec);
            h->gexec = ex;
            h->gkey = key;
        }
        FE_TRY(cudaGraphLaunch(h->gexec, st));
        return FE_OK;
    } catch (...) {
        return FE_ERR_OOM;
    }
}

fe_status fe_profile_forward(fe_handle* h, const fe_forward_args* a, void* stream, int32_t cap, int32_t* kinds,
                             float* usec, int32_t* n_launches) {
    if (!forward_args_ok(h, a) || !kinds || !usec || !n_launches || cap < 1 || cap > 4096) return FE_ERR_INVALID_ARG;
    if (cap < fe_launch_count(h, a->B, 0) + (a->dbg_hidden ? 1 : 0)) return FE_ERR_INVALID_ARG;
    const fe_status dv = check_device(h);
    if (dv != FE_OK) return dv;
    cudaStream_t st = (cudaStream_t)stream;
    try {
        while ((int)h->prof_ev.size() < cap + 1) {
            cudaEvent_t e = nullptr;
            FE_TRY(cudaEventCreate(&e));
            h->prof_ev.push_back(e);
        }
        Prof pf{h->prof_ev.data(), nullptr, kinds, cap, 0};
        const fe_status rc = enqueue_forward(h, a, st, &pf);
        if (rc != FE_OK) {
            cudaStreamSynchronize(st);
            return rc;
        }
        FE_TRY(cudaEventSynchronize(pf.ev[pf.n]));
        for (int j = 0; j < pf.n; ++j) {
            float ms = 0.f;
            FE_TRY(cudaEventElapsedTime(&ms, pf.ev[j], pf.ev[j + 1]));
            usec[j] = 1000.f * ms;
        }
        *n_launches = pf.n;
        return FE_OK;
    } catch (...) {
        return FE_ERR_OOM;
    }
}

fe_status fe_profile_graph(fe_handle* h, const fe_forward_args* a, const fe_tree* tree, void* stream, int32_t cap,
                           int32_t* kinds, double* start_us, double* end_us, int32_t* n_launches) {
    if (!forward_args_ok(h, a) || !kinds || !start_us || !end_us || !n_launches || cap < 1 || cap > 4096)
        return FE_ERR_INVALID_ARG;
    if (tree && (!tree->tok || !tree->parent || !tree->depth || !tree->mask)) return FE_ERR_INVALID_ARG;
    const int need = fe_launch_count(h, a->B, tree ? 1 : 0) + (a->dbg_hidden ? 1 : 0);
    if (cap < need) return FE_ERR_INVALID_ARG;
    const fe_status dv = check_device(h);
    if (dv != FE_OK) return dv;
    const fe_config& c = h->cfg;
    cudaStream_t st = (cudaStream_t)stream;
    try {
        if (h->prof_stamp_cap < need) {
            if (h->pexec) {
                cudaGraphExecDestroy(h->pexec);
                h->pexec = nullptr;
            }
            if (h->prof_stamps) cudaFree(h->prof_stamps);
            h->prof_stamps = nullptr;
            h->prof_stamp_cap = 0;
            FE_TRY(cudaMalloc(&h->prof_stamps, (size_t)2 * need * sizeof(unsigned long long)));
            h->prof_stamp_cap = need;
        }
        GraphKey key;
        key.args = *a;
        key.args.k_cache = nullptr;
        key.args.v_cache = nullptr;
        key.kc.assign(a->k_cache, a->k_cache + c.n_layers);
        key.vc.assign(a->v_cache, a->v_cache + c.n_layers);
        const fe_tree tk = tree ? *tree : fe_tree{};
        const bool same_tree = tk.tok == h->ptree.tok && tk.parent == h->ptree.parent && tk.depth == h->ptree.depth &&
                               tk.mask == h->ptree.mask;
        if (!h->pexec || !(key == h->pkey) || !same_tree) {
            // the same launch sequence as fe_draft_forward's graph (programmatic launches
            // included), each kernel given its stamp pair; the pairs are cleared first
            h->pkinds.assign(need, -1);
            Prof pf{nullptr, h->prof_stamps, h->pkinds.data(), need, 0};
            cudaGraph_t graph = nullptr;
            FE_TRY(cudaStreamBeginCapture(h->cap, cudaStreamCaptureModeThreadLocal));
            fe_status rc = FE_OK;
            cudaError_t e = cudaMemsetAsync(h->prof_stamps, 0, (size_t)2 * need * sizeof(unsigned long long), h->cap);
            if (e != cudaSuccess) rc = fail(e, "stamp clear", __LINE__);
            if (rc == FE_OK) rc = enqueue_forward(h, a, h->cap, &pf);
            if (rc == FE_OK && tree) {
                unsigned long long* sp = next_stamp(&pf);
                e = launch_tree(a->B, c.n_layers, a->top_k, c.vocab, a->next_tok, a->topk_id, tk.tok, tk.parent,
                                tk.depth, tk.mask, h->status, h->cap, sp);
                if (e == cudaSuccess) e = mark(&pf, FE_KERNEL_TREE, h->cap);
                if (e != cudaSuccess) rc = fail(e, "tree launch", __LINE__);
            }
            e = cudaStreamEndCapture(h->cap, &graph);
            if (rc != FE_OK) {
                if (graph) cudaGraphDestroy(graph);
                return rc;
            }
            FE_TRY(e);
            cudaGraphExec_t ex = nullptr;
            e = cudaGraphInstantiate(&ex, graph, 0);
            cudaGraphDestroy(graph);
            FE_TRY(e);
            if (h->pexec) cudaGraphExecDestroy(h->pexec);
            h->pexec = ex;
            h->pkey = key;
            h->ptree = tk;
            h->pkinds.resize(pf.n);
        }
        FE_TRY(cudaGraphLaunch(h->pexec, st));
        const int n = (int)h->pkinds.size();
        std::vector<unsigned long long> raw((size_t)2 * n);
        FE_TRY(cudaMemcpyAsync(raw.data(), h->prof_stamps, raw.size() * sizeof(unsigned long long),
                               cudaMemcpyDeviceToHost, st));
        FE_TRY(cudaStreamSynchronize(st));
        unsigned long long t0 = ~0ull;
        for (int j = 0; j < n; ++j)
            if (raw[2 * j]) t0 = std::min(t0, ~raw[2 * j]);
        for (int j = 0; j < n; ++j) {
            kinds[j] = h->pkinds[j];
            const bool ok = raw[2 * j] != 0 && raw[2 * j + 1] != 0;
            start_us[j] = ok ? (double)(~raw[2 * j] - t0) * 1e-3 : -1.0;
            end_us[j] = ok ? (double)(raw[2 * j + 1] - t0) * 1e-3 : -1.0;
        }
        *n_launches = n;
        return FE_OK;
    } catch (...) {
        return FE_ERR_OOM;
    }
}

namespace {

// the device work of one fe_draft_step_host call: inputs in, draft, tree, outputs out
// (feat_direct: the caller's features are page-locked and copied from where they are; the
// staging then holds only the tokens and prefix lengths)
fe_status enqueue_host_step(fe_handle* h, const fe_host_step_args* a, const StepLayout& L, bool feat_direct,
                            cudaStream_t st) {
    const fe_config& c = h->cfg;
    if (feat_direct) {
        FE_TRY(cudaMemcpyAsync(h->ds_in + L.feat, a->feat, (size_t)a->B * 3 * c.d * h->es, cudaMemcpyHostToDevice, st));
        FE_TRY(cudaMemcpyAsync(h->ds_in + L.tok, h->hs_in + L.tok, L.in_bytes - L.tok, cudaMemcpyHostToDevice, st));
    } else {
        FE_TRY(cudaMemcpyAsync(h->ds_in, h->hs_in, L.in_bytes, cudaMemcpyHostToDevice, st));
    }
    fe_forward_args fa{};
    fa.B = a->B; fa.top_k = a->top_k; fa.temperature = a->temperature;
    fa.feat = h->ds_in + L.feat;
    fa.next_tok = reinterpret_cast<const int32_t*>(h->ds_in + L.tok);
    fa.prefix_len = reinterpret_cast<const int32_t*>(h->ds_in + L.plen);
    fa.k_cache = a->k_cache; fa.v_cache = a->v_cache; fa.page_table = a->page_table; fa.n_pages = a->n_pages;
    fa.topk_id = reinterpret_cast<int32_t*>(h->ds_out + L.id);
    fa.topk_logit = reinterpret_cast<float*>(h->ds_out + L.logit);
    fa.topk_prob = reinterpret_cast<float*>(h->ds_out + L.prob);
    fa.lse = reinterpret_cast<float*>(h->ds_out + L.lse);
    fa.sample = a->sample;
    fa.seed = a->seed;
    fa.topk_rank = reinterpret_cast<int32_t*>(h->ds_out + L.rank);
    if (!forward_args_ok(h, &fa)) return FE_ERR_INVALID_ARG;
    const fe_status rc = enqueue_forward(h, &fa, st);
    if (rc != FE_OK) return rc;
    FE_TRY(launch_tree(a->B, c.n_layers, a->top_k, c.vocab, fa.next_tok, fa.topk_id,
                       reinterpret_cast<int32_t*>(h->ds_out + L.ttok), reinterpret_cast<int32_t*>(h->ds_out + L.tpar),
                       reinterpret_cast<int32_t*>(h->ds_out + L.tdep), h->ds_out + L.tmask, h->status, st));
    FE_TRY(cudaMemcpyAsync(h->hs_out, h->ds_out, L.out_bytes, cudaMemcpyDeviceToHost, st));
    return FE_OK;
}

}  // namespace

fe_status fe_draft_step_host(fe_handle* h, const fe_host_step_args* a, void* stream) {
    if (!h || !a) return FE_ERR_INVALID_ARG;
    const fe_config& c = h->cfg;
    if (a->B < 1 || a->B > c.max_batch || a->top_k < 1 || a->top_k > c.top_k_max) return FE_ERR_INVALID_ARG;
    if (!a->feat || !a->next_tok || !a->prefix_len || !a->k_cache || !a->v_cache || !a->topk_id || !a->topk_logit ||
        !a->topk_prob || !a->lse || !a->tree_tok || !a->tree_parent || !a->tree_depth || !a->tree_mask)
        return FE_ERR_INVALID_ARG;
    for (int i = 0; i < c.n_layers; ++i)
        if (!a->k_cache[i] || !a->v_cache[i]) return FE_ERR_INVALID_ARG;
    if (c.page_size > 0 && (!a->page_table || a->n_pages < 1)) return FE_ERR_INVALID_ARG;
    if (!(a->temperature == a->temperature)) return FE_ERR_INVALID_ARG;
    if (a->sample && !(a->temperature > 0.f)) return FE_ERR_INVALID_ARG;
    const fe_status dv = check_device(h);
    if (dv != FE_OK) return dv;
    cudaStream_t st = (cudaStream_t)stream;
    const StepLayout L = step_layout(c, h->es, a->B, a->top_k);
    const size_t B = (size_t)a->B, N = (size_t)c.n_layers, k = (size_t)a->top_k, T = 1 + N * k;
    // page-locked features (e.g. the caller's own pinned buffer) need no staging copy
    cudaPointerAttributes pa{};
    const bool feat_direct = cudaPointerGetAttributes(&pa, a->feat) == cudaSuccess && pa.type == cudaMemoryTypeHost &&
                             (reinterpret_cast<uintptr_t>(a->feat) & 15) == 0;
    cudaGetLastError();  // (an unregistered pointer may leave an error behind on older runtimes)
    // (the previous call synchronised its stream: the staging buffers are free)
    if (!feat_direct) memcpy(h->hs_in + L.feat, a->feat, B * 3 * (size_t)c.d * h->es);
    memcpy(h->hs_in + L.tok, a->next_tok, B * 4);
    memcpy(h->hs_in + L.plen, a->prefix_len, B * 4);
    try {
        if (!h->use_graph) {
            const fe_status rc = enqueue_host_step(h, a, L, feat_direct, st);
            if (rc != FE_OK) return rc;
        } else {
            HostKey key;
            key.B = a->B; key.top_k = a->top_k; key.temperature = a->temperature;
            key.sample = a->sample ? 1 : 0; key.seed = a->seed;
            key.feat_direct = feat_direct ? a->feat : nullptr;
            key.page_table = a->page_table; key.n_pages = a->n_pages;
            key.kc.assign(a->k_cache, a->k_cache + c.n_layers);
            key.vc.assign(a->v_cache, a->v_cache + c.n_layers);
            if (!h->hexec || !(key == h->hkey)) {
                cudaGraph_t graph = nullptr;
                FE_TRY(cudaStreamBeginCapture(h->cap, cudaStreamCaptureModeThreadLocal));
                const fe_status rc = enqueue_host_step(h, a, L, feat_direct, h->cap);
                cudaError_t e = cudaStreamEndCapture(h->cap, &graph);
                if (rc != FE_OK) {
                    if (graph) cudaGraphDestroy(graph);
                    return rc;
                }
                FE_TRY(e);
                cudaGraphExec_t ex = nullptr;
                e = cudaGraphInstantiate(&ex, graph, 0);
                cudaGraphDestroy(graph);
                FE_TRY(e);
                if (h->hexec) cudaGraphExecDestroy(h->hexec);
                h->hexec = ex;
                h->hkey = key;
            }
            FE_TRY(cudaGraphLaunch(h->hexec, st));
        }
        FE_TRY(cudaStreamSynchronize(st));
    } catch (...) {
        return FE_ERR_OOM;
    }
    memcpy(a->topk_id, h->hs_out + L.id, B * N * k * 4);
    memcpy(a->topk_logit, h->hs_out + L.logit, B * N * k * 4);
    memcpy(a->topk_prob, h->hs_out + L.prob, B * N * k * 4);
    memcpy(a->lse, h->hs_out + L.lse, B * N * 4);
    if (a->topk_rank) memcpy(a->topk_rank, h->hs_out + L.rank, B * N * k * 4);
    memcpy(a->tree_tok, h->hs_out + L.ttok, B * T * 4);
    memcpy(a->tree_parent, h->hs_out + L.tpar, B * T * 4);
    memcpy(a->tree_depth, h->hs_out + L.tdep, B * T * 4);
    memcpy(a->tree_mask, h->hs_out + L.tmask, B * T * T);
    return FE_OK;
}

fe_status fe_build_tree(fe_handle* h, int32_t B, int32_t top_k, const int32_t* next_tok, const int32_t* topk_id,
                        fe_tree* out, void* stream) {
    if (!h || !out || !next_tok || !topk_id) return FE_ERR_INVALID_ARG;
    if (!out->tok || !out->parent || !out->depth || !out->mask) return FE_ERR_INVALID_ARG;
    if (B < 1 || B > h->cfg.max_batch || top_k < 1 || top_k > h->cfg.top_k_max) return FE_ERR_INVALID_ARG;
    const fe_status dv = check_device(h);
    if (dv != FE_OK) return dv;
    FE_TRY(launch_tree(B, h->cfg.n_layers, top_k, h->cfg.vocab, next_tok, topk_id, out->tok, out->parent, out->depth,
                       out->mask, h->status, (cudaStream_t)stream));
    return FE_OK;
}

fe_status fe_draft_loss(fe_handle* h, const fe_forward_args* a, const float* teacher_p, const float* target_feat,
                        float alpha, float beta, float decay, float* ce, float* feat_loss, float* total, void* stream) {
    if (!forward_args_ok(h, a) || !a->dbg_logits || !a->dbg_hidden || !teacher_p || !target_feat || !ce ||
        !feat_loss || !total)
        return FE_ERR_INVALID_ARG;
    if (!(alpha == alpha) || !(beta == beta) || !(decay == decay)) return FE_ERR_INVALID_ARG;
    const fe_status rc = fe_draft_forward(h, a, stream);  // (checks the device)
    if (rc != FE_OK) return rc;
    const fe_config& c = h->cfg;
    FE_TRY(launch_loss(c.n_layers, a->B, c.vocab, c.d, a->dbg_logits, teacher_p, a->dbg_hidden, target_feat, alpha,
                       beta, decay, ce, feat_loss, total, (cudaStream_t)stream));
    return FE_OK;
}

fe_status fe_verify_greedy(fe_handle* h, int32_t B, int32_t top_k, const int32_t* prefix_len, const fe_tree* tree,
                           const int32_t* target_next, int32_t* pos_ids, int32_t* path, int32_t* n_accept,
                           int32_t* bonus, void* stream) {
    if (!h || !tree || !prefix_len || !target_next || !pos_ids || !path || !n_accept || !bonus) return FE_ERR_INVALID_ARG;
    if (!tree->tok || !tree->parent || !tree->depth) return FE_ERR_INVALID_ARG;
    if (B < 1 || B > h->cfg.max_batch || top_k < 1 || top_k > h->cfg.top_k_max) return FE_ERR_INVALID_ARG;
    const fe_status dv = check_device(h);
    if (dv != FE_OK) return dv;
    const int N = h->cfg.n_layers, T = 1 + N * top_k;
    FE_TRY(launch_verify(B, T, N, prefix_len, tree->tok, tree->parent, tree->depth, target_next, pos_ids, path,
                         n_accept, bonus, (cudaStream_t)stream));
    return FE_OK;
}

fe_status fe_verify_sampled(fe_handle* h, int32_t B, int32_t top_k, const fe_tree* tree, const int32_t* topk_rank,
                            const float* q, const float* p, const float* u_acc, const float* u_bonus, int32_t* path,
                            int32_t* n_accept, int32_t* bonus, void* stream) {
    if (!h || !tree || !topk_rank || !q || !p || !u_acc || !u_bonus || !path || !n_accept || !bonus)
        return FE_ERR_INVALID_ARG;
    if (!tree->tok || !tree->parent || !tree->depth) return FE_ERR_INVALID_ARG;
    if (B < 1 || B > h->cfg.max_batch || top_k < 1 || top_k > h->cfg.top_k_max) return FE_ERR_INVALID_ARG;
    const fe_status dv = check_device(h);
    if (dv != FE_OK) return dv;
    VerifySampledArgs va{};
    va.N = h->cfg.n_layers;
    va.T = 1 + va.N * top_k;
    va.V = h->cfg.vocab;
    va.tok = tree->tok; va.parent = tree->parent; va.depth = tree->depth; va.rank = topk_rank;
    va.q = q; va.p = p; va.u_acc = u_acc; va.u_bonus = u_bonus;
    va.rbuf = h->vs_rbuf;
    va.path = path; va.n_accept = n_accept; va.bonus = bonus; va.status = h->status;
    FE_TRY(launch_verify_sampled(va, B, (cudaStream_t)stream));
    return FE_OK;
}

fe_status fe_commit(fe_handle* h, const fe_commit_args* a, void* stream) {
    if (!h || !a) return FE_ERR_INVALID_ARG;
    const fe_config& c = h->cfg;
    if (a->B < 1 || a->B > c.max_batch || a->L < 1 || a->L > c.n_layers) return FE_ERR_INVALID_ARG;
    if (!a->feat || !a->tok || !a->n_rows || !a->prefix_len || !a->k_cache || !a->v_cache) return FE_ERR_INVALID_ARG;
    for (int i = 0; i < c.n_layers; ++i)
        if (!a->k_cache[i] || !a->v_cache[i]) return FE_ERR_INVALID_ARG;
    if (c.page_size > 0 && (!a->page_table || a->n_pages < 1)) return FE_ERR_INVALID_ARG;
    if (reinterpret_cast<uintptr_t>(a->feat) & 15) return FE_ERR_INVALID_ARG;  // copied as 16-byte vectors
    const fe_status dv = check_device(h);
    if (dv != FE_OK) return dv;
    try {
        return enqueue_commit(h, a, (cudaStream_t)stream);
    } catch (...) {
        return FE_ERR_OOM;
    }
}

fe_status fe_last_device_status(fe_handle* h, void* stream) {
    if (!h) return FE_ERR_INVALID_ARG;
    const fe_status dv = check_device(h);
    if (dv != FE_OK) return dv;
    cudaStream_t st = (cudaStream_t)stream;
    int v = 0;
    FE_TRY(cudaStreamSynchronize(st));
    FE_TRY(cudaMemcpy(&v, h->status, sizeof(int), cudaMemcpyDeviceToHost));
    FE_TRY(cudaMemset(h->status, 0, sizeof(int)));
    if (v & ST_TIMEOUT) return FE_ERR_TIMEOUT;
    if (v & ST_CAPACITY) return FE_ERR_CAPACITY;
    if (v & ST_DEVICE) return FE_ERR_DEVICE;
    return FE_OK;
}

void fe_free(fe_handle* h) {
    if (!h) return;
    // release on the handle's device, whichever device the caller has current
    int cur = -1;
    const bool have_cur = cudaGetDevice(&cur) == cudaSuccess;
    if (have_cur && cur != h->device) cudaSetDevice(h->device);
    cudaDeviceSynchronize();
    const int dev = h->device;
    release(h);
    if (have_cur && cur != dev) cudaSetDevice(cur);
}

const char* fe_last_error_detail(void) { return g_detail; }

int32_t fe_launch_count(const fe_handle* h, int32_t B, int32_t with_tree) {
    if (!h || B < 1) return -1;
    const int N = h->cfg.n_layers;
    const int lin = h->lin_mma ? 2 : linear_launches();
    // stacked: N + 1 stack launches hold all linear phases
    // (on batched handles the O projection's operand comes from the attention kernel: no prep)
    const int lin_total = (h->use_stack && B == 1) ? N + 1 : 2 * lin + N * 4 * lin - (h->lin_mma && h->attn_operand ? N : 0);
    int n = lin_total + N * attention_launches() +
            (h->lm_mma ? 3 : lmhead_launches(N * B, h->cfg.d, h->dev));
    return n + (with_tree ? 1 : 0);
}

fe_status fe_selftest_timeout(fe_handle* h, int64_t timeout_ns, void* stream) {
    if (!h || timeout_ns < 1000 || timeout_ns > 1000000000LL) return FE_ERR_INVALID_ARG;
    const fe_status dv = check_device(h);
    if (dv != FE_OK) return dv;
    FE_TRY(launch_timeout_probe(timeout_ns, h->status, (cudaStream_t)stream));
    return FE_OK;
}

}  // extern "C"

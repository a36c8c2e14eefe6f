/*
 * oracle.c -- plain, slow, fp64 CPU oracle of the FastEagle cascaded drafter.
 *
 * TEST INFRASTRUCTURE. Only the tests, __graft_entry__.smoke() and the CPU-baseline
 * leg of bench.py may load or run this library. It shares no code, header, table or
 * helper with the CUDA path (paper_2509_20416_gb300/), and it never reads a value the
 * CUDA path produced: it is the yardstick the CUDA path is measured against.
 *
 * What it computes (FastEagle, arXiv 2509.20416):
 *   - Sec. 2.1 and Eq. 1: fused feature g = FC(concat(l, m, h)) from the target's
 *     three hidden-state levels, then x0 = FC(concat(g, e)) with e the embedding of
 *     the next token; both FCs are bias-free linear maps.
 *   - Eq. 2: the cascade h_i = L_i(h_{i-1}), i = 1..N (h_0 = x0), each L_i a
 *     lightweight pre-norm decoder layer with its own parameters. Sec. 2.1 builds on
 *     EAGLE-3's single decoder layer; its internals are read as the standard LLaMA
 *     block: RMSNorm, QKV, rotate-half RoPE, (grouped-query) attention over the
 *     layer's own prefix K/V cache plus the drafted row's own key/value, O-proj and
 *     residual, RMSNorm, SwiGLU MLP and residual.
 *   - Sec. 2.1: every h_i goes through the target's frozen LM head (after the
 *     target's final RMSNorm) to give the distribution q_{t+i}.
 *   - Sec. 2.2: top-k per depth and the Backbone Expansion tree with its
 *     tree-attention (ancestor-or-self) mask; for stochastic drafting, k candidates
 *     drawn without replacement from q_{t+i} (Gumbel-top-k over counter-based deviates).
 * Every stored bf16/fp32 input is widened exactly to double; nothing is rounded in
 * between. Loops are the definitions written out: no blocking, no fusion, no
 * reordering of a sum. OpenMP only splits independent output rows across threads,
 * so results do not depend on the thread count.
 *
 * Parity pins: every function here is pinned by the `-m "not gpu"` tests (closed
 * forms, brute force, library special cases, invariants, a hand-worked tree). The
 * OR_MUTANT switch plants one known mistake per build so that a test can show the
 * pins catch it; the default build (OR_MUTANT == 0) has none.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifndef OR_MUTANT
#define OR_MUTANT 0
#endif
#define MUT(n) (OR_MUTANT == (n))

typedef struct {
    int32_t d, n_heads, n_kv_heads, head_dim, ffn, vocab, n_layers;
    int32_t dtype;             /* storage type of every input tensor: 0 float32, 1 bfloat16 */
    double rope_theta, rms_eps;
    int32_t rope_layer_offset; /* reading of the query position: 0 -> every layer at P (default),
                                  1 -> layer i at P + i - 1 */
    int32_t final_norm;        /* 1 -> RMSNorm(gamma_out) before the LM head (default), 0 -> none */
    int32_t parallel_layers;   /* 0 -> the cascade, L_i consumes h_{i-1} (Eq. 2, default);
                                  1 -> every L_i consumes x0: the "w/o cascaded structure"
                                  ablation of Sec. 3.2 (Table 2), parallel instead of serial */
} or_config;

/* ---- storage ------------------------------------------------------------------ */

static double ld(const void *p, int32_t dtype, int64_t i)
{
    if (dtype == 0)
        return (double)((const float *)p)[i];
    uint32_t u = (uint32_t)((const uint16_t *)p)[i] << 16; /* bf16 -> f32 is exact */
    float f;
    memcpy(&f, &u, 4);
    return (double)f;
}

/* Store v in the cache's storage type: float32 by C's double -> float conversion (round to
 * nearest), bfloat16 by rounding the double to the nearest bfloat16 (ties to even). The
 * cache holds stored values: a later row reads the rounded one. */
static void st(void *p, int32_t dtype, int64_t i, double v)
{
    if (dtype == 0) {
        ((float *)p)[i] = (float)v;
        return;
    }
    if (isnan(v)) {
        ((uint16_t *)p)[i] = 0x7FC0;
        return;
    }
    /* the two bfloat16 neighbours of v (bfloat16 values are exact floats, so compare in
       double): truncate the float nearest below |v|, then pick the closer, ties to even */
    const double a = fabs(v);
    float f = (float)a;
    if ((double)f > a)
        f = nextafterf(f, 0.0f);
    uint32_t u;
    memcpy(&u, &f, 4);
    uint32_t lo = u & 0xFFFF0000u, hi = lo + 0x10000u;
    float flo, fhi;
    memcpy(&flo, &lo, 4);
    memcpy(&fhi, &hi, 4);
    const double dlo = a - (double)flo, dhi = (double)fhi - a;
    uint32_t r = (dlo < dhi || (dlo == dhi && !((lo >> 16) & 1u))) ? lo : hi;
    if (v < 0)
        r |= 0x80000000u;
    ((uint16_t *)p)[i] = (uint16_t)(r >> 16);
}

void or_widen(const void *src, int32_t dtype, int64_t n, double *dst)
{
    for (int64_t i = 0; i < n; ++i)
        dst[i] = ld(src, dtype, i);
}

/* ---- primitives ---------------------------------------------------------------- */

/* y = W x with W row-major [M, K]: y_m = sum_k W[m, k] x_k. */
void or_matvec(const void *W, int32_t dtype, int64_t M, int64_t K, const double *x, double *y)
{
#pragma omp parallel for schedule(static)
    for (int64_t m = 0; m < M; ++m) {
        double s = 0.0;
        for (int64_t k = 0; k < K; ++k) {
            int64_t idx = MUT(1) ? k * M + m : m * K + k;
            s += ld(W, dtype, idx) * x[k];
        }
        y[m] = s;
    }
}

/* RMSNorm: y_j = gamma_j * x_j / sqrt(mean(x^2) + eps). */
void or_rmsnorm(const double *x, const void *gamma, int32_t dtype, int64_t n, double eps, double *y)
{
    double ss = 0.0;
    for (int64_t j = 0; j < n; ++j)
        ss += x[j] * x[j];
    double ms = MUT(6) ? ss : ss / (double)n;
    double r = 1.0 / sqrt(MUT(24) ? ms : ms + eps);
    for (int64_t j = 0; j < n; ++j)
        y[j] = ld(gamma, dtype, j) * x[j] * r;
}

/* Rotary position embedding, rotate-half pairing (j, j + hd/2), j < hd/2, rotating
 * the pair by the angle pos * theta^(-2j/hd). Applied in place to one head. */
void or_rope(double *v, int32_t hd, double pos, double theta)
{
    const int32_t half = hd / 2;
    if (MUT(3)) { /* planted mistake: interleaved pairs (2j, 2j+1) */
        for (int32_t j = 0; j < half; ++j) {
            double ang = pos * pow(theta, -2.0 * (double)j / (double)hd);
            double c = cos(ang), s = sin(ang);
            double a = v[2 * j], b = v[2 * j + 1];
            v[2 * j] = a * c - b * s;
            v[2 * j + 1] = b * c + a * s;
        }
        return;
    }
    for (int32_t j = 0; j < half; ++j) {
        double ang = pos * pow(theta, -2.0 * (double)j / (double)hd);
        double c = cos(ang), s = sin(ang);
        double a = v[j], b = v[j + half];
        if (MUT(2)) {
            v[j] = a * c + b * s;
            v[j + half] = b * c - a * s;
        } else {
            v[j] = a * c - b * s;
            v[j + half] = b * c + a * s;
        }
    }
}

/* Decode attention of one drafted row of one sequence.
 *   q      [H][hd]     queries (RoPE already applied)
 *   kc, vc [Hkv][cap][hd] this layer's cache for this sequence (storage dtype); rows
 *          0..P-1 are the prefix (keys already rotated)
 *   k_new, v_new [Hkv][hd] the row's own key (rotated) and value, key index P
 *   out    [H][hd]
 * Query head h reads KV head g(h) = floor(h * Hkv / H); scores are scaled by
 * 1/sqrt(hd); the softmax subtracts the row maximum. */
void or_attention(const double *q, int32_t H, int32_t Hkv, int32_t hd, const void *kc,
                  const void *vc, int32_t dtype, int64_t cap, int32_t P, const double *k_new,
                  const double *v_new, double *out)
{
    const double scale = MUT(4) ? 1.0 : 1.0 / sqrt((double)hd);
    const int32_t P_read = MUT(22) ? (P > 0 ? P - 1 : 0) : P;
#pragma omp parallel for schedule(static)
    for (int32_t h = 0; h < H; ++h) {
        const int32_t g = MUT(5) ? h % Hkv : (int32_t)(((int64_t)h * Hkv) / H);
        const double *qh = q + (int64_t)h * hd;
        const int32_t nk = MUT(11) ? P_read : P_read + 1;
        double *s = (double *)malloc(sizeof(double) * (size_t)(nk > 0 ? nk : 1));
        double mx = -INFINITY;
        for (int32_t t = 0; t < nk; ++t) {
            double dot = 0.0;
            if (t < P_read) {
                int64_t base = ((int64_t)g * cap + t) * hd;
                for (int32_t j = 0; j < hd; ++j)
                    dot += qh[j] * ld(kc, dtype, base + j);
            } else {
                for (int32_t j = 0; j < hd; ++j)
                    dot += qh[j] * k_new[(int64_t)g * hd + j];
            }
            s[t] = dot * scale;
            if (s[t] > mx)
                mx = s[t];
        }
        double den = 0.0;
        for (int32_t t = 0; t < nk; ++t) {
            s[t] = exp(s[t] - mx);
            den += s[t];
        }
        for (int32_t j = 0; j < hd; ++j) {
            double acc = 0.0;
            for (int32_t t = 0; t < nk; ++t) {
                double vv = (t < P_read) ? ld(vc, dtype, ((int64_t)g * cap + t) * hd + j)
                                         : v_new[(int64_t)g * hd + j];
                acc += s[t] * vv;
            }
            out[(int64_t)h * hd + j] = acc / den;
        }
        free(s);
    }
}

/* SiLU(a) = a / (1 + e^-a); the SwiGLU product silu(gate) * up. */
void or_silu_mul(const double *gate, const double *up, int64_t n, double *y)
{
    for (int64_t j = 0; j < n; ++j) {
        double a = MUT(9) ? up[j] : gate[j];
        double b = MUT(9) ? gate[j] : up[j];
        double sig = 1.0 / (1.0 + exp(-a));
        y[j] = (MUT(23) ? sig : a * sig) * b;
    }
}

/* One cascade layer L_i (Eq. 2) for one sequence, x updated in place.
 * lw: attn_norm, w_qkv [(H+2Hkv)hd, d], w_o [d, H hd], mlp_norm, w_gate [F,d],
 * w_up [F,d], w_down [d,F]. The drafted row sits at sequence position `pos`; it
 * attends to its P prefix rows in (kc, vc) plus its own key/value. When k_out / v_out
 * are given they receive the row's own key (rotated) and value, [Hkv][hd]. */
void or_layer(const or_config *c, const void *const *lw, double pos, const void *kc,
              const void *vc, int64_t cap, int32_t P, double *x, double *k_out, double *v_out)
{
    const int32_t d = c->d, H = c->n_heads, Hkv = c->n_kv_heads, hd = c->head_dim, F = c->ffn;
    const int64_t nq = (int64_t)H * hd, nkv = (int64_t)Hkv * hd;
    double *u = (double *)malloc(sizeof(double) * (size_t)d);
    double *qkv = (double *)malloc(sizeof(double) * (size_t)(nq + 2 * nkv));
    double *o = (double *)malloc(sizeof(double) * (size_t)nq);
    double *t = (double *)malloc(sizeof(double) * (size_t)d);
    double *gt = (double *)malloc(sizeof(double) * (size_t)F);
    double *up = (double *)malloc(sizeof(double) * (size_t)F);
    double *a = (double *)malloc(sizeof(double) * (size_t)F);

    /* attention block */
    or_rmsnorm(x, lw[0], c->dtype, d, c->rms_eps, u);
    or_matvec(lw[1], c->dtype, nq + 2 * nkv, d, u, qkv);
    double *q = qkv, *k = qkv + nq, *v = qkv + nq + nkv;
    if (MUT(26)) { double *tmp = k; k = v; v = tmp; }
    for (int32_t h = 0; h < H; ++h)
        or_rope(q + (int64_t)h * hd, hd, pos, c->rope_theta);
    for (int32_t g = 0; g < Hkv; ++g) {
        or_rope(k + (int64_t)g * hd, hd, pos, c->rope_theta);
        if (MUT(27))
            or_rope(v + (int64_t)g * hd, hd, pos, c->rope_theta);
    }
    or_attention(q, H, Hkv, hd, kc, vc, c->dtype, cap, P, k, v, o);
    if (k_out)
        memcpy(k_out, k, sizeof(double) * (size_t)nkv);
    if (v_out)
        memcpy(v_out, v, sizeof(double) * (size_t)nkv);
    or_matvec(lw[2], c->dtype, d, nq, o, t);
    for (int32_t j = 0; j < d; ++j)
        x[j] = MUT(7) ? t[j] : x[j] + t[j];

    /* MLP block */
    or_rmsnorm(x, lw[3], c->dtype, d, c->rms_eps, u);
    or_matvec(lw[4], c->dtype, F, d, u, gt);
    or_matvec(lw[5], c->dtype, F, d, u, up);
    or_silu_mul(gt, up, F, a);
    or_matvec(lw[6], c->dtype, d, F, a, t);
    for (int32_t j = 0; j < d; ++j)
        x[j] = MUT(8) ? t[j] : x[j] + t[j];

    free(u); free(qkv); free(o); free(t); free(gt); free(up); free(a);
}

/* Sec. 2.1: logits of one hidden state through the (optional) final RMSNorm and the
 * frozen LM head W_lm [V, d]. */
void or_lm_head(const or_config *c, const void *lm_head, const void *final_norm,
                const double *h, double *logits)
{
    double *z = (double *)malloc(sizeof(double) * (size_t)c->d);
    if (c->final_norm && !MUT(17))
        or_rmsnorm(h, final_norm, c->dtype, c->d, c->rms_eps, z);
    else
        memcpy(z, h, sizeof(double) * (size_t)c->d);
    or_matvec(lm_head, c->dtype, c->vocab, c->d, z, logits);
    free(z);
}

/* Softmax of logits / T with its log-normaliser: lse = max + log sum exp(l/T - max),
 * p_v = exp(l_v/T - lse). T <= 0 (greedy decoding) uses T = 1: the distribution the
 * drafter proposes from. */
void or_softmax(const double *logits, int64_t V, double T, double *p, double *lse)
{
    const double tt = (T > 0.0 && !MUT(20)) ? T : 1.0;
    double mx = -INFINITY;
    for (int64_t v = 0; v < V; ++v)
        if (logits[v] / tt > mx)
            mx = logits[v] / tt;
    double s = 0.0;
    for (int64_t v = 0; v < V; ++v)
        s += exp(logits[v] / tt - mx);
    double l = MUT(21) ? log(s) : mx + log(s);
    if (lse)
        *lse = l;
    if (p)
        for (int64_t v = 0; v < V; ++v)
            p[v] = exp(logits[v] / tt - l);
}

/* The k most probable tokens, best first: the first k entries of a stable sort by
 * (descending logit, ascending id). Selection by repeated scan. */
void or_topk(const double *logits, int64_t V, int32_t k, int32_t *ids)
{
    unsigned char *taken = (unsigned char *)calloc((size_t)V, 1);
    for (int32_t r = 0; r < k; ++r) {
        int64_t best = -1;
        for (int64_t v = 0; v < V; ++v) {
            if (taken[v])
                continue;
            if (best < 0 || logits[v] > logits[best] ||
                (MUT(12) && logits[v] == logits[best]))
                best = v;
        }
        ids[r] = (int32_t)best;
        taken[best] = 1;
    }
    free(taken);
}

/* ---- stochastic drafting (Sec. 2.2 "sample k candidates"): read as k draws without
 * replacement from softmax(l / T), taken by the Gumbel-top-k trick over counter-based
 * deviates, so that both sides can draw the same numbers ------------------------------ */

/* SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom number generators",
 * OOPSLA 2014): the generator seeded with s returns, as its n-th output (n >= 1), the
 * finaliser below applied to s + n * 0x9E3779B97F4A7C15 (arithmetic mod 2^64). */
uint64_t or_splitmix64(uint64_t seed, uint64_t n)
{
    uint64_t z = seed + n * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

/* A uniform deviate in (0, 1) from the top 23 bits of output n: (floor(x / 2^41) + 1/2)
 * / 2^23. Every value is an odd multiple of 2^-24 (24 significant bits), so it is exact in
 * float32 as in double, and never 0 or 1. */
double or_uniform(uint64_t seed, uint64_t n)
{
    const uint64_t x = or_splitmix64(seed, n);
    return ((double)(x >> 41) + 0.5) / 8388608.0;
}

/* k distinct candidates drawn without replacement from q = softmax(logits / T), T > 0, by
 * the Gumbel-top-k trick (Vieira 2014; Kool, van Hoof and Welling, ICML 2019): with
 * U_v uniform on (0, 1) and G_v = -log(-log U_v) a standard Gumbel deviate, the tokens
 * with the k largest keys logits_v / T + G_v, taken by descending key, have the law of k
 * successive draws without replacement from q. Token v of row `row` uses output
 * n = row * V + v + 1 of SplitMix64 seeded with `seed`, so every (row, token) has its own
 * deviate. Ties of keys go to the smaller id.
 *   drawn[k]: the candidates in draw order (descending key), or NULL;
 *   ids[k]:   the same k tokens by descending logit (ties: ascending id), so that ids[0],
 *             the most probable candidate, is the one the Backbone Expansion tree extends
 *             (Sec. 2.2). */
/* The keys of the draw above: key[v] = logits[v] / T + G_v for row `row`. */
void or_sample_keys(const double *logits, int64_t V, double T, uint64_t seed, int64_t row, double *key)
{
    for (int64_t v = 0; v < V; ++v) {
        const uint64_t n = MUT(38) ? (uint64_t)v + 1 : (uint64_t)row * (uint64_t)V + (uint64_t)v + 1;
        const double u = or_uniform(seed, n);
        const double g = MUT(37) ? log(-log(u)) : -log(-log(u));
        key[v] = (MUT(39) ? logits[v] : logits[v] / T) + g;
    }
}

void or_topk_sample(const double *logits, int64_t V, int32_t k, double T, uint64_t seed, int64_t row,
                    int32_t *ids, int32_t *drawn)
{
    double *key = (double *)malloc((size_t)V * sizeof(double));
    int32_t *d = (int32_t *)malloc((size_t)k * sizeof(int32_t));
    unsigned char *taken = (unsigned char *)calloc((size_t)V, 1);
    or_sample_keys(logits, V, T, seed, row, key);
    for (int32_t r = 0; r < k; ++r) {
        int64_t best = -1;
        for (int64_t v = 0; v < V; ++v)
            if (!taken[v] && (best < 0 || key[v] > key[best]))
                best = v;
        d[r] = (int32_t)best;
        taken[best] = 1;
    }
    if (drawn)
        memcpy(drawn, d, (size_t)k * sizeof(int32_t));
    /* order the drawn set by (descending logit, ascending id): insertion sort */
    for (int32_t r = 0; r < k; ++r)
        ids[r] = d[r];
    if (!MUT(40))
        for (int32_t r = 1; r < k; ++r) {
            const int32_t t = ids[r];
            int32_t j = r - 1;
            while (j >= 0 && (logits[ids[j]] < logits[t] || (logits[ids[j]] == logits[t] && ids[j] > t))) {
                ids[j + 1] = ids[j];
                --j;
            }
            ids[j + 1] = t;
        }
    free(taken);
    free(d);
    free(key);
}

/* or_topk_sample over R rows of logits [R, V]: row r uses counter row r0 + r. Rows are
 * independent, so OpenMP splits them. */
void or_topk_sample_rows(const double *logits, int64_t R, int64_t V, int32_t k, double T, uint64_t seed,
                         int64_t r0, int32_t *ids, int32_t *drawn)
{
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < R; ++r)
        or_topk_sample(logits + r * V, V, k, T, seed, r0 + r, ids + r * k, drawn ? drawn + r * k : NULL);
}

/* Sec. 2.2, Backbone Expansion, in level-major order with T = 1 + N k nodes.
 *   node 0: the root, token `root` (the last verified token whose embedding fed the
 *           cascade), parent -1, depth 0;
 *   level i = 1..N: nodes 1 + (i-1)k + r, r = 0..k-1, hold topk[i-1][r] in rank
 *           order at depth i; their parent is the root for i = 1 and the previous
 *           level's rank-0 (backbone) node 1 + (i-2)k otherwise;
 *   mask[a][c] = 1 iff c is a or an ancestor of a. */
void or_tree(int32_t N, int32_t k, int32_t root, const int32_t *topk, int32_t *tok,
             int32_t *parent, int32_t *depth, uint8_t *mask)
{
    const int32_t T = 1 + N * k;
    tok[0] = root;
    parent[0] = -1;
    depth[0] = 0;
    for (int32_t i = 1; i <= N; ++i) {
        for (int32_t r = 0; r < k; ++r) {
            int32_t n = 1 + (i - 1) * k + r;
            tok[n] = topk[(int64_t)(i - 1) * k + r];
            depth[n] = MUT(28) ? i - 1 : i;
            if (i == 1)
                parent[n] = 0;
            else
                parent[n] = MUT(13) ? 1 + (i - 2) * k + (k - 1) : 1 + (i - 2) * k;
        }
    }
    memset(mask, 0, (size_t)T * (size_t)T);
    for (int32_t a = 0; a < T; ++a) {
        if (!MUT(16))
            mask[(int64_t)a * T + a] = 1;
        for (int32_t c = parent[a]; c >= 0; c = parent[c])
            mask[(int64_t)a * T + c] = 1;
    }
}

/* Smooth L1 of Eq. 6: 0.5 x^2 for |x| < 1, |x| - 0.5 otherwise. */
double or_smooth_l1(double x)
{
    const double a = fabs(x);
    return a < 1.0 ? (MUT(32) ? x * x : 0.5 * x * x) : a - 0.5;
}

/* The multi-level training objective of Sec. 2.3 (Eq. 3-6), forward only, for one sequence:
 *   logits [N][V]: the drafter's logits of depth i, q_i = softmax(logits_i) (temperature 1);
 *   teacher [N][V]: the target model's teacher distribution p_{t+i};
 *   hidden, feat [N][d]: the drafter's h_i and the target features f_i.
 * ce[i] = -sum_k p_k log q_k (Eq. 4); fl[i] = sum_j SmoothL1(h_ij - f_ij) (Eq. 5);
 * returns L_total = sum_i w_i (alpha ce[i] + beta fl[i]) with w_i = decay^(N - i) for the
 * 1-based depth i (Eq. 3; the paper uses decay 0.9, alpha 0.1, beta 1). */
double or_loss(int32_t N, int64_t V, int64_t d, const double *logits, const double *teacher,
               const double *hidden, const double *feat, double alpha, double beta, double decay,
               double *ce, double *fl)
{
    double *q = (double *)malloc(sizeof(double) * (size_t)V);
    double total = 0.0;
    for (int32_t i = 0; i < N; ++i) {
        double lse;
        or_softmax(logits + (int64_t)i * V, V, 1.0, q, &lse);
        double c = 0.0;
        for (int64_t k = 0; k < V; ++k) {
            const double pk = teacher[(int64_t)i * V + k];
            c -= MUT(33) ? q[k] * log(pk) : pk * log(q[k]);
        }
        double f = 0.0;
        for (int64_t j = 0; j < d; ++j)
            f += or_smooth_l1(hidden[(int64_t)i * d + j] - feat[(int64_t)i * d + j]);
        ce[i] = c;
        fl[i] = f;
        const double w = pow(decay, (double)(MUT(31) ? i : N - 1 - i));
        total += w * (alpha * c + beta * f);
    }
    free(q);
    return total;
}

/* Verification side of one cycle (Sec. 2.4, "Parallel Verification"), for one sequence's
 * draft tree of T nodes (or_tree's tok, parent, depth):
 *   pos[a] = P + depth[a]: the sequence position of node a under tree attention (the root,
 *            the token fed to the drafter, sits right after the P-token prefix);
 *   the greedy acceptance walk: starting at the root, the child of the current node whose
 *   token equals target_next[current] (the target model's greedy token after that node) is
 *   accepted and becomes current, until no child matches. path[0..n) are the accepted node
 *   ids (-1 after), *bonus = target_next[last accepted node, or the root]; returns n. Children
 *   are searched in node order, so with repeated tokens among siblings the first one wins. */
int32_t or_accept_greedy(int32_t T, const int32_t *tok, const int32_t *parent, const int32_t *depth,
                         const int32_t *target_next, int32_t P, int32_t max_path, int32_t *pos,
                         int32_t *path, int32_t *bonus)
{
    for (int32_t a = 0; a < T; ++a)
        pos[a] = P + depth[a] + (MUT(29) ? 1 : 0);
    int32_t cur = 0, n = 0;
    while (n < max_path) {
        int32_t next = -1;
        for (int32_t c = 1; c < T && next < 0; ++c)
            if (parent[c] == cur && tok[c] == target_next[MUT(30) ? c : cur])
                next = c;
        if (next < 0)
            break;
        path[n++] = next;
        cur = next;
    }
    for (int32_t i = n; i < max_path; ++i)
        path[i] = -1;
    *bonus = target_next[cur];
    return n;
}

/* Lossless verification of a sampled draft tree (Sec. 2.4, "the speculative sampling
 * algorithm identifies the longest accepted token path"; the paper names no variant, and it
 * is read as recursive rejection sampling over each node's children in draw order), for B
 * sequences:
 *   tok, parent, depth [B][T]  the trees (or_tree's layout), T = 1 + N k;
 *   rank [B][T]    a node's position in its level's draw order (0 = drawn first; the root's
 *                  entry is not read);
 *   q [B][N][V]    the drafter's proposal at each depth, softmax(l_i / T) (the law the
 *                  level's candidates were drawn from, without replacement);
 *   p [B][T][V]    the target's next-token distribution after each node (given the node's
 *                  root path), at the same temperature;
 *   u_acc, u_bonus [B][T]  uniform deviates on (0, 1), one test and one bonus draw per node.
 * Recursive rejection sampling over draws without replacement (the multi-candidate form of
 * speculative sampling, Leviathan et al. and Chen et al. 2023; Jeon et al. 2024): at the
 * current node, with r = its p and s = the next depth's q, the children are tested in draw
 * order; child c with token x is accepted iff u_acc[c] * s(x) <= r(x), that is with
 * probability min(1, r(x) / s(x)); on rejection r becomes max(r - s, 0) renormalised and x
 * is removed from s (renormalised), the law of the next draw. An accepted child becomes the
 * current node. When every child is rejected, or the node has none, the bonus token is drawn
 * from r by inverse CDF: the smallest x with u_bonus[current] < r(0) + ... + r(x).
 * path[b][0..n) are the accepted node ids (-1 after), n_accept[b] = n, bonus[b] the drawn
 * token. Every emitted token then has the target's law.
 * margin[b] (or NULL): how far the sequence's closest decision was from going the other way,
 * in units of the error bound of a float32 walk: |u_acc * s(x) - r(x)| for a test, and the
 * distance of u_bonus to the nearer edge of the picked token's CDF interval, each divided by
 * E = 2^-24 (2 S / Z + 5). Z is the current residual's normaliser (1 for a target
 * distribution itself) and S bounds the error mass a float32 residual carries: 0 for a
 * target distribution; each rejection adds at most 5 roundings of mass one (r, s and their
 * difference, each summing to at most 1) after dividing what it carried by the normaliser it
 * consumed, S <- S / Z + 5 2^-24. A float32 walk with exact sums can only decide differently
 * where the margin is below 1. The margin does not enter the walk. */
void or_accept_sampled(int32_t B, int32_t T, int32_t N, int64_t V, const int32_t *tok, const int32_t *parent,
                       const int32_t *depth, const int32_t *rank, const double *q, const double *p,
                       const double *u_acc, const double *u_bonus, int32_t *path, int32_t *n_accept,
                       int32_t *bonus, double *margin)
{
#pragma omp parallel for schedule(static)
    for (int32_t b = 0; b < B; ++b) {
        const int32_t *tk = tok + (int64_t)b * T, *par = parent + (int64_t)b * T, *dep = depth + (int64_t)b * T;
        const int32_t *rk = rank + (int64_t)b * T;
        double *r = (double *)malloc((size_t)V * sizeof(double));
        double *s = (double *)malloc((size_t)V * sizeof(double));
        int32_t *kids = (int32_t *)malloc((size_t)T * sizeof(int32_t));
        int32_t cur = 0, n = 0;
        double closest = INFINITY;
        const double ulp = 1.0 / 16777216.0;  /* 2^-24 */
        double zcur = 1.0, serr = 0.0;        /* the error model of the margin (see above) */
        memcpy(r, p + ((int64_t)b * T + cur) * V, (size_t)V * sizeof(double));
        for (;;) {
            /* the children of cur, in draw order */
            int32_t m = 0;
            for (int32_t c = 1; c < T; ++c)
                if (par[c] == cur)
                    kids[m++] = c;
            for (int32_t i = 1; i < m; ++i) {
                const int32_t t = kids[i];
                int32_t j = i - 1;
                while (j >= 0 && (MUT(44) ? kids[j] > t : rk[kids[j]] > rk[t])) {
                    kids[j + 1] = kids[j];
                    --j;
                }
                kids[j + 1] = t;
            }
            if (m == 0 || n >= N)
                break;
            memcpy(s, q + ((int64_t)b * N + dep[cur]) * V, (size_t)V * sizeof(double));
            int32_t next = -1;
            for (int32_t i = 0; i < m && next < 0; ++i) {
                const int32_t c = kids[i], x = tk[c];
                const int accept = MUT(41) ? u_acc[(int64_t)b * T + c] * r[x] <= s[x]
                                           : u_acc[(int64_t)b * T + c] * s[x] <= r[x];
                closest = fmin(closest, fabs(u_acc[(int64_t)b * T + c] * s[x] - r[x]) /
                                            (ulp * (2.0 * serr / zcur + 5.0)));
                if (accept) {
                    next = c;
                    break;
                }
                double sr = 0.0;
                for (int64_t v = 0; v < V; ++v) {
                    const double dlt = r[v] - s[v];
                    r[v] = (MUT(42) || dlt > 0.0) ? dlt : 0.0;
                    sr += r[v];
                }
                serr = serr / zcur + 5.0;  /* in units of 2^-24 */
                zcur = sr > 0.0 ? sr : 1.0;
                if (sr > 0.0)
                    for (int64_t v = 0; v < V; ++v)
                        r[v] /= sr;
                if (!MUT(43)) {
                    const double sx = s[x];
                    s[x] = 0.0;
                    if (sx < 1.0)
                        for (int64_t v = 0; v < V; ++v)
                            s[v] /= 1.0 - sx;
                }
            }
            if (next < 0)
                break;
            path[(int64_t)b * N + n++] = next;
            cur = next;
            zcur = 1.0;
            serr = 0.0;
            memcpy(r, p + ((int64_t)b * T + cur) * V, (size_t)V * sizeof(double));
        }
        for (int32_t i = n; i < N; ++i)
            path[(int64_t)b * N + i] = -1;
        n_accept[b] = n;
        /* the bonus token: inverse CDF of r */
        const double u = u_bonus[(int64_t)b * T + cur];
        double cum = 0.0;
        int32_t pick = -1, last = 0;
        for (int64_t v = 0; v < V && pick < 0; ++v) {
            if (r[v] > 0.0)
                last = (int32_t)v;
            cum += r[v];
            if (u < cum) {
                pick = (int32_t)v;
                closest = fmin(closest, fmin(u - (cum - r[v]), cum - u) / (ulp * (2.0 * serr / zcur + 5.0)));
            }
        }
        if (pick < 0)
            closest = fmin(closest, (u - cum) / (ulp * (2.0 * serr / zcur + 5.0)));
        bonus[b] = pick >= 0 ? pick : last; /* u above a sum rounded below 1 */
        if (margin)
            margin[b] = closest;
        free(kids);
        free(s);
        free(r);
    }
}

/* The whole draft of one sequence (Eq. 1, Eq. 2, Sec. 2.1 LM head, Sec. 2.2 top-k).
 *   w     : 5 + 7N pointers: w_fuse [d,3d], w_in [d,2d], embed [V,d], lm_head [V,d],
 *           final_norm [d], then per layer attn_norm, w_qkv, w_o, mlp_norm, w_gate,
 *           w_up, w_down
 *   feat  : [3d] = concat(l, m, h) of the last verified position
 *   tok   : the next token t+1 whose embedding joins the fused feature
 *   P     : prefix length (the drafted row's sequence position under the default reading)
 *   kc, vc: N pointers, each this sequence's [Hkv][cap][hd] cache of layer i
 * Outputs: hidden [N][d]; logits [N][V] (may be NULL); lse [N]; topk_id [N][k];
 * topk_logit [N][k]; topk_prob [N][k]. */
/* Eq. 1 for one row: g = FC(concat(l, m, h)) of feat [3d], e = Embed[tok],
 * x0 = FC(concat(g, e)); w as for or_draft_seq. */
static void input_row(const or_config *c, const void *const *w, const void *feat, int32_t tok, double *x0)
{
    const int32_t d = c->d, V = c->vocab;
    double *f = (double *)malloc(sizeof(double) * (size_t)(3 * d));
    double *ge = (double *)malloc(sizeof(double) * (size_t)(2 * d));
    /* g = FC(concat(l, m, h)) */
    or_widen(feat, c->dtype, 3 * d, f);
    if (MUT(18))
        for (int32_t j = 2 * d; j < 3 * d; ++j)
            f[j] = 0.0;
    double *g = MUT(14) ? ge + d : ge;
    double *e = MUT(14) ? ge : ge + d;
    or_matvec(w[0], c->dtype, d, 3 * d, f, g);
    /* e = Embed[tok] */
    const int64_t row = MUT(15) ? (tok + 1) % V : tok;
    for (int32_t j = 0; j < d; ++j)
        e[j] = ld(w[2], c->dtype, row * d + j);
    /* x0 = FC(concat(g, e))   (Eq. 1) */
    or_matvec(w[1], c->dtype, d, 2 * d, ge, x0);
    free(f); free(ge);
}

int32_t or_draft_seq(const or_config *c, const void *const *w, const void *feat, int32_t tok,
                     int32_t P, const void *const *kc, const void *const *vc, int64_t cap,
                     int32_t top_k, double temperature, double *hidden, double *logits,
                     double *lse, int32_t *topk_id, double *topk_logit, double *topk_prob)
{
    const int32_t d = c->d, V = c->vocab, N = c->n_layers;
    if (tok < 0 || tok >= V || P < 0 || P + 1 > cap || top_k < 1 || top_k > V)
        return -1;
    double *x0 = (double *)malloc(sizeof(double) * (size_t)d);
    double *x = (double *)malloc(sizeof(double) * (size_t)d);
    double *lg = (double *)malloc(sizeof(double) * (size_t)V);
    double *pr = (double *)malloc(sizeof(double) * (size_t)V);

    input_row(c, w, feat, tok, x0);
    memcpy(x, x0, sizeof(double) * (size_t)d);

    /* h_i = L_i(h_{i-1})      (Eq. 2), or h_i = L_i(x0) for the parallel ablation */
    for (int32_t i = 0; i < N; ++i) {
        if (c->parallel_layers || MUT(10))
            memcpy(x, x0, sizeof(double) * (size_t)d);
        double pos = (double)P + (c->rope_layer_offset ? (double)i : 0.0) + (MUT(19) ? 1.0 : 0.0);
        or_layer(c, w + 5 + 7 * i, pos, kc[i], vc[i], cap, P, x, NULL, NULL);
        memcpy(hidden + (int64_t)i * d, x, sizeof(double) * (size_t)d);
    }

    /* q_{t+i} through the frozen LM head; top-k per depth (Sec. 2.1, Sec. 2.2) */
    for (int32_t i = 0; i < N; ++i) {
        or_lm_head(c, w[3], w[4], hidden + (int64_t)i * d, lg);
        or_softmax(lg, V, temperature, pr, lse + i);
        or_topk(lg, V, top_k, topk_id + (int64_t)i * top_k);
        for (int32_t r = 0; r < top_k; ++r) {
            int32_t id = topk_id[(int64_t)i * top_k + r];
            topk_logit[(int64_t)i * top_k + r] = lg[id];
            topk_prob[(int64_t)i * top_k + r] = pr[id];
        }
        if (logits)
            memcpy(logits + (int64_t)i * V, lg, sizeof(double) * (size_t)V);
    }
    free(x0); free(x); free(lg); free(pr);
    return 0;
}

/* Sec. 2.4, "Update and Iterate": the paper appends the accepted tokens and updates the
 * target's cache; the drafter's per-layer caches are read as needing rows for the accepted
 * positions too, before the next draft attends to them. Once the target has accepted a
 * path, this commit step gives them those rows.
 * Row i (0 <= i < n) sits at sequence position P + i; its inputs are feat[i] ([3d], the
 * target's fused features of the position before it) and tok[i] (the token at P + i). It
 * goes through Eq. 1 and the cascade exactly like a drafted row (no LM head): layer l
 * attends to cache rows 0 .. P + i - 1 -- which include the rows of this commit before it
 * -- plus its own key and value, and then stores its key (rotated) and value in slot
 * P + i of layer l's cache, in the cache's storage type (see st()). kc / vc: N pointers to
 * this sequence's [Hkv][cap][hd] caches, written in place. Returns 0, or -1 on an invalid
 * argument (nothing written). */
int32_t or_commit_seq(const or_config *c, const void *const *w, const void *feat, const int32_t *tok,
                      int32_t n, int32_t P, void *const *kc, void *const *vc, int64_t cap)
{
    const int32_t d = c->d, V = c->vocab, N = c->n_layers, Hkv = c->n_kv_heads, hd = c->head_dim;
    if (n < 0 || P < 0 || (int64_t)P + n > cap)
        return -1;
    for (int32_t i = 0; i < n; ++i)
        if (tok[i] < 0 || tok[i] >= V)
            return -1;
    const int64_t nkv = (int64_t)Hkv * hd;
    double *x0 = (double *)malloc(sizeof(double) * (size_t)d);
    double *x = (double *)malloc(sizeof(double) * (size_t)d);
    double *kn = (double *)malloc(sizeof(double) * (size_t)nkv);
    double *vn = (double *)malloc(sizeof(double) * (size_t)nkv);
    for (int32_t i = 0; i < n; ++i) {
        const int32_t p = P + i;
        input_row(c, w, (const unsigned char *)feat + (size_t)i * 3 * d * (c->dtype == 0 ? 4 : 2), tok[i], x0);
        memcpy(x, x0, sizeof(double) * (size_t)d);
        for (int32_t l = 0; l < N; ++l) {
            if (c->parallel_layers)
                memcpy(x, x0, sizeof(double) * (size_t)d);
            const double pos = (double)p + (c->rope_layer_offset ? (double)l : 0.0) + (MUT(36) ? 1.0 : 0.0);
            or_layer(c, w + 5 + 7 * l, pos, kc[l], vc[l], cap, MUT(34) ? P : p, x, kn, vn);
            const int32_t slot = MUT(35) ? p + 1 < cap ? p + 1 : p : p;
            for (int32_t g = 0; g < Hkv; ++g)
                for (int32_t j = 0; j < hd; ++j) {
                    st(kc[l], c->dtype, ((int64_t)g * cap + slot) * hd + j, kn[(int64_t)g * hd + j]);
                    st(vc[l], c->dtype, ((int64_t)g * cap + slot) * hd + j, vn[(int64_t)g * hd + j]);
                }
        }
    }
    free(x0); free(x); free(kn); free(vn);
    return 0;
}

/* Threads the OpenMP runtime will use (reported beside CPU timings). */
int32_t or_max_threads(void)
{
#ifdef _OPENMP
    extern int omp_get_max_threads(void);
    return (int32_t)omp_get_max_threads();
#else
    return 1;
#endif
}

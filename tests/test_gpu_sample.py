"""Stochastic drafting on the GPU (Sec. 2.2, "sample k candidates") against the oracle's
draw (or_topk_sample) on identical seeded inputs and the same counter-based deviates.

Per sequence b and depth i the GPU's drawn set, in its reported draw order (topk_rank),
must be the oracle's draw: the k largest keys logit / T + G, G from SplitMix64 output
(b N + i - 1) V + v + 1 of the call's seed. The exemption is the top-k rule's: a rank may
differ only where the oracle's adjacent key gap is below 1e-2 / min(T, 1) (the logit
tolerance carried through the 1 / T scale), and the substitute must sit in that band. The
drawn set is reported ordered by logit (ties to the smaller id), its logits and
probabilities match the oracle's, and the tree is bit-exact on the GPU's candidates. All
three LM-head kernels are covered: the CUDA-core one (float32, and bf16 forced), the 16-row
tensor-core one (N B <= 16) and the wide one (N B > 16, k <= 8 and k <= 16; N B <= 16 with z
as bf16 hi + lo, forced on the small vocabularies), plus the batched-serving workload at full
size.
"""
import numpy as np
import pytest

from fe_synth import workloads as wl
import harness as H

pytestmark = pytest.mark.gpu


def key_gap(T: float) -> float:
    return H.TIE_GAP / min(T, 1.0)


CASES = {
    # float32, N B = 3: the CUDA-core LM head
    "tiny_f32_T1": dict(name="tiny", T=1.0, seed=11),
    "tiny_f32_T07": dict(name="tiny", T=0.7, seed=2**63 + 12),
    # bf16, N B = 12: the 16-row tensor-core LM head (ragged prefixes, V % 128 != 0); the wide
    # one with z as hi + lo on the same case below
    "gqa4_bf16_16row": dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1376, vocab=5003, n_layers=4,
                                      dtype="bf16", B=3, prefix=0, top_k=8, rope_theta=1e4, seed=3, page_size=0),
                            prefix_list=[37, 0, 150], T=1.0, seed=7),
    # 313 vocabulary tiles split between neighbouring CTAs, T = 0.7
    "split_v40k_T07": dict(name=dict(d=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=704, vocab=40003, n_layers=4,
                                     dtype="bf16", B=3, prefix=0, top_k=8, rope_theta=1e4, seed=21, page_size=0),
                           prefix_list=[5, 0, 70], T=0.7, seed=99),
    # N B = 36: the wide tensor-core LM head, k <= 8
    "wide_k8": dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1408, vocab=5003, n_layers=3,
                              dtype="bf16", B=12, prefix=0, top_k=8, rope_theta=1e4, seed=9, page_size=0),
                    prefix_list=[37, 0, 150, 1, 64, 5, 300, 2, 128, 129, 7, 90], T=1.0, seed=1234),
    # N B = 160, k = 12: the wide head's 16-entry lists, three 64-row groups, T = 0.7
    "wide_k12_r160": dict(name=dict(d=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=704, vocab=3001, n_layers=5,
                                    dtype="bf16", B=32, prefix=0, top_k=12, rope_theta=1e4, seed=12, page_size=0),
                          prefix_list=[(53 * b + 7) % 97 for b in range(32)], T=0.7, seed=5),
    # k = 1: one draw per depth, a chain
    "chain_k1": dict(name=dict(d=256, n_heads=4, n_kv_heads=4, head_dim=64, ffn=688, vocab=4096, n_layers=5,
                               dtype="bf16", B=2, prefix=0, top_k=1, rope_theta=1e4, seed=8, page_size=0),
                     prefix_list=[0, 33], T=1.0, seed=3),
}


def compare_sampled(orc, cfg, g, o, b, T, seed):
    N, k, V = cfg["n_layers"], cfg["top_k"], cfg["vocab"]
    f32 = cfg["dtype"] == "f32"
    for i in range(N):
        lg = o["logits"][i]
        keys = orc.sample_keys(lg, T, seed, b * N + i)
        ids, rank = g["topk_id"][b, i], g["topk_rank"][b, i]
        assert sorted(rank.tolist()) == list(range(k)), rank
        drawn = np.empty(k, np.int64)
        drawn[rank] = ids
        H.check_topk(drawn, keys, k, gap=key_gap(T))
        # when the draws agree exactly, the oracle's own (logit-ordered) list is the GPU's
        want_ids, want_drawn = orc.topk_sample(lg[None, :], k, T, seed, row0=b * N + i)
        if np.array_equal(drawn, want_drawn[0]):
            lgd = lg[want_ids[0]]
            ties = np.any(np.abs(np.diff(lgd)) < H.TIE_GAP) if k > 1 else False
            if not ties:
                assert np.array_equal(ids, want_ids[0]), (i, ids, want_ids[0])
        # reported order: descending logit, ties to the smaller id
        gl = g["topk_logit"][b, i]
        for r in range(k - 1):
            assert gl[r] > gl[r + 1] or (gl[r] == gl[r + 1] and ids[r] < ids[r + 1])
        # the candidates' logits and probabilities
        p_ref, lse_ref = orc.softmax(lg, T)
        if f32:
            assert np.abs(gl - lg[ids]).max() <= H.TOL_F32_REL * np.abs(lg).max()
            assert np.abs(g["topk_prob"][b, i] - p_ref[ids]).max() <= H.TOL_F32_REL * max(1e-3, p_ref[ids].max())
            assert abs(g["lse"][b, i] - lse_ref) <= H.TOL_F32_REL * abs(lse_ref)
        else:
            assert np.abs(gl - lg[ids]).max() <= H.TOL_BF16_LOGIT
            assert np.abs(g["topk_prob"][b, i] - p_ref[ids]).max() <= H.TOL_BF16_PROB
            assert abs(g["lse"][b, i] - lse_ref) <= H.TOL_BF16_LOGIT
        assert ((ids >= 0) & (ids < V)).all()
    tok, par, dep, mask = orc.tree(N, k, int(g["tree_tok"][b, 0]), g["topk_id"][b])
    assert np.array_equal(g["tree_tok"][b], tok) and np.array_equal(g["tree_parent"][b], par)
    assert np.array_equal(g["tree_depth"][b], dep) and np.array_equal(g["tree_mask"][b], mask)


def _problem(cfg):
    W = wl.make_weights(cfg)
    I = wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    return W, I, ks, vs


def _run_case(orc, spec, seqs=None):
    spec = dict(spec)
    name, T, seed = spec.pop("name"), spec.pop("T"), spec.pop("seed")
    cfg = wl.make_config(name, temperature=T, **spec)
    W, I, ks, vs = _problem(cfg)
    g = H.run_gpu(cfg, W, I, ks, vs, sample=True, seed=seed)
    assert g["status"] == 0, g["status"]
    for b in (range(cfg["B"]) if seqs is None else seqs(cfg, I)):
        o = H.run_oracle(orc, cfg, W, I, ks, vs, b)
        compare_sampled(orc, cfg, g, o, b, T, seed)
    return cfg, g


@pytest.mark.parametrize("case", list(CASES))
def test_sampled_draft_matches_oracle(orc, case):
    _run_case(orc, CASES[case])


@pytest.mark.parametrize("case", ["gqa4_bf16_16row", "split_v40k_T07"])
def test_sampled_draft_wide_lm_head_hi_lo_forced(orc, monkeypatch, case):
    """N B <= 16 on the wide tensor-core LM head with z as bf16 hi + lo
    (FE_DRAFT_LMHEAD_16ROW=0; by default it takes only the large vocabularies)."""
    monkeypatch.setenv("FE_DRAFT_LMHEAD_16ROW", "0")
    _run_case(orc, CASES[case])


def test_sampled_draft_cuda_core_lm_head_forced(orc, monkeypatch):
    """bf16 on the CUDA-core LM head (FE_DRAFT_LMHEAD_CUDA_CORES=1)."""
    monkeypatch.setenv("FE_DRAFT_LMHEAD_CUDA_CORES", "1")
    _run_case(orc, CASES["gqa4_bf16_16row"])


def test_sampled_draft_full_size_batched(orc):
    """The batched-serving workload (LLaMA-3.1-8B shape, B = 32, paged) at T = 1, in the
    launch configuration the benchmark times: sequences with the shortest and longest
    prefixes and the first and last."""
    def seqs(cfg, I):
        plen = I["prefix_len"].tolist()
        return sorted({0, cfg["B"] - 1, int(np.argmin(plen)), int(np.argmax(plen))})
    _run_case(orc, dict(name="b32_l31", T=1.0, seed=20250901), seqs)


def test_sampling_is_deterministic_and_seeded():
    """The same seed gives the same draw (graph replay included); another seed, another draw;
    greedy calls on the same handle are unchanged by sampled ones."""
    import paper_2509_20416_gb300 as fe
    spec = dict(CASES["gqa4_bf16_16row"])
    cfg = wl.make_config(spec.pop("name"), temperature=1.0, prefix_list=spec["prefix_list"])
    W, I, ks, vs = _problem(cfg)
    h = fe.fe_draft_init(dict(cfg, max_batch=cfg["B"]), W)
    greedy0 = H.run_gpu(cfg, W, I, ks, vs, handle=h, dbg=False)
    a = H.run_gpu(cfg, W, I, ks, vs, handle=h, dbg=False, sample=True, seed=1)
    b = H.run_gpu(cfg, W, I, ks, vs, handle=h, dbg=False, sample=True, seed=1)
    c = H.run_gpu(cfg, W, I, ks, vs, handle=h, dbg=False, sample=True, seed=2)
    greedy1 = H.run_gpu(cfg, W, I, ks, vs, handle=h, dbg=False)
    for key in ("topk_id", "topk_rank", "topk_logit", "topk_prob", "lse"):
        assert np.array_equal(a[key], b[key]), key
        assert np.array_equal(greedy0[key], greedy1[key]), key
    assert not np.array_equal(a["topk_id"], c["topk_id"])
    # greedy: the rank is the list position
    assert (greedy0["topk_rank"] == np.arange(cfg["top_k"])).all()
    h.close()


def test_sampling_needs_a_temperature():
    import paper_2509_20416_gb300 as fe
    cfg = wl.make_config("tiny")
    W, I, ks, vs = _problem(cfg)
    h = fe.fe_draft_init(dict(cfg, max_batch=1), W)
    with pytest.raises(fe.FeError) as e:
        fe.fe_draft_forward(h, I["feat"].cuda(), I["next_tok"].cuda(), I["prefix_len"].cuda(),
                            [t.cuda() for t in ks], [t.cuda() for t in vs], cfg["top_k"], 0.0, sample=True, seed=1)
    assert e.value.code == fe.FE_ERR_INVALID_ARG
    h.close()

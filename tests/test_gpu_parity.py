"""CUDA path (through the C ABI) against the fp64 oracle on identical seeded inputs.

Small cases span several row groups, vocabulary slabs and attention splits with ragged
tails (V % 4 != 0, prefixes that end mid-page, P = 0); the five named workloads run at
full size, with the oracle computing every compared sequence one by one.
"""
import numpy as np
import pytest
import torch

from fe_synth import workloads as wl
import harness as H
import torch_ref

pytestmark = pytest.mark.gpu


def _problem(cfg):
    W = wl.make_weights(cfg)
    I = wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    return W, I, ks, vs


def _new_row_ref(cfg, W, I, o, b, i):
    """Expected key (after RoPE) and value the call appends to layer i's slot P_b."""
    d, Hh, Hkv, hd = cfg["d"], cfg["n_heads"], cfg["n_kv_heads"], cfg["head_dim"]
    if i == 0 or cfg.get("parallel_layers", 0):  # the layer's input is x0
        f = I["feat"][b].double()
        g = W["w_fuse"].double() @ f
        e = W["embed"].double()[int(I["next_tok"][b])]
        x = W["w_in"].double() @ torch.cat([g, e])
    else:
        x = torch.tensor(o["hidden"][i - 1])
    L = W["layers"][i]
    u = torch.nn.functional.rms_norm(x, (d,), weight=L["attn_norm"].double(), eps=cfg["rms_eps"])
    qkv = L["w_qkv"].double() @ u
    k = qkv[Hh * hd:(Hh + Hkv) * hd].view(Hkv, hd)
    v = qkv[(Hh + Hkv) * hd:].view(Hkv, hd)
    k = torch_ref.rope_complex(k, int(I["prefix_len"][b]), cfg["rope_theta"])
    return k, v


def _check_cache_rows(cfg, W, I, ks, vs, g, o, b):
    P = int(I["prefix_len"][b])
    ps = cfg["page_size"]
    for i in range(cfg["n_layers"]):
        kref, vref = _new_row_ref(cfg, W, I, o, b, i)
        for cache, logical, ref in ((g["k_cache"][i], ks[i], kref), (g["v_cache"][i], vs[i], vref)):
            if ps:
                tab = g["page_table"]
                new = cache[int(tab[b, P // ps]), :, P % ps, :].double()
                old = (torch.stack([cache[int(tab[b, p // ps]), :, p % ps, :] for p in range(P)], 1)
                       if P else None)
            else:
                new = cache[b, :, P, :].double()
                old = cache[b, :, :P, :]
            if P:
                assert torch.equal(old, logical[b, :, :P, :]), f"layer {i}: prefix rows were modified"
            # the new row is stored in the cache's type: one rounding of the fp32 value
            rel = 2.0 ** -8 if cfg["dtype"] == "bf16" else 1e-5
            assert torch.allclose(new, ref, rtol=rel, atol=1e-4 * max(1.0, ref.abs().max().item())), i


SMALL = {
    "tiny_f32": dict(name="tiny"),
    "gqa4_bf16_ragged": dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1376, vocab=5003,
                                       n_layers=4, dtype="bf16", B=3, prefix=0, top_k=8, rope_theta=1e4,
                                       seed=3, page_size=0), prefix_list=[37, 0, 150]),
    "gqa4_bf16_paged": dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1376, vocab=5003,
                                      n_layers=3, dtype="bf16", B=4, prefix=0, top_k=8, rope_theta=5e5,
                                      seed=4, page_size=16), prefix_list=[15, 16, 1, 200]),
    "mha128_f32_temp": dict(name=dict(d=256, n_heads=2, n_kv_heads=2, head_dim=128, ffn=520, vocab=777,
                                      n_layers=2, dtype="f32", B=2, prefix=0, top_k=3, rope_theta=1e4,
                                      seed=5, page_size=0), prefix_list=[5, 63], temperature=0.7),
    "gqa8_bf16_k32": dict(name=dict(d=512, n_heads=8, n_kv_heads=1, head_dim=64, ffn=512, vocab=4100,
                                    n_layers=2, dtype="bf16", B=2, prefix=0, top_k=32, rope_theta=1e4,
                                    seed=6, page_size=0), prefix_list=[300, 1]),
    "chain_k1_b5": dict(name=dict(d=256, n_heads=4, n_kv_heads=4, head_dim=64, ffn=688, vocab=4096,
                                  n_layers=5, dtype="bf16", B=5, prefix=0, top_k=1, rope_theta=1e4,
                                  seed=8, page_size=0), prefix_list=[0, 1, 2, 33, 64]),
    # batched handles (max_batch > 8): the linear phases run on the tensor cores; several
    # tiles per matrix, tiles split between CTAs, ragged and paged prefixes
    "tc_linear_b12_ragged": dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1408, vocab=5003,
                                           n_layers=3, dtype="bf16", B=12, prefix=0, top_k=8, rope_theta=1e4,
                                           seed=9, page_size=0),
                                 prefix_list=[37, 0, 150, 1, 64, 5, 300, 2, 128, 129, 7, 90]),
    "tc_linear_b9_paged": dict(name=dict(d=1024, n_heads=8, n_kv_heads=8, head_dim=128, ffn=2816, vocab=3001,
                                         n_layers=2, dtype="bf16", B=9, prefix=0, top_k=4, rope_theta=5e5,
                                         seed=10, page_size=16), prefix_list=[15, 16, 1, 200, 0, 31, 33, 64, 100]),
    # the "w/o cascaded structure" ablation (Sec. 3.2, Table 2): every layer consumes x0
    "parallel_gqa4_bf16": dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1376, vocab=5003,
                                         n_layers=4, dtype="bf16", B=3, prefix=0, top_k=8, rope_theta=1e4,
                                         seed=13, page_size=0, parallel_layers=1), prefix_list=[37, 0, 150]),
    "parallel_tc_b12": dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1408, vocab=5003,
                                      n_layers=3, dtype="bf16", B=12, prefix=0, top_k=8, rope_theta=1e4,
                                      seed=14, page_size=0, parallel_layers=1),
                            prefix_list=[37, 0, 150, 1, 64, 5, 300, 2, 128, 129, 7, 90]),
    # rows too long for two weight slots per warp beside them: the activations are staged in
    # two column passes. B = 1 with a 27000-wide MLP (down projection over 27 slices, the last
    # one ragged); float32 weights, B = 3 (two activation rows per CTA, then one) through the
    # 12288-column feature FC
    "twopass_down_b1": dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=27000, vocab=3001,
                                      n_layers=2, dtype="bf16", B=1, prefix=0, top_k=8, rope_theta=1e4,
                                      seed=20, page_size=0), prefix_list=[77]),
    "twopass_fuse_f32_b3": dict(name=dict(d=4096, n_heads=32, n_kv_heads=8, head_dim=128, ffn=1024, vocab=3001,
                                          n_layers=1, dtype="f32", B=3, prefix=0, top_k=4, rope_theta=5e5,
                                          seed=21, page_size=0), prefix_list=[5, 0, 70]),
    # bf16, hd 128, G = 2, 4, 8 (G = 1 below and at full size): the tensor-core attention kernel. Prefixes on both sides of
    # the 32-key chunk and 128-key split boundaries, an empty prefix, several splits per
    # sequence (combined by the last split), page sizes 16 and 8, and contiguous caches.
    "tc_attn_g4_paged16": dict(name=dict(d=512, n_heads=4, n_kv_heads=1, head_dim=128, ffn=1376, vocab=3001,
                                         n_layers=2, dtype="bf16", B=6, prefix=0, top_k=8, rope_theta=5e5,
                                         seed=15, page_size=16), prefix_list=[0, 1, 31, 32, 129, 700]),
    "tc_attn_g8_contig": dict(name=dict(d=1024, n_heads=8, n_kv_heads=1, head_dim=128, ffn=1024, vocab=3001,
                                        n_layers=2, dtype="bf16", B=3, prefix=0, top_k=8, rope_theta=1e4,
                                        seed=16, page_size=0), prefix_list=[33, 0, 517]),
    "tc_attn_g2_paged8": dict(name=dict(d=512, n_heads=4, n_kv_heads=2, head_dim=128, ffn=1376, vocab=3001,
                                        n_layers=2, dtype="bf16", B=4, prefix=0, top_k=4, rope_theta=5e5,
                                        seed=17, page_size=8), prefix_list=[7, 8, 9, 260]),
    # page sizes 64 (a chunk inside one page) and 24 (chunks straddling pages, division
    # rather than shifts for the page lookup)
    "tc_attn_g8_paged64": dict(name=dict(d=1024, n_heads=8, n_kv_heads=1, head_dim=128, ffn=1024, vocab=3001,
                                         n_layers=2, dtype="bf16", B=3, prefix=0, top_k=8, rope_theta=1e4,
                                         seed=18, page_size=64), prefix_list=[63, 64, 300]),
    "tc_attn_g4_paged24": dict(name=dict(d=512, n_heads=4, n_kv_heads=1, head_dim=128, ffn=1376, vocab=3001,
                                         n_layers=2, dtype="bf16", B=4, prefix=0, top_k=8, rope_theta=5e5,
                                         seed=19, page_size=24), prefix_list=[23, 24, 47, 400]),
    # 313 vocabulary tiles (the last one ragged) over at most 152 CTAs with d = 256: the
    # 16-row LM head splits tiles between neighbouring CTAs; 12 rows, temperature 0.7 (the
    # wide LM head with z as hi + lo on the same case below)
    "lmhead_split_v40k": dict(name=dict(d=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=704, vocab=40003,
                                        n_layers=4, dtype="bf16", B=3, prefix=0, top_k=8, rope_theta=1e4,
                                        seed=21, page_size=0), prefix_list=[5, 0, 70], temperature=0.7),
    # N * B = 160 rows: the wide tensor-core LM head with three 64-row transpose groups
    "wide_lmhead_r160": dict(name=dict(d=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=704, vocab=3001,
                                       n_layers=5, dtype="bf16", B=32, prefix=0, top_k=8, rope_theta=1e4,
                                       seed=12, page_size=0),
                             prefix_list=[(53 * b + 7) % 97 for b in range(32)]),
}


@pytest.mark.parametrize("case", list(SMALL))
def test_parity_small(orc, case):
    spec = dict(SMALL[case])
    name = spec.pop("name")
    cfg = wl.make_config(name, **spec)
    W, I, ks, vs = _problem(cfg)
    g = H.run_gpu(cfg, W, I, ks, vs)
    assert g["status"] == 0, g["status"]
    for b in range(cfg["B"]):
        o = H.run_oracle(orc, cfg, W, I, ks, vs, b)
        H.compare(orc, cfg, g, o, b)
        _check_cache_rows(cfg, W, I, ks, vs, g, o, b)


@pytest.mark.parametrize("B", [1, 2, 32])
def test_parity_tensor_core_linear_forced(orc, monkeypatch, B):
    """The tensor-core linear path chosen explicitly, at one and two sequences (operand rows
    padded to 8) and at its maximum batch of 32."""
    monkeypatch.setenv("FE_DRAFT_LINEAR_MMA", "1")
    plist = [(37 * b + 11) % 160 for b in range(B)]
    cfg = wl.make_config(dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1408, vocab=4000, n_layers=2,
                              dtype="bf16", B=B, prefix=0, top_k=8, rope_theta=1e4, seed=11 + B, page_size=0),
                         prefix_list=plist)
    W, I, ks, vs = _problem(cfg)
    g = H.run_gpu(cfg, W, I, ks, vs)
    assert g["status"] == 0, g["status"]
    for b in sorted({0, B - 1, B // 2}):
        o = H.run_oracle(orc, cfg, W, I, ks, vs, b)
        H.compare(orc, cfg, g, o, b)
        _check_cache_rows(cfg, W, I, ks, vs, g, o, b)


@pytest.mark.parametrize("case", ["tc_attn_g4_paged16", "tc_attn_g8_contig"])
def test_parity_cuda_core_attention_forced(orc, monkeypatch, case):
    """bf16 GQA attention at hd 128 on the CUDA-core kernel (FE_DRAFT_ATTN_TC=0), which the
    tensor-core kernel replaces by default for these shapes."""
    monkeypatch.setenv("FE_DRAFT_ATTN_TC", "0")
    spec = dict(SMALL[case])
    cfg = wl.make_config(spec.pop("name"), **spec)
    W, I, ks, vs = _problem(cfg)
    g = H.run_gpu(cfg, W, I, ks, vs)
    assert g["status"] == 0, g["status"]
    for b in range(cfg["B"]):
        o = H.run_oracle(orc, cfg, W, I, ks, vs, b)
        H.compare(orc, cfg, g, o, b)
        _check_cache_rows(cfg, W, I, ks, vs, g, o, b)


def test_repeat_and_graph_replay_bit_identical():
    """Two calls with identical arguments (the second replays the captured CUDA graph)
    and a call without dbg buffers all give the same bits."""
    import paper_2509_20416_gb300 as fe
    cfg = wl.make_config(SMALL["gqa4_bf16_ragged"]["name"], prefix_list=[37, 0, 150])
    W, I, ks, vs = _problem(cfg)
    h = fe.fe_draft_init(dict(cfg, max_batch=cfg["B"]), W)
    a = H.run_gpu(cfg, W, I, ks, vs, handle=h)
    b = H.run_gpu(cfg, W, I, ks, vs, handle=h)
    c = H.run_gpu(cfg, W, I, ks, vs, handle=h, dbg=False)
    for key in ("topk_id", "topk_logit", "topk_prob", "lse", "tree_mask"):
        assert np.array_equal(a[key], b[key]) and np.array_equal(a[key], c[key]), key
    assert np.array_equal(a["logits"], b["logits"])
    h.close()


FULL = ["vic13b", "l31_8b", "l33_70b", "b32_l31"]


@pytest.mark.parametrize("name", FULL)
def test_parity_full_size(orc, name):
    """The named workloads at full size, in the launch configuration the benchmark times."""
    cfg = wl.make_config(name)
    W, I, ks, vs = _problem(cfg)
    g = H.run_gpu(cfg, W, I, ks, vs)
    assert g["status"] == 0, g["status"]
    B = cfg["B"]
    plen = I["prefix_len"].tolist()
    seqs = sorted({0, B - 1, int(np.argmin(plen)), int(np.argmax(plen))})
    stats = []
    for b in seqs:
        o = H.run_oracle(orc, cfg, W, I, ks, vs, b)
        stats.append(H.compare(orc, cfg, g, o, b))
        _check_cache_rows(cfg, W, I, ks, vs, g, o, b)
    print(name, stats)


@pytest.mark.parametrize("case", ["tc_linear_b12_ragged", "tc_linear_b9_paged", "parallel_tc_b12"])
def test_deferred_split_tiles_bit_identical(monkeypatch, case):
    """A tensor-core phase followed by another leaves the tiles it shares with other CTAs to
    that phase's operand prep, which sums the shares in CTA order and applies the epilogue
    there; the QKV phase leaves them to the attention kernel, which sums the shares of the
    query, key and value columns it reads. The draft must equal the one with the reduction
    inside each phase (FE_DRAFT_LIN_DEFER=0) bit for bit: logits, hidden states, candidates,
    caches."""
    spec = dict(SMALL[case])
    cfg = wl.make_config(spec.pop("name"), **spec)
    W, I, ks, vs = _problem(cfg)
    a = H.run_gpu(cfg, W, I, ks, vs)
    monkeypatch.setenv("FE_DRAFT_LIN_DEFER", "0")
    b = H.run_gpu(cfg, W, I, ks, vs)
    assert a["status"] == 0 and b["status"] == 0
    for key in ("logits", "hidden", "topk_id", "topk_logit", "topk_prob", "lse", "tree_tok"):
        assert np.array_equal(a[key], b[key]), key
    for i in range(cfg["n_layers"]):
        assert torch.equal(a["k_cache"][i], b["k_cache"][i]) and torch.equal(a["v_cache"][i], b["v_cache"][i]), i


@pytest.mark.parametrize("case", ["tc_linear_b12_ragged", "parallel_tc_b12"])
def test_norm_on_operand_matches_oracle(orc, monkeypatch, case):
    """The tensor-core RMSNorm phases with the scale applied to the operand by their prep
    (FE_DRAFT_LIN_NORMPOST=0) instead of to the products, against the oracle, and against
    the default draft within float32 rounding of the two orders of that scale."""
    spec = dict(SMALL[case])
    cfg = wl.make_config(spec.pop("name"), **spec)
    W, I, ks, vs = _problem(cfg)
    a = H.run_gpu(cfg, W, I, ks, vs)
    monkeypatch.setenv("FE_DRAFT_LIN_NORMPOST", "0")
    g = H.run_gpu(cfg, W, I, ks, vs)
    assert a["status"] == 0 and g["status"] == 0
    for b in range(cfg["B"]):
        H.compare(orc, cfg, g, H.run_oracle(orc, cfg, W, I, ks, vs, b), b)
    scale = np.abs(g["hidden"]).max()
    assert np.abs(a["hidden"] - g["hidden"]).max() <= 1e-5 * scale


@pytest.mark.parametrize("case", ["tc_linear_b12_ragged", "parallel_tc_b12"])
def test_attention_operand_path_is_exact(monkeypatch, case):
    """Batched tensor-core drafts: the attention kernel writes the O projection's bf16 hi / lo
    operand itself. The same draft with the attention output stored in float32 and split by
    the projection's own prep (FE_DRAFT_ATTN_OPERAND=0) gives identical results."""
    spec = dict(SMALL[case])
    cfg = wl.make_config(spec.pop("name"), **spec)
    W, I, ks, vs = _problem(cfg)
    a = H.run_gpu(cfg, W, I, ks, vs)
    monkeypatch.setenv("FE_DRAFT_ATTN_OPERAND", "0")
    b = H.run_gpu(cfg, W, I, ks, vs)
    assert a["status"] == 0 and b["status"] == 0
    for key in ("logits", "hidden", "topk_id", "topk_logit", "topk_prob", "lse", "tree_tok"):
        assert np.array_equal(a[key], b[key]), key


@pytest.mark.parametrize("case", ["lmhead_split_v40k", "gqa4_bf16_ragged", "tc_linear_b9_paged"])
def test_wide_lm_head_hi_lo_forced(orc, monkeypatch, case):
    """Up to 16 hidden rows the wide LM head (whole vocabulary tiles per CTA, z as bf16 hi +
    lo) runs on vocabularies of at least four tiles per CTA (the full-size 128256-entry heads);
    FE_DRAFT_LMHEAD_16ROW=0 selects it on these small ones, against the oracle."""
    monkeypatch.setenv("FE_DRAFT_LMHEAD_16ROW", "0")
    spec = dict(SMALL[case])
    cfg = wl.make_config(spec.pop("name"), **spec)
    W, I, ks, vs = _problem(cfg)
    g = H.run_gpu(cfg, W, I, ks, vs)
    assert g["status"] == 0, g["status"]
    for b in range(cfg["B"]):
        H.compare(orc, cfg, g, H.run_oracle(orc, cfg, W, I, ks, vs, b), b)

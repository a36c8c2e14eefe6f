"""Persistent linear stacks (B = 1 drafts): the same arithmetic as separate launches.

When every linear phase has at least one 4-row group per SM, the stack kernel partitions
each matrix exactly as the separate linear launches do and sums in the same order, so the
two paths must agree bit for bit; both are also checked against the oracle."""
import numpy as np
import pytest

from fe_synth import workloads as wl
import harness as H

pytestmark = pytest.mark.gpu

CFG = dict(d=1024, n_heads=8, n_kv_heads=4, head_dim=128, ffn=2816, vocab=3001, n_layers=3, dtype="bf16", B=1,
           prefix=0, top_k=8, rope_theta=1e4, seed=21, page_size=0)


def _run(monkeypatch, stack: str, cfg):
    monkeypatch.setenv("FE_DRAFT_STACK", stack)
    W, I = wl.make_weights(cfg), wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    return H.run_gpu(cfg, W, I, ks, vs), (W, I, ks, vs)


def test_stack_matches_separate_launches_bitwise(orc, monkeypatch):
    cfg = wl.make_config(CFG, prefix_list=[300])
    a, prob = _run(monkeypatch, "1", cfg)
    b, _ = _run(monkeypatch, "0", cfg)
    assert a["status"] == 0 and b["status"] == 0
    for key in ("topk_id", "topk_logit", "topk_prob", "lse", "logits", "hidden", "tree_tok", "tree_mask"):
        assert np.array_equal(a[key], b[key]), key
    o = H.run_oracle(orc, cfg, *prob, 0)
    H.compare(orc, cfg, a, o, 0)


def test_stack_fp32_small_rows(orc, monkeypatch):
    """fp32 with fewer row groups than SMs (empty row ranges in some CTAs)."""
    cfg = wl.make_config("tiny")
    a, prob = _run(monkeypatch, "1", cfg)
    assert a["status"] == 0
    o = H.run_oracle(orc, cfg, *prob, 0)
    H.compare(orc, cfg, a, o, 0)

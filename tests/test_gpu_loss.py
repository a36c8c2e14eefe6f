"""fe_draft_loss: the training objective's forward (Sec. 2.3, Eq. 3-6) against the oracle.

Tolerances: ce = lse * sum(p) - <p, logits> with sum(p) = 1, so |d ce| <= |d lse| + max|d logit|
(twice the logit tolerance for bf16 weights, relative 1e-4 for fp32); Smooth L1 is 1-Lipschitz,
so |d feat_loss| <= sum_j |d h_j| (the hidden states are float32 on every path)."""
import numpy as np
import pytest
import torch

from fe_synth import workloads as wl
import harness as H

pytestmark = pytest.mark.gpu

CASES = {
    "tiny_f32": dict(name="tiny"),
    "gqa4_bf16": dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1376, vocab=5003, n_layers=4,
                                dtype="bf16", B=3, prefix=0, top_k=8, rope_theta=1e4, seed=15, page_size=0),
                      prefix_list=[37, 0, 150]),
}


@pytest.mark.parametrize("case", list(CASES))
def test_loss_matches_oracle(orc, case):
    import paper_2509_20416_gb300 as fe
    spec = dict(CASES[case])
    name = spec.pop("name")
    cfg = wl.make_config(name, **spec)
    B, N, V, d = cfg["B"], cfg["n_layers"], cfg["vocab"], cfg["d"]
    W, I = wl.make_weights(cfg), wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    g = torch.Generator().manual_seed(17)
    teacher = torch.softmax(2.0 * torch.randn((B, N, V), generator=g), dim=-1).float()
    target = torch.randn((N, B, d), generator=g).float()
    h = fe.fe_draft_init(dict(cfg, max_batch=B), W)
    kd, vd, table, n_pages = H.device_caches(cfg, ks, vs, I["prefix_len"])
    out = fe.fe_draft_loss(h, I["feat"].cuda(), I["next_tok"].cuda(), I["prefix_len"].cuda(), kd, vd,
                           teacher.cuda(), target.cuda(), cfg["top_k"], page_table=table, n_pages=n_pages)
    torch.cuda.synchronize()
    assert fe.fe_last_device_status(h) == fe.FE_OK
    ce, fl, tot = (out[k].cpu().numpy() for k in ("ce", "feat_loss", "total"))
    tol_ce = 2 * H.TOL_BF16_LOGIT if cfg["dtype"] == "bf16" else None
    for b in range(B):
        o = H.run_oracle(orc, cfg, W, I, ks, vs, b)
        t_o, ce_o, fl_o = orc.loss(o["logits"], teacher[b].double().numpy(), o["hidden"],
                                   target[:, b].double().numpy(), 0.1, 1.0, 0.9)
        tc = tol_ce if tol_ce is not None else H.TOL_F32_REL * np.abs(ce_o).max()
        assert np.abs(ce[b] - ce_o).max() <= tc, (b, ce[b], ce_o)
        assert np.allclose(fl[b], fl_o, rtol=1e-4, atol=1e-3), (b, fl[b], fl_o)
        w = 0.9 ** (N - 1 - np.arange(N))
        assert abs(tot[b] - t_o) <= (w * (0.1 * tc + (1e-4 * np.abs(fl_o) + 1e-3))).sum(), (b, tot[b], t_o)
    h.close()


def test_loss_rejects_missing_buffers():
    import ctypes
    import paper_2509_20416_gb300 as fe
    a = fe.fe_forward_args()
    assert fe._lib.fe_draft_loss(None, ctypes.byref(a), None, None, 0.1, 1.0, 0.9, None, None, None, None) == \
        fe.FE_ERR_INVALID_ARG

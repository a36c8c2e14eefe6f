"""fe_lm_head_topk_noalloc: the LM head + softmax statistics + top-k for callers that
cannot allocate device memory (for example while a memory pool is frozen, or on a serving
path whose memory was fixed at start-up). It must give the same results as the same step
inside fe_draft_forward, call after call, although its working memory is a fixed device
array shared by every call instead of the handle's scratch.

Kept in its own file, collected last, so that a failure here cannot hide the others.
"""
import pytest
import torch

from fe_synth import workloads as wl

pytestmark = pytest.mark.gpu

CASES = {
    # bf16, n_layers * B = 12 rows: the tensor-core LM head
    "tensor_core": dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1376, vocab=5003, n_layers=4,
                                  dtype="bf16", B=3, prefix=0, top_k=8, rope_theta=1e4, seed=31, page_size=0),
                        prefix_list=[37, 0, 150], temperature=0.0),
    # fp32: the CUDA-core LM head, at temperature 0.7
    "cuda_core": dict(name=dict(d=256, n_heads=4, n_kv_heads=4, head_dim=64, ffn=688, vocab=4099, n_layers=3,
                                dtype="f32", B=2, prefix=0, top_k=5, rope_theta=1e4, seed=32, page_size=0),
                      prefix_list=[64, 9], temperature=0.7),
}


def _setup(case):
    import paper_2509_20416_gb300 as fe
    spec = dict(CASES[case])
    name = spec.pop("name")
    cfg = wl.make_config(name, **spec)
    W = wl.make_weights(cfg)
    I = wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    h = fe.fe_draft_init(dict(cfg, max_batch=cfg["B"]), W)
    return fe, cfg, h, I, ks, vs


@pytest.mark.parametrize("case", list(CASES))
def test_noalloc_lm_head_matches_forward_twice(case, orc):
    fe, cfg, h, I, ks, vs = _setup(case)
    B, N, d, k, T = cfg["B"], cfg["n_layers"], cfg["d"], cfg["top_k"], cfg["temperature"]
    hidden = torch.empty((N, B, d), device="cuda")
    ref = fe.fe_draft_forward(h, I["feat"].cuda(), I["next_tok"].cuda(), I["prefix_len"].cuda(),
                              [t.cuda() for t in ks], [t.cuda() for t in vs], k, T, dbg_hidden=hidden)
    torch.cuda.synchronize()
    assert fe.fe_last_device_status(h) == fe.FE_OK
    for call in range(2):  # the shared array keeps the previous call's contents
        out = fe.fe_lm_head_topk_noalloc(h, hidden, B, k, T)
        torch.cuda.synchronize()
        assert fe.fe_last_device_status(h) == fe.FE_OK, call
        assert torch.equal(out["topk_id"], ref["topk_id"]), call
        for key in ("topk_logit", "topk_prob", "lse"):
            assert torch.allclose(out[key], ref[key], rtol=1e-6, atol=1e-6), (call, key)
        ids = out["topk_id"].cpu().numpy()
        assert ((ids >= 0) & (ids < cfg["vocab"])).all()
    # and against the fp64 oracle's LM head over the same hidden rows (the final norm, the
    # logits, their softmax at T and the top-k), under the parity contract
    _check_against_oracle(orc, cfg, h, hidden, out)
    h.close()


def _check_against_oracle(orc, cfg, h, hidden, out):
    import numpy as np
    import harness as H
    W = wl.make_weights(cfg)
    B, N, k, T = cfg["B"], cfg["n_layers"], cfg["top_k"], cfg["temperature"]
    hid = hidden.cpu().numpy().astype(np.float64)  # [N, B, d]
    lg = orc.lm_head(cfg, W, hid.reshape(N * B, -1)).reshape(N, B, -1)
    ids, tl, tp, lse = (out[key].cpu().numpy() for key in ("topk_id", "topk_logit", "topk_prob", "lse"))
    for b in range(B):
        for i in range(N):
            ref = lg[i, b]
            p_ref, lse_ref = orc.softmax(ref, T if T > 0 else 1.0)
            H.check_topk(ids[b, i], ref, k)
            if cfg["dtype"] == "f32":
                scale = np.abs(ref).max()
                assert abs(lse[b, i] - lse_ref) <= H.TOL_F32_REL * abs(lse_ref), (b, i)
                assert np.abs(tl[b, i] - ref[ids[b, i]]).max() <= H.TOL_F32_REL * scale, (b, i)
                assert np.abs(tp[b, i] - p_ref[ids[b, i]]).max() <= H.TOL_F32_REL * max(1e-3, p_ref.max()), (b, i)
            else:
                assert abs(lse[b, i] - lse_ref) <= H.TOL_BF16_LOGIT, (b, i)
                assert np.abs(tl[b, i] - ref[ids[b, i]]).max() <= H.TOL_BF16_LOGIT, (b, i)
                assert np.abs(tp[b, i] - p_ref[ids[b, i]]).max() <= H.TOL_BF16_PROB, (b, i)


def test_noalloc_rejects_more_rows_than_its_scratch_holds():
    import paper_2509_20416_gb300 as fe
    cfg = wl.make_config(dict(d=256, n_heads=4, n_kv_heads=4, head_dim=64, ffn=688, vocab=1000, n_layers=3,
                              dtype="bf16", B=8, prefix=4, top_k=4, rope_theta=1e4, seed=33, page_size=0))
    h = fe.fe_draft_init(dict(cfg, max_batch=8), wl.make_weights(cfg))
    hidden = torch.zeros((3, 8, 256), device="cuda")
    with pytest.raises(fe.FeError) as e:
        fe.fe_lm_head_topk_noalloc(h, hidden, 8, 4)  # 3 x 8 = 24 rows > 16
    assert e.value.code == fe.FE_ERR_INVALID_ARG
    assert "fixed scratch" in fe.fe_last_error_detail()
    h.close()

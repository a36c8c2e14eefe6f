"""fe_profile_forward: the launch-by-launch timing that bench.py's per-kernel roofline
uses. It must run the same kernels as fe_draft_forward (same outputs, bit for bit) and
report one entry per launch in launch order."""
import pytest
import torch

from fe_synth import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("spec", [dict(name="tiny"),
                                  dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1376,
                                                 vocab=5003, n_layers=3, dtype="bf16", B=2, prefix=40, top_k=8,
                                                 rope_theta=1e4, seed=41, page_size=0)),
                                  # batched: tensor-core linear phases (operand prep + product)
                                  dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1408,
                                                 vocab=5003, n_layers=3, dtype="bf16", B=12, prefix=40, top_k=8,
                                                 rope_theta=1e4, seed=42, page_size=0))])
def test_profile_forward_matches_forward(spec):
    import paper_2509_20416_gb300 as fe
    cfg = wl.make_config(spec["name"])
    W, I = wl.make_weights(cfg), wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    h = fe.fe_draft_init(dict(cfg, max_batch=cfg["B"]), W)
    args = (I["feat"].cuda(), I["next_tok"].cuda(), I["prefix_len"].cuda(), [t.cuda() for t in ks],
            [t.cuda() for t in vs], cfg["top_k"], cfg["temperature"])
    ref = fe.fe_draft_forward(h, *args)
    out = fe.alloc_outputs(h, cfg["B"], cfg["top_k"])
    prof = fe.fe_profile_forward(h, *args, out=out)
    torch.cuda.synchronize()
    assert fe.fe_last_device_status(h) == fe.FE_OK
    for key in ref:
        assert torch.equal(ref[key], out[key]), key
    N = cfg["n_layers"]
    kinds = [k for k, _ in prof]
    assert len(prof) == fe.fe_launch_count(h, cfg["B"], False)
    # linear phases run as separate launches (2 + 4 per layer) or, at B = 1 with
    # FE_DRAFT_STACK=1, as N + 1 persistent stacks
    att = [j for j, kd in enumerate(kinds) if kd == "attention"]
    assert len(att) == N
    n_lin = kinds.count("linear")
    assert n_lin in (2 + 4 * N, N + 1)
    assert all(kinds[j - 1] == "linear" for j in att)
    if cfg["B"] > 8:  # every tensor-core phase: its operand prep right before it, except the
        # O projection, whose operand the attention kernel writes
        assert kinds.count("linear_prep") == n_lin - N
        assert all(kinds[j + 1] == "linear" for j, kd in enumerate(kinds) if kd == "linear_prep")
        assert all(kinds[j + 1] == "linear" for j in att)
    assert kinds[0] in ("linear", "linear_prep") and kinds[-1] == "lm_head"
    assert all(us > 0 for _, us in prof)
    h.close()


@pytest.mark.parametrize("spec", [dict(name="tiny"),
                                  dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1376,
                                                 vocab=5003, n_layers=3, dtype="bf16", B=2, prefix=40, top_k=8,
                                                 rope_theta=1e4, seed=41, page_size=0)),
                                  dict(name=dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1408,
                                                 vocab=5003, n_layers=3, dtype="bf16", B=12, prefix=40, top_k=8,
                                                 rope_theta=1e4, seed=42, page_size=0))])
def test_profile_graph_stamps_the_real_graph(spec):
    """fe_profile_graph runs the draft's own launch sequence (programmatic launches, in a
    CUDA graph) with GPU stamps: its outputs equal fe_draft_forward's bit for bit, it reports
    every launch plus the tree kernel in stream order, every launch is stamped, launch ends
    never go backwards (each kernel waits for its predecessor), and the added times
    partition the stamped span."""
    import paper_2509_20416_gb300 as fe
    cfg = wl.make_config(spec["name"])
    W, I = wl.make_weights(cfg), wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    B, k = cfg["B"], cfg["top_k"]
    h = fe.fe_draft_init(dict(cfg, max_batch=B), W)
    tok = I["next_tok"].cuda()
    args = (I["feat"].cuda(), tok, I["prefix_len"].cuda(), [t.cuda() for t in ks], [t.cuda() for t in vs], k,
            cfg["temperature"])
    ref = fe.fe_draft_forward(h, *args)
    ref_tree = fe.fe_build_tree(h, tok, ref["topk_id"], k)
    out = fe.alloc_outputs(h, B, k)
    tree = fe.alloc_tree(h, B, k)
    for rep in range(3):  # the cached graph is replayed after the first call
        st = fe.fe_profile_graph(h, *args, out=out, tree=tree)
        torch.cuda.synchronize()
        assert fe.fe_last_device_status(h) == fe.FE_OK
        for key in ref:
            assert torch.equal(ref[key], out[key]), key
        for key in ref_tree:
            assert torch.equal(ref_tree[key], tree[key]), key
        assert len(st) == fe.fe_launch_count(h, B, True)
        assert st[-1][0] == "tree"
        assert [kd for kd, _, _ in st[:-1]] == [kd for kd, _ in fe.fe_profile_forward(h, *args, out=out)]
        assert all(s >= 0 and e >= s for _, s, e in st)
        assert min(s for _, s, _ in st) == 0.0
        ends = [e for _, _, e in st]
        assert all(b >= a for a, b in zip(ends, ends[1:]))
        its = fe.in_step_times(st)
        assert sum(a for _, _, a in its) == pytest.approx(ends[-1] - st[0][1], rel=1e-9, abs=1e-6)
    h.close()

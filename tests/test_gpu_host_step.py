"""fe_draft_step_host: one draft step from and to host memory through the C ABI (inputs
copied in, draft and tree, outputs copied back, as one CUDA graph). Its outputs must be
bit-identical to fe_draft_forward + fe_build_tree on device buffers, which the parity
tests check against the fp64 oracle."""
import pytest
import torch

from fe_synth import workloads as wl

pytestmark = pytest.mark.gpu

CASES = {
    # B <= 8 streaming kernels, contiguous caches, greedy
    "bf16_b2_contig": (dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1376, vocab=5003, n_layers=3,
                            dtype="bf16", B=2, prefix=0, top_k=8, rope_theta=1e4, seed=61, page_size=0),
                       [37, 150], 0.0),
    # batched handle (tensor-core linear phases), paged caches, temperature-scaled probabilities
    "bf16_b12_paged": (dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1408, vocab=3001, n_layers=2,
                            dtype="bf16", B=12, prefix=0, top_k=4, rope_theta=1e4, seed=62, page_size=16),
                       [3, 0, 17, 40, 8, 1, 30, 12, 5, 60, 22, 9], 0.7),
    # fp32 storage
    "f32_b3": (dict(d=256, n_heads=4, n_kv_heads=4, head_dim=64, ffn=688, vocab=4096, n_layers=3, dtype="f32",
                    B=3, prefix=0, top_k=4, rope_theta=1e4, seed=63, page_size=0), [5, 0, 63], 0.0),
    # stochastic drafting (Sec. 2.2) through the host step: the drawn set and its ranks
    "bf16_b12_paged_sampled": (dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1408, vocab=3001, n_layers=2,
                                    dtype="bf16", B=12, prefix=0, top_k=4, rope_theta=1e4, seed=64, page_size=16),
                               [3, 0, 17, 40, 8, 1, 30, 12, 5, 60, 22, 9], 1.0, 77),
}


def _setup(spec, plist):
    import paper_2509_20416_gb300 as fe
    cfg = wl.make_config(spec, prefix_list=plist)
    W, I = wl.make_weights(cfg), wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    h = fe.fe_draft_init(dict(cfg, max_batch=cfg["B"]), W)
    if cfg["page_size"]:
        table, n_pages = wl.page_plan(cfg, I["prefix_len"])
        kd = [wl.paginate(cfg, t, table, n_pages).cuda() for t in ks]
        vd = [wl.paginate(cfg, t, table, n_pages).cuda() for t in vs]
        table = table.cuda()
    else:
        kd, vd, table, n_pages = [t.cuda() for t in ks], [t.cuda() for t in vs], None, 0
    return fe, cfg, h, I, kd, vd, table, n_pages


def _device_step(fe, cfg, h, I, kd, vd, table, n_pages, temp, B=None, seed=None):
    B = B or cfg["B"]
    feat, tok, plen = I["feat"][:B].cuda(), I["next_tok"][:B].cuda(), I["prefix_len"][:B].cuda()
    out = fe.fe_draft_forward(h, feat, tok, plen, kd, vd, cfg["top_k"], temp, page_table=table, n_pages=n_pages,
                              sample=seed is not None, seed=seed or 0)
    tree = fe.fe_build_tree(h, tok, out["topk_id"], cfg["top_k"])
    torch.cuda.synchronize()
    return {**{k: v.cpu() for k, v in out.items()}, **{"tree_" + k: v.cpu() for k, v in tree.items()}}


@pytest.mark.parametrize("case", list(CASES))
def test_host_step_matches_device_step(case):
    spec, plist, temp = CASES[case][:3]
    seed = CASES[case][3] if len(CASES[case]) > 3 else None
    fe, cfg, h, I, kd, vd, table, n_pages = _setup(spec, plist)
    ref = _device_step(fe, cfg, h, I, kd, vd, table, n_pages, temp, seed=seed)
    # pageable features go through the handle's pinned staging, page-locked ones are
    # copied from directly (a graph of its own)
    for feat in (I["feat"], I["feat"].pin_memory(), I["feat"]):
        for _ in range(2):  # the first call captures the step's graph, the second replays it
            got = fe.fe_draft_step_host(h, feat, I["next_tok"], I["prefix_len"], kd, vd, cfg["top_k"], temp,
                                        page_table=table, n_pages=n_pages, sample=seed is not None, seed=seed or 0)
            for key, want in ref.items():
                assert torch.equal(got[key], want), (case, feat.is_pinned(), key)
    assert fe.fe_last_device_status(h) == fe.FE_OK
    h.close()


def test_host_step_new_arguments_recapture():
    """A different batch size (and then the first one again) re-captures the graph."""
    spec, plist, temp = CASES["bf16_b12_paged"]
    fe, cfg, h, I, kd, vd, table, n_pages = _setup(spec, plist)
    for B in (12, 5, 12):
        ref = _device_step(fe, cfg, h, I, kd, vd, table[:B] if table is not None else None, n_pages, temp, B)
        got = fe.fe_draft_step_host(h, I["feat"][:B].contiguous(), I["next_tok"][:B].contiguous(),
                                    I["prefix_len"][:B].contiguous(), kd, vd, cfg["top_k"], temp,
                                    page_table=table[:B].contiguous() if table is not None else None,
                                    n_pages=n_pages)
        for key, want in ref.items():
            assert torch.equal(got[key], want), (B, key)
    h.close()


def test_host_step_rejects_device_tensors_and_bad_sizes():
    import paper_2509_20416_gb300 as fe
    spec, plist, temp = CASES["bf16_b2_contig"]
    fe, cfg, h, I, kd, vd, table, n_pages = _setup(spec, plist)
    with pytest.raises(ValueError):
        fe.fe_draft_step_host(h, I["feat"].cuda(), I["next_tok"], I["prefix_len"], kd, vd, cfg["top_k"])
    with pytest.raises(fe.FeError):  # top_k above the handle's maximum
        fe.fe_draft_step_host(h, I["feat"], I["next_tok"], I["prefix_len"], kd, vd, cfg["top_k_max"] + 1)
    h.close()

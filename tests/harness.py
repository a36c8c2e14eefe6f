"""Test harness: run the CUDA path (through the C ABI) and the oracle on the same
seeded inputs, and compare them under the parity contract.

Parity contract (the drafter's stated tolerances):
  bf16 storage : max |d logit| <= 3e-2 over the full vocabulary, max |d prob| <= 1e-3
  fp32 storage : relative 1e-4 (max |d| <= 1e-4 * max |ref| per tensor, elementwise on lse)
  top-k ids    : identical, except at ranks where the oracle's adjacent logit gap < 1e-2
  tree         : bit-exact against the oracle's tree rule applied to the GPU's top-k
                 (and hence against the oracle's tree whenever the top-k agree)
"""
from __future__ import annotations

import numpy as np
import torch

from fe_synth import workloads as wl

TOL_BF16_LOGIT = 3e-2
TOL_BF16_PROB = 1e-3
TOL_F32_REL = 1e-4
TIE_GAP = 1e-2


def device_caches(cfg, ks, vs, prefix_len):
    """Device K/V caches in the ABI layout (contiguous, or a paged pool + page table)."""
    if cfg["page_size"]:
        table, n_pages = wl.page_plan(cfg, prefix_len)
        kd = [wl.paginate(cfg, k, table, n_pages).cuda() for k in ks]
        vd = [wl.paginate(cfg, v, table, n_pages).cuda() for v in vs]
        return kd, vd, table.cuda(), n_pages
    return [k.cuda() for k in ks], [v.cuda() for v in vs], None, 0


def run_gpu(cfg, W, I, ks, vs, top_k=None, temperature=None, dbg=True, handle=None, sample=False, seed=0):
    import paper_2509_20416_gb300 as fe
    top_k = top_k or cfg["top_k"]
    T = cfg["temperature"] if temperature is None else temperature
    h = handle or fe.fe_draft_init(dict(cfg, max_batch=cfg["B"]), W)  # weights straight from host memory
    B, N, d, V = cfg["B"], cfg["n_layers"], cfg["d"], cfg["vocab"]
    kd, vd, table, n_pages = device_caches(cfg, ks, vs, I["prefix_len"])
    feat = I["feat"].cuda()
    tok = I["next_tok"].cuda()
    plen = I["prefix_len"].cuda()
    dl = torch.full((B, N, V), float("nan"), device="cuda") if dbg else None
    dh = torch.full((N, B, d), float("nan"), device="cuda") if dbg else None
    out = fe.fe_draft_forward(h, feat, tok, plen, kd, vd, top_k, T, page_table=table, n_pages=n_pages,
                              dbg_logits=dl, dbg_hidden=dh, sample=sample, seed=seed)
    tree = fe.fe_build_tree(h, tok, out["topk_id"], top_k)
    st = fe.fe_last_device_status(h)
    res = {k: v.cpu().numpy() for k, v in out.items()}
    res.update({"tree_" + k: v.cpu().numpy() for k, v in tree.items()})
    if dbg:
        res["logits"] = dl.cpu().numpy()
        res["hidden"] = dh.cpu().numpy()
    res["status"] = st
    res["k_cache"] = [k.cpu() for k in kd]
    res["v_cache"] = [v.cpu() for v in vd]
    res["page_table"] = None if table is None else table.cpu()
    if handle is None:
        h.close()
    return res


def run_oracle(orc, cfg, W, I, ks, vs, b, top_k=None, temperature=None):
    top_k = top_k or cfg["top_k"]
    T = cfg["temperature"] if temperature is None else temperature
    return orc.draft_seq(cfg, W, I["feat"][b].contiguous(), int(I["next_tok"][b]), int(I["prefix_len"][b]),
                         [k[b].contiguous() for k in ks], [v[b].contiguous() for v in vs], cfg["max_seq"],
                         top_k, T)


def check_topk(gpu_ids, ref_logits, k, gap=TIE_GAP):
    """gpu_ids [k] against the oracle's full logits [V] (or any values the k are the largest
    of, such as sampling keys), with the near-tie exemption at `gap`."""
    order = np.argsort(-ref_logits, kind="stable")[: k + 1]
    vals = ref_logits[order]
    assert len(set(gpu_ids.tolist())) == k, "duplicate candidates"
    for r in range(k):
        if gpu_ids[r] == order[r]:
            continue
        gaps = [vals[r - 1] - vals[r]] if r > 0 else []
        gaps.append(vals[r] - vals[r + 1] if r + 1 < len(vals) else np.inf)
        assert min(gaps) < gap, (
            f"rank {r}: gpu id {gpu_ids[r]} != oracle id {order[r]} with oracle gaps {gaps}")
        # the substitute must itself sit inside the near-tie band
        assert abs(ref_logits[gpu_ids[r]] - vals[r]) < gap, (r, ref_logits[gpu_ids[r]], vals[r])


def compare(orc, cfg, g, o, b, top_k=None):
    """GPU result g (whole batch) against oracle result o (sequence b)."""
    top_k = top_k or cfg["top_k"]
    N = cfg["n_layers"]
    stats = {}
    if cfg["dtype"] == "f32":
        for key in ("hidden", "logits"):
            if key in g:
                gv = g[key][:, b] if key == "hidden" else g[key][b]
                ref = o[key]
                err = np.abs(gv - ref).max() / np.abs(ref).max()
                stats[key + "_rel"] = err
                assert err <= TOL_F32_REL, (key, err)
        lse_err = np.abs(g["lse"][b] - o["lse"]) / np.abs(o["lse"])
        assert lse_err.max() <= TOL_F32_REL, lse_err
    else:
        if "logits" in g:
            dl = np.abs(g["logits"][b] - o["logits"]).max()
            stats["max_dlogit"] = dl
            assert dl <= TOL_BF16_LOGIT, dl
        dlse = np.abs(g["lse"][b] - o["lse"]).max()
        stats["max_dlse"] = dlse
        assert dlse <= TOL_BF16_LOGIT, dlse
    for i in range(N):
        ids = g["topk_id"][b, i]
        check_topk(ids, o["logits"][i], top_k)
        # probabilities and logits of the GPU's own candidates, against the oracle's values for them
        p_ref, _ = orc.softmax(o["logits"][i], cfg["temperature"] if cfg["temperature"] > 0 else 1.0)
        dp = np.abs(g["topk_prob"][b, i] - p_ref[ids]).max()
        dlg = np.abs(g["topk_logit"][b, i] - o["logits"][i][ids]).max()
        stats["max_dprob"] = max(stats.get("max_dprob", 0.0), dp)
        if cfg["dtype"] == "f32":
            assert dp <= TOL_F32_REL * max(1e-3, p_ref[ids].max()), dp
            assert dlg <= TOL_F32_REL * np.abs(o["logits"][i]).max(), dlg
        else:
            assert dp <= TOL_BF16_PROB, dp
            assert dlg <= TOL_BF16_LOGIT, dlg
        # the GPU's reported logits are ordered (desc logit, asc id)
        gl = g["topk_logit"][b, i]
        for r in range(top_k - 1):
            assert gl[r] > gl[r + 1] or (gl[r] == gl[r + 1] and ids[r] < ids[r + 1])
    # tree: bit-exact against the oracle's rule on the GPU's own candidates
    tok, par, dep, mask = orc.tree(N, top_k, int(g["tree_tok"][b, 0]), g["topk_id"][b])
    assert np.array_equal(g["tree_tok"][b], tok)
    assert np.array_equal(g["tree_parent"][b], par)
    assert np.array_equal(g["tree_depth"][b], dep)
    assert np.array_equal(g["tree_mask"][b], mask)
    return stats


def check_kv_append(cfg, g, I, ks, vs, b, orc_layer_inputs=None):
    """The call wrote each layer's new row into slot P_b and left rows < P_b untouched."""
    P = int(I["prefix_len"][b])
    for i in range(cfg["n_layers"]):
        if cfg["page_size"]:
            ps = cfg["page_size"]
            table = g["page_table"]
            rows = [(int(table[b, p // ps]), p % ps) for p in range(P)]
            kc = g["k_cache"][i]
            got = torch.stack([kc[pg, :, s, :] for pg, s in rows], 1) if P else None
        else:
            got = g["k_cache"][i][b, :, :P, :]
        if P:
            assert torch.equal(got, ks[i][b, :, :P, :]), f"layer {i}: prefix rows modified"

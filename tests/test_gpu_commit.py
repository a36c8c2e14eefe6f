"""The commit of accepted rows (Sec. 2.4, "Update and Iterate") through the C ABI against the
fp64 oracle: the rows written into every layer's cache, the draft that follows from the
committed caches, and a multi-cycle loop (draft, greedy verification against a synthetic
target, commit) in which both sides advance in lockstep."""
import numpy as np
import pytest
import torch

import fe_synth
from fe_synth import workloads as wl
import harness as H

pytestmark = pytest.mark.gpu


def _cache_rows(cfg, cache, table, b, rows):
    """[Hkv, len(rows), hd] of sequence b from a device-layout cache (host copy)."""
    ps = cfg["page_size"]
    if ps:
        return torch.stack([cache[int(table[b, p // ps]), :, p % ps, :] for p in rows], 1)
    return cache[b][:, list(rows), :]


def _tol(cfg):
    return (1e-4, 1e-5) if cfg["dtype"] == "f32" else (2.0 ** -6, 2.0 ** -7)


def _check_rows(cfg, got, ref):
    rtol, atol = _tol(cfg)
    g, r = got.double(), ref.double()
    assert torch.allclose(g, r, rtol=rtol, atol=atol * max(1.0, r.abs().max().item())), (g - r).abs().max()


def _feats(cfg, B, L, tid):
    f = torch.empty(B, L, 3 * cfg["d"], dtype=wl.torch_dtype(cfg))
    fe_synth.fill_normal(f, cfg["seed"], tid, 1.0)
    return f


COMMIT = {
    # tensor-core attention (bf16, hd 128, G = 4), 16-row pages, one sequence with nothing to commit
    "bf16_gqa4_hd128_paged": (dict(d=512, n_heads=4, n_kv_heads=1, head_dim=128, ffn=1376, vocab=3001,
                                   n_layers=3, dtype="bf16", B=3, prefix=0, top_k=4, rope_theta=5e5,
                                   seed=41, page_size=16, max_seq=96), [20, 0, 47], [3, 1, 0]),
    # CUDA-core attention (fp32, hd 64), contiguous caches
    "f32_hd64_contig": (dict(d=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=688, vocab=777, n_layers=2,
                             dtype="f32", B=2, prefix=0, top_k=4, rope_theta=1e4, seed=42, page_size=0,
                             max_seq=64), [5, 33], [2, 2]),
    # a batched handle (tensor-core linear): 12 x 4 rows go in blocks of 2 row indices
    "bf16_b12_blocks": (dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1408, vocab=3001, n_layers=4,
                             dtype="bf16", B=12, prefix=0, top_k=4, rope_theta=1e4, seed=43, page_size=0,
                             max_seq=80), [3, 0, 17, 40, 8, 1, 30, 12, 5, 60, 22, 9], [4, 0, 1, 2, 3, 4, 4, 1, 0, 2, 3, 4]),
}


@pytest.mark.parametrize("case", list(COMMIT))
def test_commit_parity(orc, case):
    import paper_2509_20416_gb300 as fe
    spec, P, n = COMMIT[case]
    cfg = wl.make_config(spec)
    B, N, L, cap = cfg["B"], cfg["n_layers"], max(n) if max(n) > 0 else 1, cfg["max_seq"]
    W = wl.make_weights(cfg)
    ks, vs = wl.make_caches(cfg)
    feats = _feats(cfg, B, L, 70)
    toks = torch.randint(0, cfg["vocab"], (B, L), generator=torch.Generator().manual_seed(5), dtype=torch.int32)
    Pt = torch.tensor(P, dtype=torch.int32)
    nt = torch.tensor(n, dtype=torch.int32)
    h = fe.fe_draft_init(dict(cfg, max_batch=B), W)
    kd, vd, table, n_pages = H.device_caches(cfg, ks, vs, Pt + nt)  # pages for the committed rows and one more
    fe.fe_commit(h, feats.cuda(), toks.cuda(), nt.cuda(), Pt.cuda(), kd, vd, page_table=table, n_pages=n_pages)
    assert fe.fe_last_device_status(h) == 0
    kg, vg = [k.cpu() for k in kd], [v.cpu() for v in vd]
    tab = None if table is None else table.cpu()
    ko, vo = [], []
    for b in range(B):
        kb, vb = [k[b].clone() for k in ks], [v[b].clone() for v in vs]
        orc.commit_seq(cfg, W, feats[b, :n[b]].contiguous(), toks[b, :n[b]].tolist(), P[b], kb, vb, cap)
        ko.append(kb)
        vo.append(vb)
        for l in range(N):
            for got, ref, orig in ((kg[l], kb[l], ks[l][b]), (vg[l], vb[l], vs[l][b])):
                if n[b]:
                    _check_rows(cfg, _cache_rows(cfg, got, tab, b, range(P[b], P[b] + n[b])), ref[:, P[b]:P[b] + n[b]])
                keep = list(range(P[b]))
                if keep:  # the prefix is untouched
                    assert torch.equal(_cache_rows(cfg, got, tab, b, keep), orig[:, :P[b]])
    # the draft that follows reads the committed rows
    feat2 = _feats(cfg, B, 1, 71)[:, 0].contiguous()
    tok2 = torch.randint(0, cfg["vocab"], (B,), generator=torch.Generator().manual_seed(6), dtype=torch.int32)
    P2 = Pt + nt
    out = fe.fe_draft_forward(h, feat2.cuda(), tok2.cuda(), P2.cuda(), kd, vd, cfg["top_k"], 0.0,
                              page_table=table, n_pages=n_pages,
                              dbg_logits=torch.full((B, N, cfg["vocab"]), float("nan"), device="cuda"),
                              dbg_hidden=torch.full((N, B, cfg["d"]), float("nan"), device="cuda"))
    assert fe.fe_last_device_status(h) == 0
    g = {k: v.cpu().numpy() for k, v in out.items()}
    h.close()
    for b in range(B):
        o = orc.draft_seq(cfg, W, feat2[b], int(tok2[b]), int(P2[b]), ko[b], vo[b], cap, cfg["top_k"], 0.0)
        ref_logits = o["logits"]
        for i in range(N):
            H.check_topk(g["topk_id"][b, i], ref_logits[i], cfg["top_k"])
        rtol, _ = _tol(cfg)
        assert np.allclose(g["lse"][b], o["lse"], rtol=max(rtol, 1e-4), atol=3e-2 if cfg["dtype"] != "f32" else 1e-4)


def test_commit_cycle_loop(orc):
    """Three cycles of draft -> tree -> greedy verification against a synthetic target ->
    commit of the root row's successors, with the oracle following the same tokens."""
    import paper_2509_20416_gb300 as fe
    cfg = wl.make_config(dict(d=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=688, vocab=512, n_layers=3,
                              dtype="f32", B=2, prefix=0, top_k=4, rope_theta=1e4, seed=44, page_size=0,
                              max_seq=64))
    B, N, k, cap = cfg["B"], cfg["n_layers"], cfg["top_k"], cfg["max_seq"]
    W = wl.make_weights(cfg)
    ks, vs = wl.make_caches(cfg)
    h = fe.fe_draft_init(dict(cfg, max_batch=B), W)
    kd, vd, _, _ = H.device_caches(cfg, ks, vs, None)
    ko = [[k_[b].clone() for k_ in ks] for b in range(B)]
    vo = [[v_[b].clone() for v_ in vs] for b in range(B)]
    P = [10, 3]
    rng = np.random.default_rng(9)
    feat = _feats(cfg, B, 1, 80)[:, 0].contiguous()
    tok = torch.tensor([7, 300], dtype=torch.int32)
    for cycle in range(3):
        Pt = torch.tensor(P, dtype=torch.int32)
        out = fe.fe_draft_forward(h, feat.cuda(), tok.cuda(), Pt.cuda(), kd, vd, k, 0.0,
                                  dbg_logits=torch.empty((B, N, cfg["vocab"]), device="cuda"))
        tree = fe.fe_build_tree(h, tok.cuda(), out["topk_id"], k)
        tt, tp = tree["tok"].cpu().numpy(), tree["parent"].cpu().numpy()
        T = tt.shape[1]
        tn = rng.integers(0, cfg["vocab"], (B, T)).astype(np.int32)
        for b in range(B):  # plant matches along a backbone so that paths of several lengths occur
            for a in range(1, T):
                if rng.random() < 0.7:
                    tn[b, tp[b, a]] = tt[b, a]
        ver = fe.fe_verify_greedy(h, Pt.cuda(), tree, torch.from_numpy(tn).cuda(), k)
        n_acc = ver["n_accept"].cpu().numpy()
        path = ver["path"].cpu().numpy()
        bonus = ver["bonus"].cpu().numpy()
        g_ids = out["topk_id"].cpu().numpy()
        # the accepted positions' target features (synthetic) and tokens
        cf = _feats(cfg, B, N, 90 + cycle)
        ctok = torch.zeros(B, N, dtype=torch.int32)
        for b in range(B):
            for i in range(int(n_acc[b])):
                ctok[b, i] = int(tt[b, path[b, i]])
        fe.fe_commit(h, cf.cuda(), ctok.cuda(), torch.from_numpy(n_acc).cuda(), (Pt + 1).cuda(), kd, vd)
        assert fe.fe_last_device_status(h) == 0
        for b in range(B):
            o = orc.draft_seq(cfg, W, feat[b], int(tok[b]), P[b], ko[b], vo[b], cap, k, 0.0)
            for i in range(N):
                H.check_topk(g_ids[b, i], o["logits"][i], k)
            _, opath, on, obonus = orc.accept_greedy(tt[b], tp[b], tree["depth"].cpu().numpy()[b], tn[b], P[b], N)
            assert (on, obonus) == (int(n_acc[b]), int(bonus[b])) and np.array_equal(opath, path[b])
            # the oracle's caches: the drafted row at P, then the accepted rows after it
            orc.commit_seq(cfg, W, feat[b:b + 1].contiguous(), [int(tok[b])], P[b], ko[b], vo[b], cap)
            na = int(n_acc[b])
            orc.commit_seq(cfg, W, cf[b, :na].contiguous(), ctok[b, :na].tolist(), P[b] + 1, ko[b], vo[b], cap)
            for l in range(N):
                rows = range(P[b], P[b] + 1 + na)
                _check_rows(cfg, kd[l].cpu()[b][:, list(rows)], ko[b][l][:, P[b]:P[b] + 1 + na])
                _check_rows(cfg, vd[l].cpu()[b][:, list(rows)], vo[b][l][:, P[b]:P[b] + 1 + na])
            P[b] += 1 + na
        # the next cycle starts from the target's bonus token and the last accepted position's features
        tok = torch.from_numpy(bonus.astype(np.int32))
        feat = _feats(cfg, B, 1, 100 + cycle)[:, 0].contiguous()
    h.close()


def test_commit_rejects_bad_arguments():
    import paper_2509_20416_gb300 as fe
    cfg = wl.make_config(dict(d=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=512, vocab=1000, n_layers=2,
                              dtype="bf16", B=2, prefix=0, top_k=4, rope_theta=1e4, seed=45, page_size=0,
                              max_seq=32))
    W = wl.make_weights(cfg)
    ks, vs = wl.make_caches(cfg)
    h = fe.fe_draft_init(dict(cfg, max_batch=2), W)
    kd, vd, _, _ = H.device_caches(cfg, ks, vs, None)
    f = torch.zeros(2, 3, 3 * cfg["d"], dtype=torch.bfloat16, device="cuda")
    t = torch.zeros(2, 3, dtype=torch.int32, device="cuda")
    n = torch.zeros(2, dtype=torch.int32, device="cuda")
    with pytest.raises(fe.FeError) as e:  # L > n_layers
        fe.fe_commit(h, f, t, n, n, kd, vd)
    assert e.value.code == fe.FE_ERR_INVALID_ARG
    with pytest.raises(fe.FeError) as e:  # a missing layer cache
        fe.fe_commit(h, f[:, :2].contiguous(), t[:, :2].contiguous(), n, n, kd[:1] + [None], vd)
    assert e.value.code == fe.FE_ERR_INVALID_ARG
    # capacity: prefix_len + n_rows > max_seq is reported by the device
    P = torch.tensor([cfg["max_seq"] - 1, 0], dtype=torch.int32, device="cuda")
    n2 = torch.tensor([2, 0], dtype=torch.int32, device="cuda")
    fe.fe_commit(h, f[:, :2].contiguous(), t[:, :2].contiguous(), n2, P, kd, vd)
    assert fe.fe_last_device_status(h) == fe.FE_ERR_CAPACITY
    h.close()

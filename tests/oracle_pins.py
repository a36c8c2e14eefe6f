"""Pins of the fp64 oracle: checks against what the paper and mathematics fix.

Each ``pin_*`` takes an ``oracle.Oracle`` and raises AssertionError when the oracle
disagrees with a closed form, a brute-force sum, a library special case, an invariant
or the hand-worked tree fixtures under tests/golden/. ``test_oracle_pins.py`` runs them
on the real oracle; ``test_oracle_mutants.py`` runs them on builds with one planted
mistake each and requires every mutant to fail at least one pin.
"""
from __future__ import annotations

import json
import math
import os
from fractions import Fraction

import numpy as np
import torch

import fe_synth
from fe_synth import workloads as wl

import torch_ref

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bfloat16 bit patterns (uint16), round to nearest even."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def _bf16_value(b: np.ndarray) -> np.ndarray:
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


# ---- linear algebra -------------------------------------------------------------------

def pin_matvec_bruteforce(orc):
    """y = W x on a non-square matrix against an exact rational sum (both storage types)."""
    rng = np.random.default_rng(11)
    W = rng.standard_normal((5, 7)).astype(np.float32)
    x = rng.standard_normal(7)
    exact = [sum(Fraction(float(W[m, k])) * Fraction(float(x[k])) for k in range(7))
             for m in range(5)]
    y = orc.matvec(W, x)
    for m in range(5):
        assert abs(y[m] - float(exact[m])) <= 1e-13 * (1 + abs(float(exact[m]))), (m, y[m])
    Wb = _bf16_bits(W)
    Wv = _bf16_value(Wb)
    exact = [sum(Fraction(float(Wv[m, k])) * Fraction(float(x[k])) for k in range(7))
             for m in range(5)]
    y = orc.matvec(Wb, x)
    for m in range(5):
        assert abs(y[m] - float(exact[m])) <= 1e-13 * (1 + abs(float(exact[m])))


def pin_rmsnorm(orc):
    n = 12
    # constant vector: mean(x^2) = c^2, so y = gamma c / sqrt(c^2 + eps); eps matters at c=1e-3
    c, eps = 1e-3, 1e-5
    gamma = np.linspace(0.5, 2.0, n).astype(np.float32)
    y = orc.rmsnorm(np.full(n, c), gamma, eps)
    want = gamma.astype(np.float64) * c / math.sqrt(c * c + eps)
    assert np.allclose(y, want, rtol=1e-13, atol=0)
    # unit gain, eps = 0: the output has root-mean-square exactly 1 and is scale invariant
    rng = np.random.default_rng(3)
    x = rng.standard_normal(n) * 7.0
    y = orc.rmsnorm(x, np.ones(n, np.float32), 0.0)
    assert abs(math.sqrt(np.mean(y * y)) - 1.0) < 1e-14
    y2 = orc.rmsnorm(x * 1e3, np.ones(n, np.float32), 0.0)
    assert np.allclose(y, y2, rtol=1e-13)


# ---- RoPE -----------------------------------------------------------------------------

def pin_rope(orc):
    hd, theta = 8, 10000.0
    half = hd // 2
    rng = np.random.default_rng(5)
    v = rng.standard_normal(hd)
    assert np.allclose(orc.rope(v, 0.0, theta), v, rtol=0, atol=0)  # position 0: identity
    for m in (1.0, 3.0, 17.0):
        for j in range(half):
            w = m * theta ** (-2.0 * j / hd)
            e = np.zeros(hd)
            e[j] = 1.0
            r = orc.rope(e, m, theta)
            want = np.zeros(hd)
            want[j], want[j + half] = math.cos(w), math.sin(w)
            assert np.allclose(r, want, atol=1e-15), (m, j, r)
            e = np.zeros(hd)
            e[j + half] = 1.0
            r = orc.rope(e, m, theta)
            want = np.zeros(hd)
            want[j], want[j + half] = -math.sin(w), math.cos(w)
            assert np.allclose(r, want, atol=1e-15), (m, j, r)
    # norm preservation and dependence on the relative position only
    q, k = rng.standard_normal(hd), rng.standard_normal(hd)
    assert abs(np.linalg.norm(orc.rope(q, 9.0, theta)) - np.linalg.norm(q)) < 1e-13
    a = orc.rope(q, 5.0, theta) @ orc.rope(k, 2.0, theta)
    b = orc.rope(q, 105.0, theta) @ orc.rope(k, 102.0, theta)
    assert abs(a - b) < 1e-12
    # the complex-rotation form
    want = torch_ref.rope_complex(torch.tensor(q), 7.0, theta).numpy()
    assert np.allclose(orc.rope(q, 7.0, theta), want, atol=1e-14)


# ---- attention ------------------------------------------------------------------------

def _kv(rng, Hkv, cap, hd):
    return (rng.standard_normal((Hkv, cap, hd)).astype(np.float32),
            rng.standard_normal((Hkv, cap, hd)).astype(np.float32))


def pin_attention(orc):
    rng = np.random.default_rng(7)
    H, Hkv, hd, cap = 4, 2, 8, 10
    kc, vc = _kv(rng, Hkv, cap, hd)
    q = rng.standard_normal((H, hd))
    kn, vn = rng.standard_normal((Hkv, hd)), rng.standard_normal((Hkv, hd))
    # P = 0: the only key is the row's own; output = own value of the head's group
    o = orc.attention(q, kc, vc, 0, kn, vn)
    for h in range(H):
        assert np.allclose(o[h], vn[h * Hkv // H], atol=1e-15)
    # all keys equal: uniform weights, output = mean of the P + 1 values
    P = 6
    kc_eq = np.repeat(kn.astype(np.float32)[:, None, :], cap, axis=1)
    kn_eq = kc_eq[:, 0, :].astype(np.float64)
    o = orc.attention(q, kc_eq, vc, P, kn_eq, vn)
    for h in range(H):
        g = h * Hkv // H
        mean = (vc[g, :P].astype(np.float64).sum(0) + vn[g]) / (P + 1)
        assert np.allclose(o[h], mean, atol=1e-13)
    # two keys, closed form of the scaled softmax
    q1 = np.zeros((1, 4)); q1[0, 0] = 1.0
    kc1 = np.zeros((1, 2, 4), np.float32); kc1[0, 0, 0] = 2.0
    vc1 = np.zeros((1, 2, 4), np.float32); vc1[0, 0, 1] = 1.0
    kn1 = np.zeros((1, 4)); kn1[0, 0] = -1.0
    vn1 = np.zeros((1, 4)); vn1[0, 2] = 1.0
    o = orc.attention(q1, kc1, vc1, 1, kn1, vn1)
    s0, s1 = 2.0 / 2.0, -1.0 / 2.0  # q.k / sqrt(4)
    w0 = math.exp(s0) / (math.exp(s0) + math.exp(s1))
    assert np.allclose(o[0], [0.0, w0, 1.0 - w0, 0.0], atol=1e-15)
    # grouped-query attention equals MHA over replicated KV heads
    rep = H // Hkv
    kc_r = np.repeat(kc, rep, axis=0)
    vc_r = np.repeat(vc, rep, axis=0)
    o_gqa = orc.attention(q, kc, vc, P, kn, vn)
    o_mha = orc.attention(q, kc_r, vc_r, P, np.repeat(kn, rep, 0), np.repeat(vn, rep, 0))
    assert np.allclose(o_gqa, o_mha, atol=1e-14)
    # library special case: torch scaled_dot_product_attention in fp64
    keys = torch.cat([torch.tensor(kc_r[:, :P], dtype=torch.float64),
                      torch.tensor(np.repeat(kn, rep, 0))[:, None]], 1)
    vals = torch.cat([torch.tensor(vc_r[:, :P], dtype=torch.float64),
                      torch.tensor(np.repeat(vn, rep, 0))[:, None]], 1)
    ref = torch.nn.functional.scaled_dot_product_attention(torch.tensor(q)[:, None], keys, vals)
    assert np.allclose(o_gqa, ref[:, 0].numpy(), atol=1e-13)


def pin_silu_mul(orc):
    g = np.array([0.0, 1.0, -2.0, 30.0])
    u = np.array([5.0, 2.0, 3.0, 0.5])
    y = orc.silu_mul(g, u)
    want = [0.0, 2.0 / (1.0 + math.exp(-1.0)), -6.0 / (1.0 + math.exp(2.0)),
            15.0 / (1.0 + math.exp(-30.0))]
    assert np.allclose(y, want, rtol=1e-15, atol=0)


# ---- softmax, top-k, tree ---------------------------------------------------------------

def pin_softmax(orc):
    p, lse = orc.softmax(np.log([1.0, 2.0, 3.0]))
    assert np.allclose(p, [1 / 6, 2 / 6, 3 / 6], rtol=1e-14) and abs(lse - math.log(6)) < 1e-14
    p, lse = orc.softmax(np.log([1.0, 2.0, 3.0]), T=2.0)  # p ~ sqrt of the weights
    s = 1 + math.sqrt(2) + math.sqrt(3)
    assert np.allclose(p, [1 / s, math.sqrt(2) / s, math.sqrt(3) / s], rtol=1e-14)
    assert abs(lse - math.log(s)) < 1e-14
    p0, _ = orc.softmax(np.log([1.0, 2.0, 3.0]), T=0.0)  # greedy: the T = 1 distribution
    assert np.allclose(p0, [1 / 6, 2 / 6, 3 / 6], rtol=1e-14)
    rng = np.random.default_rng(9)
    lg = rng.standard_normal(5000) * 4 + 600.0  # large offset: needs the max shift
    p, lse = orc.softmax(lg)
    assert abs(p.sum() - 1.0) < 1e-12
    m = lg.max()
    assert abs(lse - (m + math.log(math.fsum(math.exp(v - m) for v in lg)))) < 1e-10


def pin_topk(orc):
    rng = np.random.default_rng(2)
    lg = np.round(rng.standard_normal(300) * 3, 1)  # many exact ties
    for k in (1, 5, 17, 300):
        want = np.argsort(-lg, kind="stable")[:k]
        assert np.array_equal(orc.topk(lg, k), want), k


def pin_topk_sample(orc):
    """Stochastic drafting (Sec. 2.2 "sample k candidates", read as k draws without
    replacement by the Gumbel-top-k trick): the counter-based
    deviates, the law of the draws without replacement, and the order the tree uses."""
    # SplitMix64 seeded with 0: its first outputs as published (Steele et al. 2014)
    for n, want in enumerate([0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F], start=1):
        assert orc.splitmix64(0, n) == want
        u = orc.uniform(0, n)
        assert u == ((want >> 41) + 0.5) / 2 ** 23 and float(np.float32(u)) == u  # exact in float32
    us = [orc.uniform(12345, n) for n in range(1, 20001)]
    assert 0.0 < min(us) and max(us) < 1.0 and abs(np.mean(us) - 0.5) < 0.01

    # the law of two draws without replacement from q = softmax(l / T), brute force over all
    # 20 ordered pairs of a 5-token vocabulary: P(a, then b) = q_a q_b / (1 - q_a)
    lg = np.array([0.3, -1.2, 1.0, 0.0, 0.7])
    R = 200_000
    for T in (1.0, 0.5):
        q = np.exp(lg / T - np.max(lg / T))
        q /= q.sum()
        ids, drawn = orc.topk_sample(np.tile(lg, (R, 1)), 2, T, seed=99)
        counts = np.zeros((5, 5))
        np.add.at(counts, (drawn[:, 0], drawn[:, 1]), 1)
        for a in range(5):
            for b in range(5):
                p = 0.0 if a == b else q[a] * q[b] / (1 - q[a])
                tol = 5 * math.sqrt(p * (1 - p) / R) + 1e-4
                assert abs(counts[a, b] / R - p) <= tol, (T, a, b, counts[a, b] / R, p)
    # the first draw of a larger vocabulary follows q itself
    rng = np.random.default_rng(3)
    lg = rng.standard_normal(40)
    q = np.exp(lg - lg.max())
    q /= q.sum()
    _, drawn = orc.topk_sample(np.tile(lg, (R, 1)), 3, 1.0, seed=5)
    freq = np.bincount(drawn[:, 0], minlength=40) / R
    assert np.all(np.abs(freq - q) <= 5 * np.sqrt(q * (1 - q) / R) + 1e-4)
    assert all(len(set(r)) == 3 for r in drawn[:1000])  # without replacement

    # row r of a batch draws with counter row0 + r, as a single-row call with that counter
    lg = rng.standard_normal((6, 50))
    ids_b, drawn_b = orc.topk_sample(lg, 4, 0.8, seed=7, row0=11)
    for r in range(6):
        ids_1, drawn_1 = orc.topk_sample(lg[r], 4, 0.8, seed=7, row0=11 + r)
        assert np.array_equal(ids_b[r], ids_1) and np.array_equal(drawn_b[r], drawn_1)

    # the tree's order: the drawn set by descending logit, ties to the smaller id, so rank 0
    # is the most probable candidate (the backbone)
    lg = np.array([1.0, 1.0, 1.0, 1.0, 0.0, 0.0, 2.0])
    ids, drawn = orc.topk_sample(np.tile(lg, (500, 1)), 4, 1.0, seed=3)
    for i, d in zip(ids, drawn):
        assert sorted(i) == sorted(d)
        assert list(i) == sorted(d, key=lambda v: (-lg[v], v))
    # k = V: every token, in the stable descending-logit order
    ids, _ = orc.topk_sample(lg, 7, 1.0, seed=4)
    assert np.array_equal(ids, np.argsort(-lg, kind="stable"))
    # T -> 0: the draws become the greedy top-k (the Gumbel deviates are bounded by the
    # uniforms on the 2^-24 grid: |G| < 17, far below the logit gaps / T)
    lg = rng.permutation(np.arange(30) * 1e-3)
    for seed in range(5):
        ids, drawn = orc.topk_sample(lg, 5, 1e-9, seed=seed)
        assert np.array_equal(ids, orc.topk(lg, 5)) and np.array_equal(drawn, orc.topk(lg, 5))


def _check_tree_invariants(N, k, root, topk, tok, par, dep, mask):
    T = 1 + N * k
    assert tok.shape == (T,) and mask.shape == (T, T)
    assert tok[0] == root and par[0] == -1 and dep[0] == 0
    assert dep.max() == N and (dep <= N).all()
    for n in range(1, T):
        assert 0 <= par[n] < n and dep[n] == dep[par[n]] + 1
    # level i holds q_{t+i}'s candidates in rank order
    for i in range(1, N + 1):
        assert list(tok[1 + (i - 1) * k: 1 + i * k]) == list(topk[i - 1])
    # exactly one backbone chain of length N made of rank-0 nodes; side branches are leaves
    backbone = [0] + [1 + (i - 1) * k for i in range(1, N + 1)]
    for a, b in zip(backbone, backbone[1:]):
        assert par[b] == a
    has_child = set(int(p) for p in par[1:])
    assert has_child == set(backbone[:-1])
    for i in range(1, N + 1):  # at most k - 1 side branches per level
        assert sum(1 for n in range(T) if dep[n] == i and n not in backbone) == k - 1
    # mask: ancestor-or-self, lower-triangular, popcount = depth + 1
    assert (np.triu(mask, 1) == 0).all() and (np.diag(mask) == 1).all()
    for a in range(T):
        anc = {a}
        c = par[a]
        while c >= 0:
            anc.add(int(c))
            c = par[c]
        assert set(np.nonzero(mask[a])[0].tolist()) == anc
        assert mask[a].sum() == dep[a] + 1
    if k == 1:
        assert list(par) == list(range(-1, T - 1))


def pin_tree(orc):
    for name in ("tree_backbone_n3_k3.json", "tree_chain_n4_k1.json"):
        with open(os.path.join(GOLDEN, name)) as f:
            G = json.load(f)
        tok, par, dep, mask = orc.tree(G["N"], G["k"], G["root"], np.array(G["topk"]))
        assert tok.tolist() == G["tok"], name
        assert par.tolist() == G["parent"], name
        assert dep.tolist() == G["depth"], name
        assert ["".join(str(int(b)) for b in row) for row in mask] == G["mask"], name
    rng = np.random.default_rng(4)
    for N, k in ((1, 1), (1, 5), (5, 1), (4, 3), (8, 10)):
        topk = rng.integers(0, 1000, size=(N, k)).astype(np.int32)
        out = orc.tree(N, k, 77, topk)
        _check_tree_invariants(N, k, 77, topk, *out)


# ---- the whole cascade -------------------------------------------------------------------

def mini_cfg(**kw):
    base = dict(d=16, n_heads=4, n_kv_heads=2, head_dim=4, ffn=24, vocab=40, n_layers=3,
                dtype="f32", B=2, prefix=3, top_k=5, rope_theta=100.0, seed=21, page_size=0,
                max_seq=8)
    base.update(kw)
    return wl.make_config(base)


def _mini_problem(cfg):
    W = wl.make_weights(cfg)
    # non-trivial gains so a norm with a wrong gain index would show
    for L in W["layers"]:
        for key in ("attn_norm", "mlp_norm"):
            t = torch.empty(cfg["d"], dtype=wl.torch_dtype(cfg))
            fe_synth.fill_normal(t, cfg["seed"], 900 + len(key), 0.3)
            L[key] = (t.float() + 1.0).to(t.dtype)
    t = torch.empty(cfg["d"], dtype=wl.torch_dtype(cfg))
    fe_synth.fill_normal(t, cfg["seed"], 950, 0.3)
    W["final_norm"] = (t.float() + 1.0).to(t.dtype)
    # larger weights than 0.02 so every block moves the hidden state visibly
    scale = 0.4
    for key in ("w_fuse", "w_in", "embed", "lm_head"):
        W[key] = (W[key].float() * (scale / 0.02)).to(W[key].dtype)
    for L in W["layers"]:
        for key in ("w_qkv", "w_o", "w_gate", "w_up", "w_down"):
            L[key] = (L[key].float() * (scale / 0.02)).to(L[key].dtype)
    I = wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    return W, I, ks, vs


def _draft_both(orc, cfg, W, I, ks, vs, b, **kw):
    P = int(I["prefix_len"][b])
    kcs = [k[b].contiguous() for k in ks]
    vcs = [v[b].contiguous() for v in vs]
    o = orc.draft_seq(cfg, W, I["feat"][b].contiguous(), int(I["next_tok"][b]), P, kcs, vcs,
                      cfg["max_seq"], cfg["top_k"], cfg["temperature"], **kw)
    r = torch_ref.draft(cfg, W, I["feat"][b], int(I["next_tok"][b]), P, kcs, vcs, cfg["top_k"],
                        cfg["temperature"], kw.get("rope_layer_offset", 0))
    return o, r


def _agree(o, r, tol=1e-10):
    for key in ("hidden", "logits", "lse"):
        a, b = o[key], r[key].numpy()
        assert np.allclose(a, b, rtol=tol, atol=tol * max(1.0, np.abs(b).max())), key
    # probabilities of the chosen candidates, and the candidates themselves
    p = r["prob"].numpy()
    for i in range(o["topk_id"].shape[0]):
        assert np.array_equal(o["topk_id"][i], r["topk_id"][i].numpy())
        assert np.allclose(o["topk_prob"][i], p[i][o["topk_id"][i]], rtol=tol, atol=1e-15)
        assert np.allclose(o["topk_logit"][i], o["logits"][i][o["topk_id"][i]], rtol=0, atol=0)


def _handworked_layer2(x0_or_h1):
    """Layer 2 of the hand-worked draft, in the closed form derived in the fixture. Its
    input normalises to u = (0.2, 1.4) under both readings, so the attention output is
    the same; the residual base is h1 (the cascade) or x0 (the parallel ablation)."""
    c, s = math.cos(1.0), math.sin(1.0)
    s_c = (0.2 * c - 1.4 * s) / math.sqrt(2.0)
    w_c = 1.0 / (1.0 + math.exp(math.sqrt(2.0) - s_c))
    o = (w_c * -1.0 + (1 - w_c) * 7.0, w_c * 3.0 + (1 - w_c) * 1.0)
    x = (x0_or_h1[0] + o[0], x0_or_h1[1] + o[1])
    r = math.sqrt((x[0] ** 2 + x[1] ** 2) / 2)
    u2 = (x[0] / r, x[1] / r)
    silu = u2[0] / (1.0 + math.exp(-u2[0]))
    h2 = (x[0], x[1] + silu * u2[1])
    rz = math.sqrt((h2[0] ** 2 + h2[1] ** 2) / 2)
    z2 = (2 * h2[0] / rz, h2[1] / rz)
    return np.array(h2), np.array([5 * z2[0], 5 * z2[1], 5 * (z2[0] + z2[1])])


def pin_draft_handworked(orc):
    """The whole draft on a 2-wide, two-layer model worked by hand
    (tests/golden/draft_handworked_n2_k2.json): Eq. 1's fusion and concat order, the
    attention over the cached row and the row's own key (scale, RoPE at position P), the
    residuals, SwiGLU's gate/up order, the final norm's gain, the LM head, top-k, the tree,
    and the parallel ablation's residual base."""
    g = json.load(open(os.path.join(GOLDEN, "draft_handworked_n2_k2.json")))
    cfg = dict(g["cfg"], parallel_layers=0)
    f32 = lambda a: torch.tensor(a, dtype=torch.float32)
    W = dict(w_fuse=f32(g["w_fuse"]), w_in=f32(g["w_in"]), embed=f32(g["embed"]), lm_head=f32(g["lm_head"]),
             final_norm=f32(g["final_norm"]),
             layers=[{k: f32(v) for k, v in L.items() if not k.endswith("row0")} for L in g["layers"]])
    kcs, vcs = [], []
    for L in g["layers"]:
        kc, vc = torch.zeros((1, 2, 2)), torch.zeros((1, 2, 2))
        kc[0, 0], vc[0, 0] = f32(L["k_cache_row0"]), f32(L["v_cache_row0"])
        kcs.append(kc)
        vcs.append(vc)
    feat = f32(g["feat"])
    h2, lg2 = _handworked_layer2(g["h1"])
    for par in (0, 1):
        cfg["parallel_layers"] = par
        o = orc.draft_seq(cfg, W, feat, g["tok"], g["P"], kcs, vcs, 2, 2)
        assert np.allclose(o["hidden"][0], g["h1"], rtol=1e-13, atol=1e-13), par
        assert np.allclose(o["logits"][0], g["logits1"], rtol=1e-13, atol=1e-13), par
        assert o["topk_id"][0].tolist() == g["topk1"]
        assert abs(o["lse"][0] - math.log(math.exp(2) + math.exp(7) + math.exp(9))) < 1e-12
        want_h2, want_lg2 = (h2, lg2) if par == 0 else _handworked_layer2((1.0, 7.0))
        assert np.allclose(o["hidden"][1], want_h2, rtol=1e-12, atol=1e-12), (par, o["hidden"][1], want_h2)
        assert np.allclose(o["logits"][1], want_lg2, rtol=1e-12, atol=1e-12), (par, o["logits"][1], want_lg2)
        if par == 0:
            assert o["topk_id"][1].tolist() == g["topk2"]
            tok, parent, depth, _ = orc.tree(2, 2, g["tok"], o["topk_id"])
            assert (tok.tolist(), parent.tolist(), depth.tolist()) == (g["tree_tok"], g["tree_parent"],
                                                                       g["tree_depth"])


def pin_draft_n1(orc):
    """N = 1: the drafter is a single EAGLE-style decoder layer plus the LM head."""
    for dtype in ("f32", "bf16"):
        cfg = mini_cfg(n_layers=1, dtype=dtype)
        W, I, ks, vs = _mini_problem(cfg)
        for b in range(cfg["B"]):
            o, r = _draft_both(orc, cfg, W, I, ks, vs, b)
            _agree(o, r)


def pin_cascade(orc):
    """N = 3 with grouped-query heads: h_i = L_i(h_{i-1}) (Eq. 2), T = 1 and T = 0.7."""
    for T in (0.0, 0.7):
        cfg = mini_cfg(temperature=T)
        W, I, ks, vs = _mini_problem(cfg)
        o, r = _draft_both(orc, cfg, W, I, ks, vs, 1)
        _agree(o, r)
    cfg = mini_cfg(n_layers=2, rope_layer_offset=1)
    W, I, ks, vs = _mini_problem(cfg)
    o, r = _draft_both(orc, cfg, W, I, ks, vs, 0, rope_layer_offset=1)
    _agree(o, r)


def pin_truncation(orc):
    """Layers 1..j of an N-layer cascade equal a j-layer cascade with the same first j layers."""
    cfg = mini_cfg(n_layers=4, B=1)
    W, I, ks, vs = _mini_problem(cfg)
    o4 = orc.draft_seq(cfg, W, I["feat"][0].contiguous(), int(I["next_tok"][0]), 3,
                       [k[0].contiguous() for k in ks], [v[0].contiguous() for v in vs],
                       cfg["max_seq"], cfg["top_k"])
    cfg2 = dict(cfg, n_layers=2)
    W2 = dict(W, layers=W["layers"][:2])
    o2 = orc.draft_seq(cfg2, W2, I["feat"][0].contiguous(), int(I["next_tok"][0]), 3,
                       [k[0].contiguous() for k in ks[:2]], [v[0].contiguous() for v in vs[:2]],
                       cfg["max_seq"], cfg["top_k"])
    for key in ("hidden", "logits", "lse", "topk_id"):
        assert np.array_equal(o4[key][:2], o2[key]), key


def pin_parallel_layers(orc):
    """The parallel ablation (Sec. 3.2, Table 2: every L_i consumes x0): layer i's output
    equals a one-layer cascade built from L_i alone (same features, token, position and
    layer-i cache), and differs from the cascade's h_i beyond the first layer."""
    cfg = mini_cfg(n_layers=3, B=1)
    W, I, ks, vs = _mini_problem(cfg)
    feat, tok = I["feat"][0].contiguous(), int(I["next_tok"][0])
    kb = [k[0].contiguous() for k in ks]
    vb = [v[0].contiguous() for v in vs]
    par = orc.draft_seq(dict(cfg, parallel_layers=1), W, feat, tok, 3, kb, vb, cfg["max_seq"], cfg["top_k"])
    cas = orc.draft_seq(cfg, W, feat, tok, 3, kb, vb, cfg["max_seq"], cfg["top_k"])
    for i in range(cfg["n_layers"]):
        one = orc.draft_seq(dict(cfg, n_layers=1), dict(W, layers=[W["layers"][i]]), feat, tok, 3, [kb[i]],
                            [vb[i]], cfg["max_seq"], cfg["top_k"])
        for key in ("hidden", "logits", "lse", "topk_id"):
            assert np.array_equal(par[key][i], one[key][0]), (i, key)
    assert np.array_equal(par["hidden"][0], cas["hidden"][0])
    assert np.abs(par["hidden"][1:] - cas["hidden"][1:]).max() > 1e-3


def pin_accept_greedy(orc):
    """Tree positions and the greedy acceptance walk (Sec. 2.4): hand-worked cases on a
    Backbone Expansion tree, and brute force over every root-to-node path of random trees
    (the walk must end at the deepest node whose whole path matches the target)."""
    g = json.load(open(os.path.join(GOLDEN, "accept_greedy_n3_k3.json")))
    for case in g["cases"]:
        pos, path, n, bonus = orc.accept_greedy(g["tok"], g["parent"], g["depth"], case["target_next"], g["P"],
                                                g["N"])
        assert pos.tolist() == g["pos"], case["why"]
        assert (n, path.tolist(), bonus) == (case["n"], case["path"], case["bonus"]), case["why"]
    rng = np.random.default_rng(5)
    for trial in range(200):
        N, k, V = int(rng.integers(1, 6)), int(rng.integers(1, 5)), 12
        topk = np.stack([rng.permutation(V)[:k] for _ in range(N)]).astype(np.int32)
        tok, par, dep, _ = orc.tree(N, k, int(rng.integers(0, V)), topk)
        T = len(tok)
        tn = rng.integers(0, V, T).astype(np.int32)
        for a in range(1, T):  # plant matches so that walks of every length occur
            if rng.random() < 0.6:
                tn[par[a]] = tok[a]
        pos, path, n, bonus = orc.accept_greedy(tok, par, dep, tn, 7, N)
        assert np.array_equal(pos, 7 + dep)

        def ok(a):  # every edge on a's root path carries the target's token
            while par[a] >= 0:
                if tok[a] != tn[par[a]]:
                    return False
                a = par[a]
            return True
        best = max((a for a in range(T) if ok(a)), key=lambda a: (dep[a], -a))
        assert n == dep[best] and bonus == tn[best]
        chain, a = [], best
        while par[a] >= 0:
            chain.append(a)
            a = par[a]
        assert path[:n].tolist() == chain[::-1] and (path[n:] == -1).all()


def _sampled_trees(orc, N, k, V, drafter_logits, R, seed):
    """R Backbone Expansion trees whose levels are drawn by orc.topk_sample (T = 1):
    returns tok, parent, depth, rank [R, T] and the tree order ids [R, N, k]."""
    lg = np.tile(np.asarray(drafter_logits), (R, 1))  # row r * N + i: depth i + 1 of trial r
    ids, drawn = orc.topk_sample(lg, k, 1.0, seed=seed)
    ids, drawn = ids.reshape(R, N, k), drawn.reshape(R, N, k)
    T = 1 + N * k
    tok = np.zeros((R, T), np.int32)
    tok[:, 1:] = ids.reshape(R, N * k)
    par = np.array([-1] + [0 if i == 0 else 1 + (i - 1) * k for i in range(N) for _ in range(k)], np.int32)
    dep = np.array([0] + [i + 1 for i in range(N) for _ in range(k)], np.int32)
    rank = np.zeros((R, T), np.int32)
    rank[:, 1:] = np.argmax(ids[:, :, :, None] == drawn[:, :, None, :], axis=3).reshape(R, N * k)
    return tok, np.tile(par, (R, 1)), np.tile(dep, (R, 1)), rank, ids


def pin_accept_sampled(orc):
    """Lossless verification of a sampled tree (Sec. 2.4, read as recursive rejection
    sampling over the children in draw order): with a one-hot
    target it is the greedy walk; with the target equal to the drafter it accepts the first
    draw; and every emitted token has the target's law (Monte Carlo on a 4-token vocabulary,
    5 sigma), which a wrong test ratio, residual, proposal update or test order breaks."""
    rng = np.random.default_rng(21)
    sm = lambda x: np.exp(x - x.max(-1, keepdims=True)) / np.exp(x - x.max(-1, keepdims=True)).sum(-1, keepdims=True)
    # (a) one-hot targets reduce the walk to or_accept_greedy, for any proposal and test order
    for N, k in ((1, 1), (2, 3), (3, 2), (4, 4), (5, 1)):
        B, V, T = 40, 12, 1 + N * k
        topk = np.stack([np.stack([rng.permutation(V)[:k] for _ in range(N)]) for _ in range(B)]).astype(np.int32)
        trees = [orc.tree(N, k, int(rng.integers(0, V)), topk[b]) for b in range(B)]
        tok, par, dep = (np.stack([t[j] for t in trees]) for j in range(3))
        rank = np.zeros((B, T), np.int32)
        for b in range(B):
            for i in range(N):
                rank[b, 1 + i * k:1 + (i + 1) * k] = rng.permutation(k)
        tn = rng.integers(0, V, (B, T)).astype(np.int32)
        for b in range(B):
            for a in range(1, T):
                if rng.random() < 0.6:
                    tn[b, par[b, a]] = tok[b, a]
        p = np.zeros((B, T, V))
        np.put_along_axis(p, tn[:, :, None], 1.0, axis=2)
        q = sm(rng.standard_normal((B, N, V)) * 2)
        path, n, bonus = orc.accept_sampled(tok, par, dep, rank, q, p, rng.random((B, T)), rng.random((B, T)))
        for b in range(B):
            _, gpath, gn, gbonus = orc.accept_greedy(tok[b], par[b], dep[b], tn[b], 0, N)
            assert (n[b], path[b].tolist(), bonus[b]) == (gn, gpath.tolist(), gbonus), (N, k, b)
    # (b) target = drafter at every node with children: the first-drawn child is accepted
    N, k, V, R = 3, 3, 9, 300
    lg = rng.standard_normal((N, V))
    tok, par, dep, rank, ids = _sampled_trees(orc, N, k, V, lg, R, seed=8)
    q = np.tile(sm(lg), (R, 1, 1))
    p = np.zeros((R, 1 + N * k, V))
    p[:, 0] = q[:, 0]
    p[:, 1:1 + (N - 1) * k] = np.repeat(q[:, 1:], k, axis=1)
    p[:, 1 + (N - 1) * k:] = 1.0 / V
    path, n, _ = orc.accept_sampled(tok, par, dep, rank, q, p, rng.random((R, 1 + N * k)),
                                    rng.random((R, 1 + N * k)))
    for r in range(R):
        for j in range(n[r]):
            assert rank[r, path[r, j]] == 0
        assert n[r] >= 1
    # (c) the law of the emitted tokens equals the target's, token by token
    N, k, V, R = 2, 2, 4, 400_000
    lg = np.array([[2.0, 0.5, 0.0, -1.0], [-0.5, 1.5, 0.0, 1.0]])  # the drafter's depth-1 and depth-2 logits
    q = sm(lg)
    p_root = np.array([0.1, 0.2, 0.6, 0.1])
    p_a = sm(rng.standard_normal((V, V)) * 1.5)        # after token a
    p_ab = sm(rng.standard_normal((V, V, V)) * 1.5)    # after tokens a, b
    tok, par, dep, rank, ids = _sampled_trees(orc, N, k, V, lg, R, seed=77)
    P = np.zeros((R, 1 + N * k, V))
    P[:, 0] = p_root
    P[:, 1:1 + k] = p_a[tok[:, 1:1 + k]]
    P[:, 1 + k:] = p_ab[tok[:, 1][:, None], tok[:, 1 + k:]]  # level 2 hangs under the level-1 backbone
    path, n, bonus = orc.accept_sampled(tok, par, dep, rank, np.tile(q, (R, 1, 1)), P, rng.random((R, 1 + N * k)),
                                        rng.random((R, 1 + N * k)))
    rows = np.arange(R)
    emitted = np.full((R, N + 1), -1)
    for j in range(N):
        emitted[:, j] = np.where(n > j, tok[rows, np.maximum(path[:, j], 0)], -1)
    emitted[rows, n] = bonus

    def law(sel, want, what):
        cnt = int(sel.sum())
        if cnt < 2000:
            return
        freq = np.bincount(emitted[sel, len(what)], minlength=V) / cnt
        tol = 5 * np.sqrt(want * (1 - want) / cnt) + 1e-4
        assert np.all(np.abs(freq - want) <= tol), (what, freq, want)
    law(np.ones(R, bool), p_root, ())
    for a in range(V):
        law((n >= 1) & (emitted[:, 0] == a), p_a[a], (a,))
        for b in range(V):
            law((n >= 2) & (emitted[:, 0] == a) & (emitted[:, 1] == b), p_ab[a, b], (a, b))


def pin_loss(orc):
    """The training objective of Sec. 2.3 (Eq. 3-6): Smooth L1 closed forms, a two-layer,
    three-token example worked by hand, and the reductions of the cross-entropy to a library
    log-sum-exp (one-hot teacher) and to the entropy (teacher = drafter)."""
    # Eq. 6
    for x, want in ((0.0, 0.0), (0.5, 0.125), (-0.5, 0.125), (2.0, 1.5), (-3.0, 2.5), (1.0, 0.5), (-1.0, 0.5)):
        assert abs(orc.smooth_l1(x) - want) < 1e-15, x
    assert abs(orc.smooth_l1(1 - 1e-9) - orc.smooth_l1(1 + 1e-9)) < 1e-8  # continuous at |x| = 1
    # worked by hand: layer 1 uniform q over 3 tokens, one-hot p -> log 3; h - f = (0.5, 2) ->
    # 0.125 + 1.5. Layer 2 logits (0, ln 3, 0) -> q = (1/5, 3/5, 1/5), p = (0, 1/2, 1/2) ->
    # -(ln(3/5) + ln(1/5)) / 2 = ln(25/3) / 2; h - f = (-3, 0.75) -> 2.5 + 0.28125.
    # w = (0.9, 1) for N = 2 (w_i = 0.9^(N - i)), alpha 0.1, beta 1.
    logits = np.array([[0.0, 0.0, 0.0], [0.0, math.log(3.0), 0.0]])
    teacher = np.array([[1.0, 0.0, 0.0], [0.0, 0.5, 0.5]])
    hidden = np.array([[0.5, 2.0], [-3.0, 1.0]])
    feat = np.array([[0.0, 0.0], [0.0, 0.25]])
    ce_want = [math.log(3.0), 0.5 * math.log(25.0 / 3.0)]
    fl_want = [1.625, 2.78125]
    tot_want = 0.9 * (0.1 * ce_want[0] + fl_want[0]) + 1.0 * (0.1 * ce_want[1] + fl_want[1])
    tot, ce, fl = orc.loss(logits, teacher, hidden, feat)
    assert np.allclose(ce, ce_want, rtol=1e-14, atol=1e-14) and np.allclose(fl, fl_want, rtol=0, atol=1e-15)
    assert abs(tot - tot_want) < 1e-13
    # reductions to library routines, random data
    rng = np.random.default_rng(3)
    N, V, d = 4, 50, 16
    lg = rng.normal(0, 2, (N, V))
    lse = np.log(np.exp(lg - lg.max(1, keepdims=True)).sum(1)) + lg.max(1)
    y = rng.integers(0, V, N)
    onehot = np.zeros((N, V))
    onehot[np.arange(N), y] = 1.0
    z = np.zeros((N, d))
    tot, ce, fl = orc.loss(lg, onehot, z, z, alpha=1.0, beta=1.0, decay=1.0)
    assert np.allclose(ce, lse - lg[np.arange(N), y], rtol=1e-12) and abs(tot - ce.sum()) < 1e-10
    q = torch.softmax(torch.tensor(lg), dim=1).numpy()
    tot, ce, fl = orc.loss(lg, q, z, z)
    assert np.allclose(ce, -(q * np.log(q)).sum(1), rtol=1e-12)
    # the weights follow the depth: only the last layer carries weight 1
    tot, ce, fl = orc.loss(lg, onehot, z, z, alpha=1.0, beta=0.0, decay=0.5)
    assert abs(tot - sum(0.5 ** (N - 1 - i) * ce[i] for i in range(N))) < 1e-12


def pin_zero_blocks(orc):
    """W_o = W_down = 0: every layer passes x0 through, so all N distributions coincide."""
    cfg = mini_cfg(n_layers=3, B=1)
    W, I, ks, vs = _mini_problem(cfg)
    for L in W["layers"]:
        L["w_o"] = torch.zeros_like(L["w_o"])
        L["w_down"] = torch.zeros_like(L["w_down"])
    o = orc.draft_seq(cfg, W, I["feat"][0].contiguous(), int(I["next_tok"][0]), 3,
                      [k[0].contiguous() for k in ks], [v[0].contiguous() for v in vs],
                      cfg["max_seq"], cfg["top_k"])
    f = I["feat"][0].double()
    x0 = W["w_in"].double() @ torch.cat([W["w_fuse"].double() @ f,
                                         W["embed"].double()[int(I["next_tok"][0])]])
    for i in range(3):
        assert np.allclose(o["hidden"][i], x0.numpy(), rtol=1e-13, atol=1e-13)
        assert np.array_equal(o["topk_id"][i], o["topk_id"][0])
        assert np.array_equal(o["logits"][i], o["logits"][0])
    tok, par, dep, mask = orc.tree(3, cfg["top_k"], 1, o["topk_id"])
    k = cfg["top_k"]
    for i in range(1, 3):
        assert list(tok[1 + i * k: 1 + (i + 1) * k]) == list(tok[1:1 + k])


def pin_commit(orc):
    """The commit of accepted rows (Sec. 2.4, "Update and Iterate"): against the torch
    reference (each row through Eq. 1 and the cascade, its keys and values stored before
    the next row runs); one commit of n rows equals n commits of one row; rows other than
    P .. P + n - 1 stay untouched; a row does not depend on the rows after it; n = 0 is a
    no-op; bfloat16 storage rounds to the nearest value."""
    cfg = mini_cfg(n_layers=3, B=1, max_seq=12)
    W, I, ks, vs = _mini_problem(cfg)
    N, d, cap, P, n = cfg["n_layers"], cfg["d"], cfg["max_seq"], 3, 4
    feats = torch.empty(n, 3 * d, dtype=torch.float32)
    fe_synth.fill_normal(feats, 31, 1, 1.0)
    toks = [5, 0, cfg["vocab"] - 1, 17]
    base_k = [k[0].clone() for k in ks]
    base_v = [v[0].clone() for v in vs]

    def run(feat_rows, tok_rows, P0, kc, vc):
        orc.commit_seq(cfg, W, feat_rows.contiguous(), tok_rows, P0, kc, vc, cap)

    ko, vo = [t.clone() for t in base_k], [t.clone() for t in base_v]
    run(feats, toks, P, ko, vo)
    kr, vr = [t.clone() for t in base_k], [t.clone() for t in base_v]
    torch_ref.commit(cfg, W, feats, toks, P, kr, vr)
    for l in range(N):
        for a, b, base in ((ko[l], kr[l], base_k[l]), (vo[l], vr[l], base_v[l])):
            rows = slice(P, P + n)
            assert torch.allclose(a[:, rows], b[:, rows], rtol=1e-6, atol=1e-6), l
            assert torch.equal(a[:, :P], base[:, :P]) and torch.equal(a[:, P + n:], base[:, P + n:]), l
            assert not torch.equal(a[:, rows], base[:, rows])
    # n commits of one row each
    k1, v1 = [t.clone() for t in base_k], [t.clone() for t in base_v]
    for i in range(n):
        run(feats[i:i + 1], toks[i:i + 1], P + i, k1, v1)
    assert all(torch.equal(a, b) for a, b in zip(k1 + v1, ko + vo))
    # causality: changing the last row leaves the earlier rows as they were
    k2, v2 = [t.clone() for t in base_k], [t.clone() for t in base_v]
    run(feats, toks[:-1] + [toks[-1] + 1], P, k2, v2)
    for l in range(N):
        assert torch.equal(k2[l][:, :P + n - 1], ko[l][:, :P + n - 1])
        assert not torch.equal(k2[l][:, P + n - 1], ko[l][:, P + n - 1])
    # nothing to commit
    k3, v3 = [t.clone() for t in base_k], [t.clone() for t in base_v]
    run(feats[:0], [], P, k3, v3)
    assert all(torch.equal(a, b) for a, b in zip(k3 + v3, base_k + base_v))
    # bfloat16 caches: the stored value is the nearest bfloat16 of the exact one
    cb = mini_cfg(n_layers=2, B=1, max_seq=12, dtype="bf16")
    Wb, Ib, ksb, vsb = _mini_problem(cb)
    kb, vb = [k[0].clone() for k in ksb], [v[0].clone() for v in vsb]
    fb = feats[:2].to(torch.bfloat16)
    orc.commit_seq(cb, Wb, fb.contiguous(), toks[:2], P, kb, vb, cap)
    kx, vx = [k[0].clone().double() for k in ksb], [v[0].clone().double() for v in vsb]
    torch_ref.commit(cb, Wb, fb, toks[:1], P, kx, vx)  # the first row, exact (float64)
    for l in range(2):
        for a, x in ((kb[l], kx[l]), (vb[l], vx[l])):
            got = a[:, P].double()
            ex = x[:, P]
            ulp = torch.exp2(torch.floor(torch.log2(ex.abs().clamp_min(1e-30))) - 7)
            assert ((got - ex).abs() <= 0.5 * ulp * (1 + 1e-12) + 1e-300).all(), l


ALL_PINS = [pin_commit, pin_loss, pin_accept_greedy, pin_parallel_layers, pin_matvec_bruteforce, pin_rmsnorm, pin_rope, pin_attention, pin_silu_mul,
            pin_softmax, pin_topk, pin_topk_sample, pin_accept_sampled, pin_tree, pin_draft_handworked, pin_draft_n1, pin_cascade, pin_truncation,
            pin_zero_blocks]

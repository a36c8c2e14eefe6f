"""The seeded generator: published SplitMix64 outputs, a pure-Python re-derivation,
and the moments of its normal deviates (CPU only)."""
import struct

import pytest

import numpy as np
import torch

import fe_synth
from fe_synth import workloads as wl

M64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15


def sm64(z):
    z = (z + GAMMA) & M64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & M64
    return z ^ (z >> 31)


def test_splitmix64_published_sequence():
    # the first three outputs of SplitMix64 seeded with 0 (Steele et al. 2014 reference code)
    want = [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]
    got = [fe_synth.splitmix64((i * GAMMA) & M64) for i in range(3)]
    assert got == want


def test_normal_matches_python_rederivation():
    seed, tid, n = 5, 1234, 64
    t = torch.empty(n, dtype=torch.float32)
    fe_synth.fill_normal(t, seed, tid, 0.02)
    key = sm64(sm64(seed) ^ sm64(tid ^ 0x5851F42D4C957F2D))
    for i in range(n):
        s = 0
        for j in range(3):
            w = sm64((key + 3 * i + j) & M64)
            s += sum((w >> (16 * q)) & 0xFFFF for q in range(4))
        v = struct.unpack("f", struct.pack("f", ((s - 393210) / 65536.0) * 0.02))[0]
        assert t[i].item() == v
    b = torch.empty(n, dtype=torch.bfloat16)
    fe_synth.fill_normal(b, seed, tid, 0.02)
    assert torch.equal(b, t.to(torch.bfloat16))  # torch's float->bf16 rounding is RNE too


def test_normal_moments():
    t = torch.empty(1 << 20, dtype=torch.float32)
    fe_synth.fill_normal(t, 0, 77, 1.0)
    x = t.double().numpy()
    assert abs(x.mean()) < 5e-3 and abs(x.var() - 1.0) < 5e-3
    assert np.abs(x).max() <= 6.0


def test_uniform_and_permutation():
    t = torch.empty(10000, dtype=torch.int32)
    fe_synth.fill_uniform_int(t, 7, 3, 256, 4096)
    assert int(t.min()) >= 256 and int(t.max()) <= 4096
    p = torch.empty(1000, dtype=torch.int32)
    fe_synth.permutation(p, 7, 8)
    assert sorted(p.tolist()) == list(range(1000))


def test_page_plan_covers_every_row():
    cfg = wl.make_config("b32_l31", B=4, prefix=(3, 40), max_seq=48)
    plen = wl.make_inputs(cfg)["prefix_len"]
    table, n_pages = wl.page_plan(cfg, plen)
    used = table[table >= 0].tolist()
    assert sorted(used) == list(range(n_pages))
    for b in range(cfg["B"]):
        need = (int(plen[b]) + 1 + 15) // 16
        assert (table[b, :need] >= 0).all() and (table[b, need:] < 0).all()


@pytest.mark.parametrize("ps", [8, 16, 24])
def test_paginate_places_every_row_at_its_page_and_slot(ps):
    """Row p of sequence b lands at pool[table[b, p // ps], :, p % ps]: the addressing the
    paged attention uses, for page sizes that do and do not divide the chunk length."""
    cfg = wl.make_config("tiny", B=3, prefix=0, page_size=ps, max_seq=70)
    plen = torch.tensor([0, 23, 69], dtype=torch.int32)
    table, n_pages = wl.page_plan(cfg, plen)
    g = torch.Generator().manual_seed(1)
    logical = torch.randn((3, 2, 70, 8), generator=g)
    pool = wl.paginate(cfg, logical, table, n_pages)
    assert pool.shape == (n_pages, 2, ps, 8)
    for b in range(3):
        for p in range(int(plen[b]) + 1):
            assert torch.equal(pool[int(table[b, p // ps]), :, p % ps], logical[b, :, p])


def _weight_numel(W):
    """Elements of every weight tensor make_weights builds, by name (embedding separately)."""
    mats = [W["w_fuse"], W["w_in"], W["lm_head"], W["final_norm"]]
    for L in W["layers"]:
        mats += [L[n] for n in ("attn_norm", "w_qkv", "w_o", "mlp_norm", "w_gate", "w_up", "w_down")]
    return sum(t.numel() for t in mats), W["embed"].shape, W["w_fuse"].element_size()


@pytest.mark.parametrize("name", ["tiny", "vic13b", "l31_8b", "l33_70b", "b32_l31"])
def test_roofline_bytes_and_flops_count_the_generated_tensors(monkeypatch, name):
    """The bytes and flops the roofline divides by equal a count over the tensors the
    generator actually builds (shapes only: meta tensors, so full-size workloads cost
    nothing): every weight once, the gathered embedding rows, the features, and each
    layer's K/V prefix read plus the new row; flops = 2 per weight element per row (the
    LM head for all N rows) + 4·H·hd per key."""
    monkeypatch.setattr(wl, "_normal", lambda shape, seed, tid, std, dt: torch.empty(shape, dtype=dt, device="meta"))
    cfg = wl.make_config(name)
    W = wl.make_weights(cfg)
    n_w, emb_shape, es = _weight_numel(W)
    V, d = emb_shape
    B, N, Hkv, hd, H = cfg["B"], cfg["n_layers"], cfg["n_kv_heads"], cfg["head_dim"], cfg["n_heads"]
    plen = wl.make_inputs(cfg)["prefix_len"].tolist() if name == "b32_l31" else [cfg["prefix"]] * B
    kv_elems = N * sum(p + 1 for p in plen) * 2 * Hkv * hd
    want = (n_w + B * d + B * 3 * d + kv_elems) * es
    assert wl.algorithmic_bytes(cfg, plen) == want
    parts = wl.kernel_bytes(cfg, plen)
    assert sum(parts.values()) == want
    assert parts["attention"] == kv_elems * es and parts["lm_head"] == (V * d + d) * es
    # matrices only (norm gains are not multiplied), per row; the LM head over all N rows
    mats = [W["w_fuse"], W["w_in"]] + [L[n] for L in W["layers"] for n in ("w_qkv", "w_o", "w_gate", "w_up", "w_down")]
    flops = 2 * sum(t.numel() for t in mats) * B + 2 * W["lm_head"].numel() * N * B
    flops += N * sum(4 * H * hd * (p + 1) for p in plen)
    assert wl.algorithmic_flops(cfg, plen) == flops
    fparts = wl.kernel_flops(cfg, plen)
    assert sum(fparts.values()) == flops
    assert fparts["lm_head"] == 2 * W["lm_head"].numel() * N * B
    assert fparts["attention"] == N * sum(4 * H * hd * (p + 1) for p in plen)

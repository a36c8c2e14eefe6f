"""The seeded generator: published SplitMix64 outputs, a pure-Python re-derivation,
and the moments of its normal deviates (CPU only)."""
import struct

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

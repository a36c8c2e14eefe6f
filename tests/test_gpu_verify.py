"""fe_verify_greedy: tree positions and the greedy acceptance walk (Sec. 2.4), against the
hand-worked golden cases and the oracle, bit for bit."""
import json
import os

import numpy as np
import pytest
import torch

from fe_synth import workloads as wl

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


@pytest.fixture(scope="module")
def handle():
    import paper_2509_20416_gb300 as fe
    cfg = wl.make_config("tiny", B=32)  # N = 3 layers
    h = fe.fe_draft_init(dict(cfg, max_batch=32), wl.make_weights(cfg))
    yield fe, h
    h.close()


def test_verify_golden(handle):
    fe, h = handle
    g = json.load(open(os.path.join(GOLDEN, "accept_greedy_n3_k3.json")))
    N, k = g["N"], g["k"]
    topk = torch.tensor(g["tok"][1:], dtype=torch.int32).view(1, N, k).cuda()
    tok = torch.tensor([g["tok"][0]], dtype=torch.int32).cuda()
    tree = fe.fe_build_tree(h, tok, topk, k)
    plen = torch.tensor([g["P"]], dtype=torch.int32).cuda()
    for case in g["cases"]:
        tn = torch.tensor([case["target_next"]], dtype=torch.int32).cuda()
        out = fe.fe_verify_greedy(h, plen, tree, tn, k)
        torch.cuda.synchronize()
        assert out["pos_ids"][0].tolist() == g["pos"], case["why"]
        assert int(out["n_accept"][0]) == case["n"], case["why"]
        assert out["path"][0].tolist() == case["path"], case["why"]
        assert int(out["bonus"][0]) == case["bonus"], case["why"]
    assert fe.fe_last_device_status(h) == fe.FE_OK


@pytest.mark.parametrize("k", [1, 3, 8])
def test_verify_matches_oracle(orc, handle, k):
    fe, h = handle
    B, N, V = 32, 3, 4096
    rng = np.random.default_rng(100 + k)
    topk = np.stack([np.stack([rng.permutation(64)[:k] for _ in range(N)]) for _ in range(B)]).astype(np.int32)
    root = rng.integers(0, V, B).astype(np.int32)
    tree = fe.fe_build_tree(h, torch.from_numpy(root).cuda(), torch.from_numpy(topk).cuda(), k)
    T = 1 + N * k
    tn = rng.integers(0, 64, (B, T)).astype(np.int32)
    tok, par, dep = (tree[n].cpu().numpy() for n in ("tok", "parent", "depth"))
    for b in range(B):  # plant a matching path of random length, ending on or off the backbone
        L = int(rng.integers(0, N + 1))
        cur = 0
        for lev in range(1, L + 1):
            r = 0 if lev < L else int(rng.integers(0, k))
            child = 1 + (lev - 1) * k + r
            tn[b, cur] = tok[b, child]
            cur = child
    plen = rng.integers(0, 4000, B).astype(np.int32)
    out = fe.fe_verify_greedy(h, torch.from_numpy(plen).cuda(), tree, torch.from_numpy(tn).cuda(), k)
    torch.cuda.synchronize()
    lengths = set()
    for b in range(B):
        pos, path, n, bonus = orc.accept_greedy(tok[b], par[b], dep[b], tn[b], int(plen[b]), N)
        assert np.array_equal(out["pos_ids"][b].cpu().numpy(), pos)
        assert np.array_equal(out["path"][b].cpu().numpy(), path)
        assert int(out["n_accept"][b]) == n and int(out["bonus"][b]) == bonus
        lengths.add(n)
    assert len(lengths) > 1

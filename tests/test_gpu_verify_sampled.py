"""fe_verify_sampled: lossless verification of a sampled draft tree (Sec. 2.4; recursive
rejection sampling over each node's children in draw order) against the oracle's
or_accept_sampled on the same float32 inputs.

Trees: k candidates per depth drawn without replacement from q = softmax(logit / T) by the
oracle's sampler (or_topk_sample), arranged by fe_build_tree, with their draw ranks; logits
~ N(0, 3^2) so that q and the target's distributions p (the next depth's logits plus noise)
hold probabilities well above rounding; and, end to end, a sampled GPU draft's own tree, ranks
and q. Deviates are seeded float32 values, exact in both precisions.

The GPU walks in float32 elementwise (with its sums in double), the oracle in float64, so a
decision the two may take differently is one within the float32 walk's rounding. The bound:
a rejection pass computes r - s and its clamp in float32, at most 5 roundings of total mass
one (r, s and the difference each sum to at most 1); the error mass a residual carries is
divided by the normaliser Z it is rescaled with, so after passes with normalisers Z_1..Z_j
it is S_j = S_(j-1) / Z_(j-1) + 5 ulps (S_0 = 0 for a target distribution itself), and a
decision or the bonus CDF is off by at most E = (2 S_j / Z_j + 5) ulps (ulp = 2^-24: the 1 / Z
rescale doubles S, and u s(x) adds three roundings). The oracle reports each sequence's
closest decision in units of E (or_accept_sampled's margin): the smallest |u s(x) - r(x)|
over its tests and the distance of u_bonus to its pick's CDF edges. Sequences with a margin
below 1 are exempt and counted (they must be few, and still valid walks); all others must
match exactly. The one-hot-target special case must reduce exactly to fe_verify_greedy.
"""
import numpy as np
import pytest
import torch

from fe_synth import workloads as wl

pytestmark = pytest.mark.gpu

EPS = 1.0  # margins are in units of the float32 walk's error bound

# (B, N, k, V, T, seed, noise sigma of the target's logits)
SYNTH = {
    "v5003_n3_k8": (24, 3, 8, 5003, 1.0, 31, 0.7),
    "v5003_n3_k8_T07": (24, 3, 8, 5003, 0.7, 32, 1.5),
    "v4096_n6_k1": (16, 6, 1, 4096, 1.0, 33, 0.5),
    "v3001_n5_k16": (8, 5, 16, 3001, 1.0, 34, 0.7),
    "v2048_n4_k32": (4, 4, 32, 2048, 1.0, 35, 1.0),
    "v128256_n3_k8": (4, 3, 8, 128256, 1.0, 36, 0.7),
}


def _uniforms(shape, gen):
    """float32 deviates (m + 1/2) / 2^23 in (0, 1), exact in both precisions."""
    m = torch.randint(0, 2 ** 23, shape, generator=gen, dtype=torch.int64)
    return ((m.double() + 0.5) / 2 ** 23).float()


def _handle(N, V, k, B):
    import paper_2509_20416_gb300 as fe
    cfg = wl.make_config(dict(d=128, n_heads=2, n_kv_heads=2, head_dim=64, ffn=128, vocab=V, n_layers=N,
                              dtype="f32", B=B, prefix=4, top_k=k, rope_theta=1e4, seed=1, page_size=0))
    return fe, fe.fe_draft_init(dict(cfg, max_batch=B, top_k_max=max(k, 16)), wl.make_weights(cfg))


def _targets(logits_next, dep, sigma, T, gen):
    """p[b, c] = softmax((logits of depth min(depth(c), N - 1) + noise) / T)."""
    B, N, V = logits_next.shape
    nxt = torch.clamp(dep, max=N - 1).long()
    base = logits_next[torch.arange(B)[:, None], nxt]
    return torch.softmax((base + torch.randn(base.shape, generator=gen) * sigma) / T, dim=-1).float().contiguous()


def _node_rank(topk_rank):
    rk = topk_rank.cpu().numpy().reshape(topk_rank.shape[0], -1)
    return np.concatenate([np.zeros((rk.shape[0], 1), np.int32), rk], axis=1)  # the root's entry is unused


def _check_walk(path, n, bonus, par, N, V):
    assert 0 <= n <= N and 0 <= bonus < V
    prev = 0
    for j in range(N):
        if j < n:
            assert par[path[j]] == prev
            prev = path[j]
        else:
            assert path[j] == -1


def _compare(orc, fe, h, tree, topk_rank, q, p, u_acc, u_bonus, k, N, V, label, max_exempt):
    got = fe.fe_verify_sampled(h, tree, topk_rank, q, p.cuda(), u_acc.cuda(), u_bonus.cuda(), k)
    torch.cuda.synchronize()
    assert fe.fe_last_device_status(h) == fe.FE_OK
    g_path, g_n, g_bonus = (got[x].cpu().numpy() for x in ("path", "n_accept", "bonus"))
    tok, par, dp = (tree[x].cpu().numpy() for x in ("tok", "parent", "depth"))
    path, n, bonus, margin = orc.accept_sampled(tok, par, dp, _node_rank(topk_rank), q.cpu().double().numpy(),
                                                p.double().numpy(), u_acc.double().numpy(),
                                                u_bonus.double().numpy(), want_margin=True)
    B = tok.shape[0]
    exempt, accepted = 0, 0
    for b in range(B):
        _check_walk(g_path[b], int(g_n[b]), int(g_bonus[b]), par[b], N, V)
        if margin[b] < EPS:
            exempt += 1
            continue
        assert np.array_equal(g_path[b], path[b]), (label, b, g_path[b], path[b], margin[b])
        assert int(g_n[b]) == int(n[b]), (label, b)
        assert int(g_bonus[b]) == int(bonus[b]), (label, b, int(g_bonus[b]), int(bonus[b]), margin[b])
        accepted += int(n[b])
    print(label, f"exempt {exempt}/{B}", f"accepted tokens {accepted}", f"min margin {margin.min():.2e}")
    assert exempt <= max_exempt, (label, exempt)
    return accepted


@pytest.mark.parametrize("case", list(SYNTH))
def test_sampled_verification_matches_oracle(orc, case):
    B, N, k, V, T, seed, sigma = SYNTH[case]
    fe, h = _handle(N, V, k, B)
    gen = torch.Generator().manual_seed(seed)
    logits = torch.randn((B, N, V), generator=gen, dtype=torch.float64) * 3.0
    ids, drawn = orc.topk_sample(logits.reshape(B * N, V).numpy(), k, T, seed)
    ids, drawn = ids.reshape(B, N, k), drawn.reshape(B, N, k)
    # each candidate's position in draw order
    rank = np.array([[[list(drawn[b, i]).index(x) for x in ids[b, i]] for i in range(N)] for b in range(B)],
                    np.int32)
    root = torch.randint(0, V, (B,), generator=gen, dtype=torch.int32)
    tree = fe.fe_build_tree(h, root.cuda(), torch.from_numpy(ids).int().cuda(), k)
    q = torch.softmax(logits / T, dim=-1).float().contiguous()
    dep = tree["depth"].cpu()
    p = _targets(logits.float(), dep, sigma, T, gen)
    Tn = 1 + N * k
    u_acc, u_bonus = _uniforms((B, Tn), gen), _uniforms((B, Tn), gen)
    acc = _compare(orc, fe, h, tree, torch.from_numpy(rank).cuda(), q.cuda(), p, u_acc, u_bonus, k, N, V, case,
                   max(1, B // 8))
    assert acc > 0 or k == 1
    h.close()


def test_sampled_draft_then_verification_end_to_end(orc):
    """A sampled GPU draft (T = 0.25, so q is not flat) feeds its own tree, draw ranks and
    q = softmax(logits / T) to fe_verify_sampled."""
    import paper_2509_20416_gb300 as fe
    T = 0.25
    cfg = wl.make_config(dict(d=512, n_heads=8, n_kv_heads=2, head_dim=64, ffn=1376, vocab=5003, n_layers=3,
                              dtype="bf16", B=24, prefix=0, top_k=8, rope_theta=1e4, seed=3, page_size=0),
                         temperature=T, prefix_list=[(29 * b + 3) % 70 for b in range(24)])
    W, I = wl.make_weights(cfg), wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    h = fe.fe_draft_init(dict(cfg, max_batch=cfg["B"]), W)
    B, N, V, k = cfg["B"], cfg["n_layers"], cfg["vocab"], cfg["top_k"]
    logits = torch.empty((B, N, V), device="cuda")
    tok = I["next_tok"].cuda()
    out = fe.fe_draft_forward(h, I["feat"].cuda(), tok, I["prefix_len"].cuda(), [t.cuda() for t in ks],
                              [t.cuda() for t in vs], k, T, dbg_logits=logits, sample=True, seed=17)
    tree = fe.fe_build_tree(h, tok, out["topk_id"], k)
    q = torch.softmax(logits / T, dim=-1).contiguous()
    gen = torch.Generator().manual_seed(1017)
    p = _targets(logits.cpu(), tree["depth"].cpu(), 0.5, T, gen)
    Tn = 1 + N * k
    u_acc, u_bonus = _uniforms((B, Tn), gen), _uniforms((B, Tn), gen)
    _compare(orc, fe, h, tree, out["topk_rank"], q, p, u_acc, u_bonus, k, N, V, "draft_T025", max(1, B // 8))
    h.close()


def test_one_hot_targets_reduce_to_the_greedy_walk():
    """With every target distribution one-hot at a token, the sampled walk is the greedy one
    (fe_verify_greedy with that token as the target's next), for any proposal and draw order:
    the child holding the token passes its test (r = 1), the others fail (r = 0), the
    residual stays one-hot, and the bonus is the token."""
    fe, h, cfg, out, tree, q = _small_draft(24, 3, 8, 5003, 1.0, 17)
    B, N, V, k = cfg["B"], cfg["n_layers"], cfg["vocab"], cfg["top_k"]
    Tn = 1 + N * k
    gen = torch.Generator().manual_seed(77)
    tok = tree["tok"].cpu()
    par = tree["parent"].cpu()
    # the target's token after node c: one of c's children's tokens (3 in 4) or a random one
    tn = torch.randint(0, V, (B, Tn), generator=gen, dtype=torch.int32)
    for b in range(B):
        for c in range(Tn):
            kids = [x for x in range(1, Tn) if int(par[b, x]) == c]
            if kids and torch.rand(1, generator=gen).item() < 0.75:
                tn[b, c] = tok[b, kids[int(torch.randint(0, len(kids), (1,), generator=gen))]]
    p = torch.zeros((B, Tn, V))
    p.scatter_(2, tn.long().unsqueeze(-1), 1.0)
    u_acc, u_bonus = _uniforms((B, Tn), gen), _uniforms((B, Tn), gen)
    got = fe.fe_verify_sampled(h, tree, out["topk_rank"], q, p.cuda(), u_acc.cuda(), u_bonus.cuda(), k)
    plen = torch.zeros(B, dtype=torch.int32).cuda()
    want = fe.fe_verify_greedy(h, plen, tree, tn.cuda(), k)
    torch.cuda.synchronize()
    for key in ("path", "n_accept", "bonus"):
        assert torch.equal(got[key], want[key]), key
    assert int(want["n_accept"].sum()) > 0
    h.close()


def test_sampled_verification_is_repeatable():
    """The same inputs give the same bits (the residual buffer's old contents do not leak)."""
    fe, h, cfg, out, tree, q = _small_draft(8, 5, 16, 3001, 1.0, 20)
    B, N, V, k = cfg["B"], cfg["n_layers"], cfg["vocab"], cfg["top_k"]
    Tn = 1 + N * k
    gen = torch.Generator().manual_seed(5)
    p = torch.softmax(torch.randn((B, Tn, V), generator=gen), dim=-1).cuda()
    u_acc, u_bonus = _uniforms((B, Tn), gen).cuda(), _uniforms((B, Tn), gen).cuda()
    a = fe.fe_verify_sampled(h, tree, out["topk_rank"], q, p, u_acc, u_bonus, k)
    a = {x: y.clone() for x, y in a.items()}
    b = fe.fe_verify_sampled(h, tree, out["topk_rank"], q, p, u_acc, u_bonus, k)
    torch.cuda.synchronize()
    for key in a:
        assert torch.equal(a[key], b[key]), key
    h.close()


def _small_draft(B, N, k, V, T, seed):
    """A sampled GPU draft of a small bf16 drafter: handle, config, outputs, tree, q."""
    import paper_2509_20416_gb300 as fe
    cfg = wl.make_config(dict(d=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=704, vocab=V, n_layers=N,
                              dtype="bf16", B=B, prefix=0, top_k=k, rope_theta=1e4, seed=seed, page_size=0),
                         temperature=T, prefix_list=[(29 * b + 3) % 70 for b in range(B)])
    W, I = wl.make_weights(cfg), wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    h = fe.fe_draft_init(dict(cfg, max_batch=B), W)
    logits = torch.empty((B, N, V), device="cuda")
    tok = I["next_tok"].cuda()
    out = fe.fe_draft_forward(h, I["feat"].cuda(), tok, I["prefix_len"].cuda(), [t.cuda() for t in ks],
                              [t.cuda() for t in vs], k, T, dbg_logits=logits, sample=True, seed=seed)
    tree = fe.fe_build_tree(h, tok, out["topk_id"], k)
    q = torch.softmax(logits / T, dim=-1).contiguous()
    torch.cuda.synchronize()
    assert fe.fe_last_device_status(h) == fe.FE_OK
    return fe, h, cfg, out, tree, q

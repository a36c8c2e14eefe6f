"""Named workload shapes and the synthetic-input recipe.

The five named workloads are drafters shaped like the paper's targets (Vicuna-13B and
LLaMA-3.x, Sec. 3 "Setup"; the 70B and batched-serving shapes follow Table 1 and
Table 3). There are no trained weights or benchmark prompts here, so every tensor is
drawn from the seeded generator:

  features concat(l, m, h)   [B, 3d]       ~ N(0, 1)
  all weight matrices, embed                ~ N(0, 0.02^2)
  RMSNorm gains                             = 1
  prefix K/V caches (post-RoPE)             ~ N(0, 1)
  next token ids                            uniform in [0, V)
  prefix lengths                            fixed P, or uniform in [lo, hi] per sequence
  page assignment (paged caches)            a seeded permutation of the page pool

Weight layout (canonical, row-major [out, in], y = W x):
  w_fuse [d, 3d], w_in [d, 2d], embed [V, d], lm_head [V, d], final_norm [d];
  per layer: attn_norm [d], w_qkv [(H + 2 Hkv) hd, d] (q rows, then k rows, then v rows),
  w_o [d, H hd], mlp_norm [d], w_gate [F, d], w_up [F, d], w_down [d, F].
Logical cache layout (per layer): [B, Hkv, cap, hd]; the paged device layout is built
from it by ``paginate``.
"""
from __future__ import annotations

import copy


import torch

from . import fill_normal, fill_uniform_int, permutation

WORKLOADS = {
    # fp32, L2-resident; the oracle finishes it in well under a second
    "tiny": dict(d=256, n_heads=4, n_kv_heads=4, head_dim=64, ffn=688, vocab=4096, n_layers=3,
                 dtype="f32", B=1, prefix=64, top_k=4, rope_theta=1e4, seed=0, page_size=0),
    # Vicuna-13B-shaped drafter (MHA)
    "vic13b": dict(d=5120, n_heads=40, n_kv_heads=40, head_dim=128, ffn=13824, vocab=32000,
                   n_layers=5, dtype="bf16", B=1, prefix=512, top_k=8, rope_theta=1e4, seed=0,
                   page_size=0),
    # LLaMA-3.1-8B-shaped drafter (GQA 32/8)
    "l31_8b": dict(d=4096, n_heads=32, n_kv_heads=8, head_dim=128, ffn=14336, vocab=128256,
                   n_layers=6, dtype="bf16", B=1, prefix=1024, top_k=8, rope_theta=5e5, seed=0,
                   page_size=0),
    # LLaMA-3.3-70B-shaped drafter (GQA 64/8)
    "l33_70b": dict(d=8192, n_heads=64, n_kv_heads=8, head_dim=128, ffn=28672, vocab=128256,
                    n_layers=8, dtype="bf16", B=1, prefix=2048, top_k=10, rope_theta=5e5, seed=0,
                    page_size=0),
    # batched serving, LLaMA-3.1-8B shape, ragged prefixes in a 16-token page pool
    "b32_l31": dict(d=4096, n_heads=32, n_kv_heads=8, head_dim=128, ffn=14336, vocab=128256,
                    n_layers=6, dtype="bf16", B=32, prefix=(256, 4096), top_k=8, rope_theta=5e5,
                    seed=7, page_size=16),
}

RMS_EPS = 1e-5  # not stated in the paper; the LLaMA default

# tensor ids of the generator streams
TID_W_FUSE, TID_W_IN, TID_EMBED, TID_LM_HEAD = 1, 2, 3, 4
TID_FEAT, TID_TOK, TID_PREFIX, TID_PAGES = 5, 6, 7, 8


def tid_layer(i: int, j: int) -> int:
    """Layer i's streams: j = 0 qkv, 1 o, 2 gate, 3 up, 4 down, 5 K cache, 6 V cache."""
    return 1000 + 16 * i + j


def make_config(name_or_dict, **overrides) -> dict:
    w = copy.deepcopy(WORKLOADS[name_or_dict]) if isinstance(name_or_dict, str) else dict(name_or_dict)
    w.update(overrides)
    w.setdefault("rms_eps", RMS_EPS)
    w.setdefault("temperature", 0.0)
    w.setdefault("parallel_layers", 0)  # 1: the parallel (non-cascaded) ablation, Sec. 3.2
    p = w["prefix"]
    pmax = p[1] if isinstance(p, (tuple, list)) else p
    if w.get("prefix_list") is not None:  # explicit per-sequence prefix lengths
        assert len(w["prefix_list"]) == w["B"]
        pmax = max(w["prefix_list"])
    # capacity: the prefix plus the drafted row, rounded up to a whole 16-row block
    w.setdefault("max_seq", ((pmax + 1 + 15) // 16) * 16)
    w.setdefault("top_k_max", max(16, w["top_k"]))
    return w


def torch_dtype(cfg: dict):
    return torch.float32 if cfg["dtype"] == "f32" else torch.bfloat16


def _normal(shape, seed, tid, std, dt):
    t = torch.empty(shape, dtype=dt)
    fill_normal(t, seed, tid, std)
    return t


def make_weights(cfg: dict) -> dict:
    d, H, Hkv, hd = cfg["d"], cfg["n_heads"], cfg["n_kv_heads"], cfg["head_dim"]
    F, V, N, s = cfg["ffn"], cfg["vocab"], cfg["n_layers"], cfg["seed"]
    dt = torch_dtype(cfg)
    W = dict(
        w_fuse=_normal((d, 3 * d), s, TID_W_FUSE, 0.02, dt),
        w_in=_normal((d, 2 * d), s, TID_W_IN, 0.02, dt),
        embed=_normal((V, d), s, TID_EMBED, 0.02, dt),
        lm_head=_normal((V, d), s, TID_LM_HEAD, 0.02, dt),
        final_norm=torch.ones(d, dtype=dt),
        layers=[],
    )
    for i in range(N):
        W["layers"].append(dict(
            attn_norm=torch.ones(d, dtype=dt),
            w_qkv=_normal(((H + 2 * Hkv) * hd, d), s, tid_layer(i, 0), 0.02, dt),
            w_o=_normal((d, H * hd), s, tid_layer(i, 1), 0.02, dt),
            mlp_norm=torch.ones(d, dtype=dt),
            w_gate=_normal((F, d), s, tid_layer(i, 2), 0.02, dt),
            w_up=_normal((F, d), s, tid_layer(i, 3), 0.02, dt),
            w_down=_normal((d, F), s, tid_layer(i, 4), 0.02, dt),
        ))
    return W


def make_inputs(cfg: dict) -> dict:
    """Per-call inputs: features, next tokens, prefix lengths."""
    B, d, V, s = cfg["B"], cfg["d"], cfg["vocab"], cfg["seed"]
    feat = _normal((B, 3 * d), s, TID_FEAT, 1.0, torch_dtype(cfg))
    tok = torch.empty(B, dtype=torch.int32)
    fill_uniform_int(tok, s, TID_TOK, 0, V - 1)
    p = cfg["prefix"]
    plen = torch.empty(B, dtype=torch.int32)
    if cfg.get("prefix_list") is not None:
        plen = torch.tensor(cfg["prefix_list"], dtype=torch.int32)
    elif isinstance(p, (tuple, list)):
        fill_uniform_int(plen, s, TID_PREFIX, p[0], p[1])
    else:
        plen.fill_(p)
    return dict(feat=feat, next_tok=tok, prefix_len=plen)


def make_caches(cfg: dict, layers=None) -> tuple[list, list]:
    """Logical per-layer caches [B, Hkv, cap, hd] ~ N(0, 1) (all slots drawn; only the
    first P_b rows of sequence b are read)."""
    B, Hkv, hd, cap, s = cfg["B"], cfg["n_kv_heads"], cfg["head_dim"], cfg["max_seq"], cfg["seed"]
    dt = torch_dtype(cfg)
    ks, vs = [], []
    for i in (range(cfg["n_layers"]) if layers is None else layers):
        ks.append(_normal((B, Hkv, cap, hd), s, tid_layer(i, 5), 1.0, dt))
        vs.append(_normal((B, Hkv, cap, hd), s, tid_layer(i, 6), 1.0, dt))
    return ks, vs


def page_plan(cfg: dict, prefix_len: torch.Tensor) -> tuple[torch.Tensor, int]:
    """Page table [B, max_pages] (int32, -1 = unused) covering rows 0..P_b of every
    sequence, with physical pages assigned by a seeded permutation of the pool."""
    ps, B = cfg["page_size"], cfg["B"]
    max_pages = (cfg["max_seq"] + ps - 1) // ps
    need = [(int(prefix_len[b]) + 1 + ps - 1) // ps for b in range(B)]
    n_pages = sum(need)
    perm = torch.empty(n_pages, dtype=torch.int32)
    permutation(perm, cfg["seed"], TID_PAGES)
    table = torch.full((B, max_pages), -1, dtype=torch.int32)
    c = 0
    for b in range(B):
        for lp in range(need[b]):
            table[b, lp] = perm[c]
            c += 1
    return table, n_pages


def paginate(cfg: dict, logical: torch.Tensor, table: torch.Tensor, n_pages: int) -> torch.Tensor:
    """Scatter a logical [B, Hkv, cap, hd] cache into the paged pool
    [n_pages, Hkv, page_size, hd] described by ``table``."""
    ps = cfg["page_size"]
    B, Hkv, cap, hd = logical.shape
    pool = torch.zeros((n_pages, Hkv, ps, hd), dtype=logical.dtype)
    for b in range(B):
        for lp in range(table.shape[1]):
            pg = int(table[b, lp])
            if pg < 0:
                continue
            lo, hi = lp * ps, min(cap, (lp + 1) * ps)
            pool[pg, :, : hi - lo, :] = logical[b, :, lo:hi, :]
    return pool


def algorithmic_bytes(cfg: dict, prefix_len) -> int:
    """Bytes the method must move per draft: every weight once (the shared LM head once
    for all N rows), each layer's K/V read of P_b + 1 rows ... counted as P_b prefix rows
    read plus the new row written, plus the features and token ids."""
    d, H, Hkv, hd, F, V, N = (cfg[k] for k in ("d", "n_heads", "n_kv_heads", "head_dim", "ffn",
                                               "vocab", "n_layers"))
    es = 4 if cfg["dtype"] == "f32" else 2
    w = d * 3 * d + d * 2 * d + V * d
    w += N * ((H + 2 * Hkv) * hd * d + d * H * hd + 2 * F * d + d * F + 2 * d) + d
    kv_rows = sum(int(p) + 1 for p in prefix_len)
    kv = N * kv_rows * 2 * Hkv * hd
    B = len(prefix_len)
    emb = B * d  # the embedding rows gathered
    feat = B * 3 * d
    return int((w + kv + emb + feat) * es)


def kernel_bytes(cfg: dict, prefix_len) -> dict:
    """algorithmic_bytes split by kernel family (the parts sum to it): 'linear' = the
    weight-streaming phases (W_fuse, W_in and every layer's W_qkv, W_o, W_gate/up, W_down
    with the layer's two norm gains, plus the features and gathered embedding rows they
    read), 'attention' = every layer's K/V traffic, 'lm_head' = the LM head and final norm."""
    d, H, Hkv, hd, F, V, N = (cfg[k] for k in ("d", "n_heads", "n_kv_heads", "head_dim", "ffn",
                                               "vocab", "n_layers"))
    es = 4 if cfg["dtype"] == "f32" else 2
    B = len(prefix_len)
    lin = d * 3 * d + d * 2 * d + N * ((H + 2 * Hkv) * hd * d + d * H * hd + 2 * F * d + d * F + 2 * d)
    lin += B * d + B * 3 * d
    kv = N * sum(int(p) + 1 for p in prefix_len) * 2 * Hkv * hd
    return {"linear": int(lin * es), "attention": int(kv * es), "lm_head": int((V * d + d) * es)}


def algorithmic_flops(cfg: dict, prefix_len) -> int:
    d, H, Hkv, hd, F, V, N = (cfg[k] for k in ("d", "n_heads", "n_kv_heads", "head_dim", "ffn",
                                               "vocab", "n_layers"))
    B = len(prefix_len)
    per_row = d * 3 * d + d * 2 * d + N * ((H + 2 * Hkv) * hd * d + d * H * hd + 3 * F * d)
    f = 2 * per_row * B + 2 * V * d * N * B
    f += sum(4 * H * hd * (int(p) + 1) for p in prefix_len) * N
    return int(f)


def kernel_flops(cfg: dict, prefix_len) -> dict:
    """algorithmic_flops split by kernel family (the parts sum to it): 'linear' = the
    products with every weight matrix but the LM head, 'attention' = q.K and p.V over each
    layer's P_b + 1 keys, 'lm_head' = the LM head over all N * B hidden rows."""
    d, H, Hkv, hd, F, V, N = (cfg[k] for k in ("d", "n_heads", "n_kv_heads", "head_dim", "ffn",
                                               "vocab", "n_layers"))
    B = len(prefix_len)
    per_row = d * 3 * d + d * 2 * d + N * ((H + 2 * Hkv) * hd * d + d * H * hd + 3 * F * d)
    att = sum(4 * H * hd * (int(p) + 1) for p in prefix_len) * N
    return {"linear": int(2 * per_row * B), "attention": int(att), "lm_head": int(2 * V * d * N * B)}


def n_tree(cfg: dict, top_k=None) -> int:
    return 1 + cfg["n_layers"] * (top_k or cfg["top_k"])


def describe(cfg: dict) -> str:
    return (f"d{cfg['d']} H{cfg['n_heads']}/{cfg['n_kv_heads']}x{cfg['head_dim']} F{cfg['ffn']} "
            f"V{cfg['vocab']} N{cfg['n_layers']} B{cfg['B']} P{cfg['prefix']} k{cfg['top_k']} "
            f"{cfg['dtype']}" + (f" paged{cfg['page_size']}" if cfg['page_size'] else ""))




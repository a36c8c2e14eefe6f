"""An independent second opinion for the oracle's pins, in plain PyTorch fp64 on CPU.

Written from the same definitions as the oracle but along a different route, so that
an error in one does not repeat in the other: library routines instead of loops
(``torch.nn.functional.rms_norm``, ``scaled_dot_product_attention``, ``silu``), grouped-
query attention by replicating KV heads rather than by index arithmetic, and RoPE as a
complex rotation of (x_j + i x_{j+hd/2}) rather than as rotate-half.

Test code only: it is never compared with the CUDA path.
"""
from __future__ import annotations

import torch
import torch.nn.functional as F


def _d(t):
    return t.to(torch.float64)


def rope_complex(x: torch.Tensor, pos: float, theta: float) -> torch.Tensor:
    """x [..., hd]; pairs (j, j + hd/2) as complex numbers rotated by pos * theta^(-2j/hd)."""
    hd = x.shape[-1]
    half = hd // 2
    j = torch.arange(half, dtype=torch.float64)
    ang = pos * theta ** (-2.0 * j / hd)
    z = torch.complex(x[..., :half], x[..., half:]) * torch.polar(torch.ones_like(ang), ang)
    return torch.cat([z.real, z.imag], dim=-1)


def layer(cfg: dict, L: dict, x: torch.Tensor, pos: float, kc: torch.Tensor, vc: torch.Tensor,
          P: int) -> torch.Tensor:
    """One pre-norm decoder layer for one sequence; kc, vc [Hkv, cap, hd]."""
    return layer_kv(cfg, L, x, pos, kc, vc, P)[0]


def layer_kv(cfg: dict, L: dict, x: torch.Tensor, pos: float, kc: torch.Tensor, vc: torch.Tensor,
             P: int):
    """layer() returning also the row's own key (rotated) and value, [Hkv, hd] each."""
    d, H, Hkv, hd = cfg["d"], cfg["n_heads"], cfg["n_kv_heads"], cfg["head_dim"]
    eps = cfg["rms_eps"]
    u = F.rms_norm(x, (d,), weight=_d(L["attn_norm"]), eps=eps)
    qkv = _d(L["w_qkv"]) @ u
    q = qkv[: H * hd].view(H, hd)
    k = qkv[H * hd:(H + Hkv) * hd].view(Hkv, hd)
    v = qkv[(H + Hkv) * hd:].view(Hkv, hd)
    q = rope_complex(q, pos, cfg["rope_theta"])
    k = rope_complex(k, pos, cfg["rope_theta"])
    keys = torch.cat([_d(kc[:, :P, :]), k[:, None, :]], dim=1)   # [Hkv, P+1, hd]
    vals = torch.cat([_d(vc[:, :P, :]), v[:, None, :]], dim=1)
    rep = H // Hkv
    keys = keys.repeat_interleave(rep, dim=0)
    vals = vals.repeat_interleave(rep, dim=0)
    o = F.scaled_dot_product_attention(q[:, None, :], keys, vals)  # scale 1/sqrt(hd)
    x = x + _d(L["w_o"]) @ o.reshape(H * hd)
    u = F.rms_norm(x, (d,), weight=_d(L["mlp_norm"]), eps=eps)
    a = F.silu(_d(L["w_gate"]) @ u) * (_d(L["w_up"]) @ u)
    return x + _d(L["w_down"]) @ a, k, v


def draft(cfg: dict, W: dict, feat: torch.Tensor, tok: int, P: int, kcs, vcs, top_k: int,
          temperature: float = 0.0, rope_layer_offset: int = 0) -> dict:
    """The whole draft of one sequence (kcs[i], vcs[i]: [Hkv, cap, hd])."""
    d = cfg["d"]
    g = _d(W["w_fuse"]) @ _d(feat)
    e = _d(W["embed"])[tok]
    x = _d(W["w_in"]) @ torch.cat([g, e])
    hs = []
    for i, L in enumerate(W["layers"]):
        x = layer(cfg, L, x, P + (i if rope_layer_offset else 0), kcs[i], vcs[i], P)
        hs.append(x)
    h = torch.stack(hs)
    z = F.rms_norm(h, (d,), weight=_d(W["final_norm"]), eps=cfg["rms_eps"])
    logits = z @ _d(W["lm_head"]).T
    T = temperature if temperature > 0 else 1.0
    logp = torch.log_softmax(logits / T, dim=-1)
    lse = torch.logsumexp(logits / T, dim=-1)
    order = torch.sort(-logits, dim=-1, stable=True).indices[:, :top_k]
    return dict(hidden=h, logits=logits, lse=lse, prob=logp.exp(), topk_id=order)


def commit(cfg: dict, W: dict, feats: torch.Tensor, toks, P: int, kcs, vcs) -> None:
    """Commit rows at positions P, P + 1, ..: each row runs Eq. 1 and the cascade, then its
    per-layer key and value are stored (in the caches' dtype) in slot P + i before the next
    row runs; kcs[i], vcs[i] [Hkv, cap, hd] are written in place."""
    for i, tok in enumerate(toks):
        g = _d(W["w_fuse"]) @ _d(feats[i])
        e = _d(W["embed"])[int(tok)]
        x = _d(W["w_in"]) @ torch.cat([g, e])
        for l, L in enumerate(W["layers"]):
            x, k, v = layer_kv(cfg, L, x, P + i, kcs[l], vcs[l], P + i)
            kcs[l][:, P + i, :] = k.to(kcs[l].dtype)
            vcs[l][:, P + i, :] = v.to(vcs[l].dtype)

"""GB300 (sm_103a) FastEagle cascaded drafter: Python binding of libfe_draft.so.

The functions here carry the C ABI's names (include/fe_draft.h) and only marshal
arguments: torch tensors become device pointers, dicts become the ABI's structs, and
PyTorch provides device memory and the current CUDA stream. Every step of a draft runs
in the library's CUDA kernels; there is no CPU or PyTorch fallback. If the compiled
library is missing, importing this package raises (build it with
``python -c "import __graft_entry__ as g; g.build()"``).
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libfe_draft.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: the CUDA extension has not been built "
                      "(run __graft_entry__.build())")

_lib = ctypes.CDLL(LIB_PATH)

FE_OK, FE_ERR_INVALID_ARG, FE_ERR_UNSUPPORTED, FE_ERR_CUDA = 0, -1, -2, -3
FE_ERR_OOM, FE_ERR_CAPACITY, FE_ERR_TIMEOUT, FE_ERR_DEVICE = -4, -5, -6, -7
FE_F32, FE_BF16 = 0, 1

_vp = ctypes.c_void_p
_i32 = ctypes.c_int32


class fe_config(ctypes.Structure):
    _fields_ = [("d", _i32), ("n_heads", _i32), ("n_kv_heads", _i32), ("head_dim", _i32),
                ("ffn", _i32), ("vocab", _i32), ("n_layers", _i32), ("top_k_max", _i32),
                ("max_batch", _i32), ("max_seq", _i32), ("page_size", _i32),
                ("rope_theta", ctypes.c_float), ("rms_eps", ctypes.c_float), ("dtype", ctypes.c_int),
                ("parallel_layers", _i32)]


class fe_layer_weights(ctypes.Structure):
    _fields_ = [(n, _vp) for n in ("attn_norm", "w_qkv", "w_o", "mlp_norm", "w_gate", "w_up", "w_down")]


class fe_weights(ctypes.Structure):
    _fields_ = [("w_fuse", _vp), ("w_in", _vp), ("embed", _vp), ("lm_head", _vp), ("final_norm", _vp),
                ("layers", ctypes.POINTER(fe_layer_weights))]


class fe_forward_args(ctypes.Structure):
    _fields_ = [("B", _i32), ("top_k", _i32), ("temperature", ctypes.c_float),
                ("feat", _vp), ("next_tok", _vp), ("prefix_len", _vp),
                ("k_cache", ctypes.POINTER(_vp)), ("v_cache", ctypes.POINTER(_vp)),
                ("page_table", _vp), ("n_pages", _i32),
                ("topk_id", _vp), ("topk_logit", _vp), ("topk_prob", _vp), ("lse", _vp),
                ("dbg_logits", _vp), ("dbg_hidden", _vp), ("sample", _i32), ("seed", ctypes.c_uint64),
                ("topk_rank", _vp)]


class fe_tree(ctypes.Structure):
    _fields_ = [("tok", _vp), ("parent", _vp), ("depth", _vp), ("mask", _vp)]


class fe_commit_args(ctypes.Structure):
    _fields_ = [("B", _i32), ("L", _i32), ("feat", _vp), ("tok", _vp), ("n_rows", _vp), ("prefix_len", _vp),
                ("k_cache", ctypes.POINTER(_vp)), ("v_cache", ctypes.POINTER(_vp)),
                ("page_table", _vp), ("n_pages", _i32)]


class fe_host_step_args(ctypes.Structure):
    _fields_ = [("B", _i32), ("top_k", _i32), ("temperature", ctypes.c_float), ("feat", _vp), ("next_tok", _vp),
                ("prefix_len", _vp), ("k_cache", ctypes.POINTER(_vp)), ("v_cache", ctypes.POINTER(_vp)),
                ("page_table", _vp), ("n_pages", _i32), ("topk_id", _vp), ("topk_logit", _vp), ("topk_prob", _vp),
                ("lse", _vp), ("tree_tok", _vp), ("tree_parent", _vp), ("tree_depth", _vp), ("tree_mask", _vp),
                ("sample", _i32), ("seed", ctypes.c_uint64), ("topk_rank", _vp)]


_lib.fe_draft_init.argtypes = [ctypes.POINTER(fe_config), ctypes.POINTER(fe_weights), _vp, ctypes.POINTER(_vp)]
_lib.fe_draft_init.restype = ctypes.c_int
_lib.fe_draft_forward.argtypes = [_vp, ctypes.POINTER(fe_forward_args), _vp]
_lib.fe_draft_forward.restype = ctypes.c_int
_lib.fe_build_tree.argtypes = [_vp, _i32, _i32, _vp, _vp, ctypes.POINTER(fe_tree), _vp]
_lib.fe_build_tree.restype = ctypes.c_int
_lib.fe_last_device_status.argtypes = [_vp, _vp]
_lib.fe_last_device_status.restype = ctypes.c_int
_lib.fe_free.argtypes = [_vp]
_lib.fe_free.restype = None
_lib.fe_status_str.argtypes = [ctypes.c_int]
_lib.fe_status_str.restype = ctypes.c_char_p
_lib.fe_launch_count.argtypes = [_vp, _i32, _i32]
_lib.fe_launch_count.restype = _i32
_lib.fe_selftest_timeout.argtypes = [_vp, ctypes.c_int64, _vp]
_lib.fe_selftest_timeout.restype = ctypes.c_int
_lib.fe_lm_head_topk_noalloc.argtypes = [_vp, _vp, _i32, _i32, ctypes.c_float, _vp, _vp, _vp, _vp, _vp]
_lib.fe_lm_head_topk_noalloc.restype = ctypes.c_int
_lib.fe_profile_forward.argtypes = [_vp, ctypes.POINTER(fe_forward_args), _vp, _i32, _vp, _vp, ctypes.POINTER(_i32)]
_lib.fe_profile_forward.restype = ctypes.c_int
_lib.fe_profile_graph.argtypes = [_vp, ctypes.POINTER(fe_forward_args), _vp, _vp, _i32, _vp, _vp, _vp,
                                  ctypes.POINTER(_i32)]
_lib.fe_profile_graph.restype = ctypes.c_int
_lib.fe_draft_loss.argtypes = [_vp, ctypes.POINTER(fe_forward_args), _vp, _vp, ctypes.c_float, ctypes.c_float,
                               ctypes.c_float, _vp, _vp, _vp, _vp]
_lib.fe_draft_loss.restype = ctypes.c_int
_lib.fe_verify_greedy.argtypes = [_vp, _i32, _i32, _vp, ctypes.POINTER(fe_tree), _vp, _vp, _vp, _vp, _vp, _vp]
_lib.fe_verify_greedy.restype = ctypes.c_int
_lib.fe_verify_sampled.argtypes = [_vp, _i32, _i32, ctypes.POINTER(fe_tree), _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                   _vp]
_lib.fe_verify_sampled.restype = ctypes.c_int
_lib.fe_draft_step_host.argtypes = [_vp, ctypes.POINTER(fe_host_step_args), _vp]
_lib.fe_draft_step_host.restype = ctypes.c_int
_lib.fe_commit.argtypes = [_vp, ctypes.POINTER(fe_commit_args), _vp]
_lib.fe_commit.restype = ctypes.c_int
_lib.fe_last_error_detail.argtypes = []
_lib.fe_last_error_detail.restype = ctypes.c_char_p


class FeError(RuntimeError):
    def __init__(self, code: int, where: str):
        detail = fe_last_error_detail() if code in (FE_ERR_CUDA, FE_ERR_OOM) else ""
        super().__init__(f"{where}: {fe_status_str(code)} ({code})" + (f" [{detail}]" if detail else ""))
        self.code = code


def fe_last_error_detail() -> str:
    return _lib.fe_last_error_detail().decode()


def fe_status_str(code: int) -> str:
    return _lib.fe_status_str(code).decode()


def _check(code: int, where: str) -> None:
    if code != FE_OK:
        raise FeError(code, where)


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _p(t) -> int | None:
    """The address of a contiguous tensor (host or device memory), or the int / None given."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if not t.is_contiguous():
        raise ValueError("buffers passed to the drafter must be contiguous")
    return t.data_ptr()


def _dp(t) -> int | None:
    """As _p, for a buffer the kernels read or write: a tensor must be on a CUDA device. A
    host address given to a kernel faults, or, on a GPU that can reach host memory, reads
    and writes host memory the caller did not mean to share."""
    if t is not None and not isinstance(t, int) and not t.is_cuda:
        raise ValueError("buffers the kernels access must be CUDA tensors")
    return _p(t)


def make_config(cfg: dict) -> fe_config:
    return fe_config(cfg["d"], cfg["n_heads"], cfg["n_kv_heads"], cfg["head_dim"], cfg["ffn"], cfg["vocab"],
                     cfg["n_layers"], cfg["top_k_max"], cfg.get("max_batch", cfg.get("B", 1)), cfg["max_seq"],
                     cfg.get("page_size", 0), float(cfg["rope_theta"]), float(cfg["rms_eps"]),
                     FE_F32 if cfg["dtype"] == "f32" else FE_BF16, int(cfg.get("parallel_layers", 0)))


class Handle:
    """An initialised drafter (owns a fe_handle*)."""

    def __init__(self, ptr: int, cfg: dict):
        self.ptr = ptr
        self.cfg = dict(cfg)

    def __del__(self):
        self.close()

    def close(self):
        if getattr(self, "ptr", None):
            _lib.fe_free(self.ptr)
            self.ptr = None


def fe_draft_init(cfg: dict, weights: dict, stream=None) -> Handle:
    """weights: dict of tensors (host or device) in the canonical layout:
    w_fuse, w_in, embed, lm_head, final_norm, and layers: list of dicts with attn_norm,
    w_qkv, w_o, mlp_norm, w_gate, w_up, w_down."""
    L = weights["layers"]
    arr = (fe_layer_weights * len(L))()
    for i, l in enumerate(L):
        arr[i] = fe_layer_weights(_p(l["attn_norm"]), _p(l["w_qkv"]), _p(l["w_o"]), _p(l["mlp_norm"]),
                                  _p(l["w_gate"]), _p(l["w_up"]), _p(l["w_down"]))
    w = fe_weights(_p(weights["w_fuse"]), _p(weights["w_in"]), _p(weights["embed"]), _p(weights["lm_head"]),
                   _p(weights["final_norm"]), arr)
    c = make_config(cfg)
    out = _vp()
    _check(_lib.fe_draft_init(ctypes.byref(c), ctypes.byref(w), _stream(stream), ctypes.byref(out)),
           "fe_draft_init")
    return Handle(out.value, cfg)


def alloc_outputs(h: Handle, B: int, top_k: int, device="cuda") -> dict:
    N = h.cfg["n_layers"]
    return dict(topk_id=torch.empty((B, N, top_k), dtype=torch.int32, device=device),
                topk_logit=torch.empty((B, N, top_k), dtype=torch.float32, device=device),
                topk_prob=torch.empty((B, N, top_k), dtype=torch.float32, device=device),
                lse=torch.empty((B, N), dtype=torch.float32, device=device),
                topk_rank=torch.empty((B, N, top_k), dtype=torch.int32, device=device))


def _forward_args(h: Handle, feat, next_tok, prefix_len, kc, vc, top_k, temperature, page_table, n_pages, out,
                  dbg_logits, dbg_hidden, sample, seed) -> fe_forward_args:
    a = fe_forward_args(int(next_tok.shape[0]), top_k, float(temperature), _dp(feat), _dp(next_tok),
                        _dp(prefix_len), kc, vc, _dp(page_table), int(n_pages), _dp(out["topk_id"]),
                        _dp(out["topk_logit"]), _dp(out["topk_prob"]), _dp(out["lse"]), _dp(dbg_logits),
                        _dp(dbg_hidden))
    a.sample = 1 if sample else 0
    a.seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    a.topk_rank = _dp(out.get("topk_rank"))
    return a


def fe_draft_forward(h: Handle, feat, next_tok, prefix_len, k_cache, v_cache, top_k: int,
                     temperature: float = 0.0, page_table=None, n_pages: int = 0, out: dict | None = None,
                     dbg_logits=None, dbg_hidden=None, stream=None, sample: bool = False, seed: int = 0) -> dict:
    """One draft. feat [B, 3d], next_tok [B] i32, prefix_len [B] i32 (device tensors);
    k_cache / v_cache: lists of per-layer device tensors (see include/fe_draft.h). With
    sample (and temperature > 0) the candidates are drawn (stochastic drafting, seeded by
    ``seed``); out["topk_rank"] then gives each one's position in draw order."""
    B = int(next_tok.shape[0])
    if out is None:
        out = alloc_outputs(h, B, top_k, feat.device)
    N = h.cfg["n_layers"]
    kc = (_vp * N)(*[_dp(t) for t in k_cache])
    vc = (_vp * N)(*[_dp(t) for t in v_cache])
    a = _forward_args(h, feat, next_tok, prefix_len, kc, vc, top_k, temperature, page_table, n_pages, out,
                      dbg_logits, dbg_hidden, sample, seed)
    _check(_lib.fe_draft_forward(h.ptr, ctypes.byref(a), _stream(stream)), "fe_draft_forward")
    return out


FE_KERNEL_NAMES = {0: "linear", 1: "attention", 2: "lm_prep", 3: "lm_head", 4: "copy", 5: "linear_prep",
                   6: "tree"}


def fe_profile_forward(h: Handle, feat, next_tok, prefix_len, k_cache, v_cache, top_k: int,
                       temperature: float = 0.0, page_table=None, n_pages: int = 0, out: dict | None = None,
                       dbg_hidden=None, stream=None, sample: bool = False, seed: int = 0) -> list[tuple[str, float]]:
    """One draft launched eagerly with a CUDA event after every launch (include/fe_draft.h).
    Returns [(kernel family, device microseconds)] in launch order."""
    B = int(next_tok.shape[0])
    if out is None:
        out = alloc_outputs(h, B, top_k, feat.device)
    N = h.cfg["n_layers"]
    kc = (_vp * N)(*[_dp(t) for t in k_cache])
    vc = (_vp * N)(*[_dp(t) for t in v_cache])
    a = _forward_args(h, feat, next_tok, prefix_len, kc, vc, top_k, temperature, page_table, n_pages, out, None,
                      dbg_hidden, sample, seed)
    cap = fe_launch_count(h, B, False) + 1
    kinds = (_i32 * cap)()
    usec = (ctypes.c_float * cap)()
    n = _i32(0)
    _check(_lib.fe_profile_forward(h.ptr, ctypes.byref(a), _stream(stream), cap, ctypes.cast(kinds, _vp),
                                   ctypes.cast(usec, _vp), ctypes.byref(n)), "fe_profile_forward")
    return [(FE_KERNEL_NAMES.get(kinds[j], str(kinds[j])), float(usec[j])) for j in range(n.value)]


def fe_profile_graph(h: Handle, feat, next_tok, prefix_len, k_cache, v_cache, top_k: int,
                     temperature: float = 0.0, page_table=None, n_pages: int = 0, out: dict | None = None,
                     tree: dict | None = None, stream=None, sample: bool = False,
                     seed: int = 0) -> list[tuple[str, float, float]]:
    """One draft (plus the tree kernel when ``tree`` is given) run as the CUDA graph
    fe_draft_forward uses, with every kernel's first start and last exit stamped on the GPU
    (include/fe_draft.h). Returns [(kernel family, start us, end us)] in launch order, times
    from the run's earliest start."""
    B = int(next_tok.shape[0])
    if out is None:
        out = alloc_outputs(h, B, top_k, feat.device)
    N = h.cfg["n_layers"]
    kc = (_vp * N)(*[_dp(t) for t in k_cache])
    vc = (_vp * N)(*[_dp(t) for t in v_cache])
    a = _forward_args(h, feat, next_tok, prefix_len, kc, vc, top_k, temperature, page_table, n_pages, out, None,
                      None, sample, seed)
    t = None
    if tree is not None:
        t = fe_tree(_dp(tree["tok"]), _dp(tree["parent"]), _dp(tree["depth"]), _dp(tree["mask"]))
    cap = fe_launch_count(h, B, tree is not None) + 1
    kinds = (_i32 * cap)()
    t0 = (ctypes.c_double * cap)()
    t1 = (ctypes.c_double * cap)()
    n = _i32(0)
    _check(_lib.fe_profile_graph(h.ptr, ctypes.byref(a), ctypes.byref(t) if t is not None else None, _stream(stream),
                                 cap, ctypes.cast(kinds, _vp), ctypes.cast(t0, _vp), ctypes.cast(t1, _vp),
                                 ctypes.byref(n)), "fe_profile_graph")
    return [(FE_KERNEL_NAMES.get(kinds[j], str(kinds[j])), float(t0[j]), float(t1[j])) for j in range(n.value)]


def in_step_times(launches: list[tuple[str, float, float]]) -> list[tuple[str, float, float]]:
    """[(family, span us, added us)] from fe_profile_graph's stamps: the span is a launch's
    first start to last exit; the added time is how far its end lies past the previous
    launch's end (the first launch: its span), so the added times partition the step."""
    res, prev_end = [], None
    for kind, s, e in launches:
        if s < 0 or e < 0:
            continue
        add = (e - s) if prev_end is None else max(0.0, e - prev_end)
        res.append((kind, e - s, add))
        prev_end = e if prev_end is None else max(prev_end, e)
    return res


def fe_draft_loss(h: Handle, feat, next_tok, prefix_len, k_cache, v_cache, teacher_p, target_feat, top_k: int,
                  alpha: float = 0.1, beta: float = 1.0, decay: float = 0.9, page_table=None, n_pages: int = 0,
                  stream=None) -> dict:
    """Forward of the training objective (include/fe_draft.h): teacher_p [B, N, V], target_feat
    [N, B, d] (float32, device). Returns the draft's outputs plus logits, hidden, ce, feat_loss
    and total."""
    B = int(next_tok.shape[0])
    N, d, V = h.cfg["n_layers"], h.cfg["d"], h.cfg["vocab"]
    dev = feat.device
    out = alloc_outputs(h, B, top_k, dev)
    out.update(logits=torch.empty((B, N, V), device=dev), hidden=torch.empty((N, B, d), device=dev),
               ce=torch.empty((B, N), device=dev), feat_loss=torch.empty((B, N), device=dev),
               total=torch.empty(B, device=dev))
    kc = (_vp * N)(*[_dp(t) for t in k_cache])
    vc = (_vp * N)(*[_dp(t) for t in v_cache])
    a = fe_forward_args(B, top_k, 1.0, _dp(feat), _dp(next_tok), _dp(prefix_len), kc, vc, _dp(page_table),
                        int(n_pages), _dp(out["topk_id"]), _dp(out["topk_logit"]), _dp(out["topk_prob"]),
                        _dp(out["lse"]), _dp(out["logits"]), _dp(out["hidden"]))
    _check(_lib.fe_draft_loss(h.ptr, ctypes.byref(a), _dp(teacher_p), _dp(target_feat), float(alpha), float(beta),
                              float(decay), _dp(out["ce"]), _dp(out["feat_loss"]), _dp(out["total"]), _stream(stream)),
           "fe_draft_loss")
    return out


def alloc_tree(h: Handle, B: int, top_k: int, device="cuda") -> dict:
    T = 1 + h.cfg["n_layers"] * top_k
    return dict(tok=torch.empty((B, T), dtype=torch.int32, device=device),
                parent=torch.empty((B, T), dtype=torch.int32, device=device),
                depth=torch.empty((B, T), dtype=torch.int32, device=device),
                mask=torch.empty((B, T, T), dtype=torch.uint8, device=device))


def fe_build_tree(h: Handle, next_tok, topk_id, top_k: int, out: dict | None = None, stream=None) -> dict:
    B = int(next_tok.shape[0])
    if out is None:
        out = alloc_tree(h, B, top_k, next_tok.device)
    t = fe_tree(_dp(out["tok"]), _dp(out["parent"]), _dp(out["depth"]), _dp(out["mask"]))
    _check(_lib.fe_build_tree(h.ptr, B, top_k, _dp(next_tok), _dp(topk_id), ctypes.byref(t), _stream(stream)),
           "fe_build_tree")
    return out


def alloc_host_step_outputs(h: Handle, B: int, top_k: int) -> dict:
    """Host (pinned) tensors for fe_draft_step_host's outputs."""
    N = h.cfg["n_layers"]
    T = 1 + N * top_k
    e = lambda shape, dt: torch.empty(shape, dtype=dt).pin_memory()
    return dict(topk_id=e((B, N, top_k), torch.int32), topk_logit=e((B, N, top_k), torch.float32),
                topk_prob=e((B, N, top_k), torch.float32), lse=e((B, N), torch.float32),
                topk_rank=e((B, N, top_k), torch.int32),
                tree_tok=e((B, T), torch.int32), tree_parent=e((B, T), torch.int32), tree_depth=e((B, T), torch.int32),
                tree_mask=e((B, T, T), torch.uint8))


def fe_draft_step_host(h: Handle, feat, next_tok, prefix_len, k_cache, v_cache, top_k: int, temperature: float = 0.0,
                       page_table=None, n_pages: int = 0, out: dict | None = None, stream=None, sample: bool = False,
                       seed: int = 0) -> dict:
    """One draft step from and to host memory (include/fe_draft.h): feat [B, 3d], next_tok
    [B], prefix_len [B] are CPU tensors; the caches (and page table) are device tensors.
    Returns CPU tensors topk_id, topk_logit, topk_prob, lse, tree_tok, tree_parent,
    tree_depth, tree_mask."""
    for t in (feat, next_tok, prefix_len):
        if t.is_cuda or not t.is_contiguous():
            raise ValueError("fe_draft_step_host takes contiguous host tensors")
    B = int(next_tok.shape[0])
    if out is None:
        out = alloc_host_step_outputs(h, B, top_k)
    N = h.cfg["n_layers"]
    kc = (_vp * N)(*[_dp(t) for t in k_cache])
    vc = (_vp * N)(*[_dp(t) for t in v_cache])
    a = fe_host_step_args(B, top_k, float(temperature), _p(feat), _p(next_tok), _p(prefix_len), kc, vc,
                          _dp(page_table), int(n_pages), _p(out["topk_id"]), _p(out["topk_logit"]),
                          _p(out["topk_prob"]), _p(out["lse"]), _p(out["tree_tok"]), _p(out["tree_parent"]),
                          _p(out["tree_depth"]), _p(out["tree_mask"]))
    a.sample = 1 if sample else 0
    a.seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    a.topk_rank = _p(out.get("topk_rank"))
    _check(_lib.fe_draft_step_host(h.ptr, ctypes.byref(a), _stream(stream)), "fe_draft_step_host")
    return out


def fe_verify_greedy(h: Handle, prefix_len, tree: dict, target_next, top_k: int, out: dict | None = None,
                     stream=None) -> dict:
    """Tree positions and the greedy acceptance walk (include/fe_draft.h). tree: the dict
    fe_build_tree returns; target_next [B, T] int32 (device)."""
    B = int(prefix_len.shape[0])
    N = h.cfg["n_layers"]
    T = 1 + N * top_k
    dev = prefix_len.device
    if out is None:
        out = dict(pos_ids=torch.empty((B, T), dtype=torch.int32, device=dev),
                   path=torch.empty((B, N), dtype=torch.int32, device=dev),
                   n_accept=torch.empty(B, dtype=torch.int32, device=dev),
                   bonus=torch.empty(B, dtype=torch.int32, device=dev))
    t = fe_tree(_dp(tree["tok"]), _dp(tree["parent"]), _dp(tree["depth"]), _dp(tree["mask"]))
    _check(_lib.fe_verify_greedy(h.ptr, B, int(top_k), _dp(prefix_len), ctypes.byref(t), _dp(target_next),
                                 _dp(out["pos_ids"]), _dp(out["path"]), _dp(out["n_accept"]), _dp(out["bonus"]),
                                 _stream(stream)), "fe_verify_greedy")
    return out


def fe_verify_sampled(h: Handle, tree: dict, topk_rank, q, p, u_acc, u_bonus, top_k: int, out: dict | None = None,
                      stream=None) -> dict:
    """Lossless verification of a sampled tree (include/fe_draft.h): tree from fe_build_tree,
    topk_rank [B, N, k] int32 (fe_draft_forward's draw positions), q [B, N, V] and p [B, T, V]
    float32 distributions, u_acc / u_bonus [B, T] float32 uniforms (device tensors). Returns
    path [B, N], n_accept [B] and bonus [B]."""
    B = int(topk_rank.shape[0])
    N = h.cfg["n_layers"]
    dev = topk_rank.device
    if out is None:
        out = dict(path=torch.empty((B, N), dtype=torch.int32, device=dev),
                   n_accept=torch.empty(B, dtype=torch.int32, device=dev),
                   bonus=torch.empty(B, dtype=torch.int32, device=dev))
    t = fe_tree(_dp(tree["tok"]), _dp(tree["parent"]), _dp(tree["depth"]), _dp(tree["mask"]))
    _check(_lib.fe_verify_sampled(h.ptr, B, int(top_k), ctypes.byref(t), _dp(topk_rank), _dp(q), _dp(p), _dp(u_acc),
                                  _dp(u_bonus), _dp(out["path"]), _dp(out["n_accept"]), _dp(out["bonus"]),
                                  _stream(stream)), "fe_verify_sampled")
    return out


def fe_commit(h: Handle, feat, tok, n_rows, prefix_len, k_cache, v_cache, page_table=None, n_pages: int = 0,
              stream=None) -> None:
    """Commit accepted rows into the caches (include/fe_draft.h): feat [B, L, 3d], tok [B, L]
    int32, n_rows [B] int32, prefix_len [B] int32 (device tensors)."""
    B, L = int(tok.shape[0]), int(tok.shape[1])
    N = h.cfg["n_layers"]
    kc = (_vp * N)(*[_dp(t) for t in k_cache])
    vc = (_vp * N)(*[_dp(t) for t in v_cache])
    a = fe_commit_args(B, L, _dp(feat), _dp(tok), _dp(n_rows), _dp(prefix_len), kc, vc, _dp(page_table), int(n_pages))
    _check(_lib.fe_commit(h.ptr, ctypes.byref(a), _stream(stream)), "fe_commit")


def fe_last_device_status(h: Handle, stream=None) -> int:
    return int(_lib.fe_last_device_status(h.ptr, _stream(stream)))


def fe_free(h: Handle) -> None:
    h.close()


def fe_launch_count(h: Handle, B: int, with_tree: bool = True) -> int:
    return int(_lib.fe_launch_count(h.ptr, B, 1 if with_tree else 0))


def fe_selftest_timeout(h: Handle, timeout_ns: int, stream=None) -> int:
    return int(_lib.fe_selftest_timeout(h.ptr, int(timeout_ns), _stream(stream)))


def fe_lm_head_topk_noalloc(h: Handle, hidden, B: int, top_k: int, temperature: float = 0.0,
                            out: dict | None = None, stream=None) -> dict:
    """LM head + softmax statistics + top-k over hidden [N, B, d] (float32, device) without
    allocating device memory inside the library (see include/fe_draft.h). Output buffers
    are allocated here by PyTorch unless given in ``out``."""
    if out is None:
        out = alloc_outputs(h, B, top_k, hidden.device)
    _check(_lib.fe_lm_head_topk_noalloc(h.ptr, _dp(hidden), int(B), int(top_k), float(temperature),
                                        _dp(out["topk_id"]), _dp(out["topk_logit"]), _dp(out["topk_prob"]),
                                        _dp(out["lse"]), _stream(stream)), "fe_lm_head_topk_noalloc")
    return out

"""fp64 CPU oracle of the FastEagle cascaded drafter -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline / reference leg of
``bench.py`` may import this package. The product path (``paper_2509_20416_gb300``)
never imports it, and it never imports the product path: the two share no code.

This file only marshals arguments into ``oracle.c`` (compiled with gcc into
``liboracle.so``); every number is computed there, in double precision, from the
paper's definitions (Eq. 1-2 and Sec. 2.1 for the cascade and LM head, Sec. 2.2 for
top-k and the Backbone Expansion tree).

``build(mutant=n)`` compiles a copy with one planted mistake (``OR_MUTANT=n``); the
mutation tests use it to show that the pins catch plausible errors.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_lock = threading.Lock()
_cache: dict = {}

# Number of planted-mistake variants compiled by build(mutant=n) (n = 1..N_MUTANTS).
N_MUTANTS = 44
_UNUSED_MUTANTS = {25}  # ids with no planted mistake


def lib_path(mutant: int = 0, outdir: str | None = None) -> str:
    name = "liboracle.so" if mutant == 0 else f"liboracle_m{mutant}.so"
    return os.path.join(outdir or _HERE, name)


def build(mutant: int = 0, outdir: str | None = None, force: bool = False) -> str:
    out = lib_path(mutant, outdir)
    if force or not os.path.exists(out) or os.path.getmtime(out) < os.path.getmtime(_SRC):
        tmp = out + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
               f"-DOR_MUTANT={mutant}", _SRC, "-o", tmp, "-lm"]
        subprocess.check_call(cmd)
        os.replace(tmp, out)
    return out


class Config(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("ffn", ctypes.c_int32), ("vocab", ctypes.c_int32),
                ("n_layers", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("rope_theta", ctypes.c_double), ("rms_eps", ctypes.c_double),
                ("rope_layer_offset", ctypes.c_int32), ("final_norm", ctypes.c_int32),
                ("parallel_layers", ctypes.c_int32)]


_P = ctypes.c_void_p
_D = ctypes.POINTER(ctypes.c_double)


def _dp(a: np.ndarray):
    assert a.dtype == np.float64 and a.flags.c_contiguous
    return a.ctypes.data_as(_D)


def _ptr(t) -> int:
    """Address of a contiguous host buffer (numpy array or CPU torch tensor)."""
    if isinstance(t, np.ndarray):
        assert t.flags.c_contiguous
        return t.ctypes.data
    assert t.device.type == "cpu" and t.is_contiguous()
    return t.data_ptr()


def _dtype_code(t) -> int:
    if isinstance(t, np.ndarray):
        return {np.dtype(np.float32): 0, np.dtype(np.uint16): 1}[t.dtype]
    import torch
    return {torch.float32: 0, torch.bfloat16: 1}[t.dtype]


class Oracle:
    """ctypes view of one compiled oracle (the default build, or a planted mutant)."""

    def __init__(self, path: str):
        L = ctypes.CDLL(path)
        L.or_widen.argtypes = [_P, ctypes.c_int32, ctypes.c_int64, _D]
        L.or_matvec.argtypes = [_P, ctypes.c_int32, ctypes.c_int64, ctypes.c_int64, _D, _D]
        L.or_rmsnorm.argtypes = [_D, _P, ctypes.c_int32, ctypes.c_int64, ctypes.c_double, _D]
        L.or_rope.argtypes = [_D, ctypes.c_int32, ctypes.c_double, ctypes.c_double]
        L.or_attention.argtypes = [_D, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, _P, _P,
                                   ctypes.c_int32, ctypes.c_int64, ctypes.c_int32, _D, _D, _D]
        L.or_silu_mul.argtypes = [_D, _D, ctypes.c_int64, _D]
        L.or_layer.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(_P), ctypes.c_double, _P, _P,
                               ctypes.c_int64, ctypes.c_int32, _D, _D, _D]
        L.or_lm_head.argtypes = [ctypes.POINTER(Config), _P, _P, _D, _D]
        L.or_softmax.argtypes = [_D, ctypes.c_int64, ctypes.c_double, _D, _D]
        L.or_topk.argtypes = [_D, ctypes.c_int64, ctypes.c_int32, ctypes.POINTER(ctypes.c_int32)]
        L.or_smooth_l1.argtypes = [ctypes.c_double]
        L.or_smooth_l1.restype = ctypes.c_double
        L.or_loss.argtypes = [ctypes.c_int32, ctypes.c_int64, ctypes.c_int64, _D, _D, _D, _D, ctypes.c_double,
                              ctypes.c_double, ctypes.c_double, _D, _D]
        L.or_loss.restype = ctypes.c_double
        _I = ctypes.POINTER(ctypes.c_int32)
        L.or_accept_greedy.argtypes = [ctypes.c_int32, _I, _I, _I, _I, ctypes.c_int32, ctypes.c_int32, _I, _I, _I]
        L.or_accept_greedy.restype = ctypes.c_int32
        L.or_tree.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                              ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int32),
                              ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int32),
                              ctypes.POINTER(ctypes.c_uint8)]
        L.or_draft_seq.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(_P), _P, ctypes.c_int32,
                                   ctypes.c_int32, ctypes.POINTER(_P), ctypes.POINTER(_P),
                                   ctypes.c_int64, ctypes.c_int32, ctypes.c_double, _D, _D, _D,
                                   ctypes.POINTER(ctypes.c_int32), _D, _D]
        L.or_draft_seq.restype = ctypes.c_int32
        L.or_max_threads.restype = ctypes.c_int32
        L.or_splitmix64.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
        L.or_splitmix64.restype = ctypes.c_uint64
        L.or_uniform.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
        L.or_uniform.restype = ctypes.c_double
        L.or_accept_sampled.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64, _I, _I, _I,
                                        _I, _D, _D, _D, _D, _I, _I, _I, _D]
        L.or_sample_keys.argtypes = [_D, ctypes.c_int64, ctypes.c_double, ctypes.c_uint64, ctypes.c_int64, _D]
        L.or_topk_sample_rows.argtypes = [_D, ctypes.c_int64, ctypes.c_int64, ctypes.c_int32, ctypes.c_double,
                                          ctypes.c_uint64, ctypes.c_int64, _I, _I]
        L.or_commit_seq.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(_P), _P, _I, ctypes.c_int32,
                                    ctypes.c_int32, ctypes.POINTER(_P), ctypes.POINTER(_P), ctypes.c_int64]
        L.or_commit_seq.restype = ctypes.c_int32
        self.L = L
        self.path = path

    # -- primitives (used by the pins) ------------------------------------------------
    def matvec(self, W, x):
        W = np.ascontiguousarray(W)
        M, K = W.shape
        x = np.ascontiguousarray(x, dtype=np.float64)
        y = np.zeros(M)
        self.L.or_matvec(_ptr(W), _dtype_code(W), M, K, _dp(x), _dp(y))
        return y

    def rmsnorm(self, x, gamma, eps):
        x = np.ascontiguousarray(x, dtype=np.float64)
        gamma = np.ascontiguousarray(gamma)
        y = np.zeros_like(x)
        self.L.or_rmsnorm(_dp(x), _ptr(gamma), _dtype_code(gamma), x.size, eps, _dp(y))
        return y

    def rope(self, v, pos, theta):
        v = np.array(v, dtype=np.float64)
        self.L.or_rope(_dp(v), v.size, float(pos), float(theta))
        return v

    def attention(self, q, kc, vc, P, k_new, v_new):
        """q [H,hd] f64; kc, vc [Hkv,cap,hd] (float32 or bf16-as-uint16); k_new, v_new [Hkv,hd]."""
        q = np.ascontiguousarray(q, dtype=np.float64)
        H, hd = q.shape
        Hkv, cap, _ = kc.shape
        kn = np.ascontiguousarray(k_new, dtype=np.float64)
        vn = np.ascontiguousarray(v_new, dtype=np.float64)
        out = np.zeros_like(q)
        kc = np.ascontiguousarray(kc)
        vc = np.ascontiguousarray(vc)
        self.L.or_attention(_dp(q), H, Hkv, hd, _ptr(kc), _ptr(vc), _dtype_code(kc), cap, P,
                            _dp(kn), _dp(vn), _dp(out))
        return out

    def silu_mul(self, gate, up):
        g = np.ascontiguousarray(gate, dtype=np.float64)
        u = np.ascontiguousarray(up, dtype=np.float64)
        y = np.zeros_like(g)
        self.L.or_silu_mul(_dp(g), _dp(u), g.size, _dp(y))
        return y

    def softmax(self, logits, T=1.0):
        lg = np.ascontiguousarray(logits, dtype=np.float64)
        p = np.zeros_like(lg)
        lse = ctypes.c_double()
        self.L.or_softmax(_dp(lg), lg.size, T, _dp(p), ctypes.byref(lse))
        return p, lse.value

    def topk(self, logits, k):
        lg = np.ascontiguousarray(logits, dtype=np.float64)
        ids = np.zeros(k, dtype=np.int32)
        self.L.or_topk(_dp(lg), lg.size, k, ids.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)))
        return ids

    def splitmix64(self, seed: int, n: int) -> int:
        return int(self.L.or_splitmix64(seed, n))

    def uniform(self, seed: int, n: int) -> float:
        return float(self.L.or_uniform(seed, n))

    def topk_sample(self, logits, k: int, T: float, seed: int, row0: int = 0):
        """k candidates drawn without replacement from softmax(logits / T) per row (the
        Gumbel-top-k trick: the k largest logit / T + G). logits [R, V] (or [V]); row r uses counter row0 + r. Returns
        (ids by descending logit, ids in draw order), each [R, k] (or [k])."""
        lg = np.ascontiguousarray(logits, dtype=np.float64)
        one = lg.ndim == 1
        lg = lg.reshape(-1, lg.shape[-1])
        R, V = lg.shape
        ids = np.zeros((R, k), np.int32)
        drawn = np.zeros((R, k), np.int32)
        i32 = ctypes.POINTER(ctypes.c_int32)
        self.L.or_topk_sample_rows(_dp(lg), R, V, k, float(T), seed, row0, ids.ctypes.data_as(i32),
                                   drawn.ctypes.data_as(i32))
        return (ids[0], drawn[0]) if one else (ids, drawn)

    def sample_keys(self, logits, T: float, seed: int, row: int) -> np.ndarray:
        """The keys logits / T + G of topk_sample's draw for one row (the value the draw
        ranks by), [V] float64."""
        lg = np.ascontiguousarray(logits, dtype=np.float64).reshape(-1)
        key = np.zeros_like(lg)
        self.L.or_sample_keys(_dp(lg), lg.size, float(T), seed, row, _dp(key))
        return key

    def accept_sampled(self, tok, parent, depth, rank, q, p, u_acc, u_bonus, want_margin: bool = False):
        """Lossless verification of B sampled trees (Sec. 2.4; recursive rejection
        sampling over each node's children in draw order): tok, parent,
        depth, rank [B, T] int; q [B, N, V], p [B, T, V], u_acc, u_bonus [B, T] float.
        Returns (path [B, N] with -1 after the accepted nodes, n_accept [B], bonus [B]), and
        with want_margin each sequence's closest decision margin [B] (probability units)."""
        i32 = ctypes.POINTER(ctypes.c_int32)
        tok, parent, depth, rank = (np.ascontiguousarray(a, dtype=np.int32) for a in (tok, parent, depth, rank))
        q, p, u_acc, u_bonus = (np.ascontiguousarray(a, dtype=np.float64) for a in (q, p, u_acc, u_bonus))
        B, T = tok.shape
        N, V = q.shape[1], q.shape[2]
        assert p.shape == (B, T, V) and q.shape == (B, N, V) and u_acc.shape == u_bonus.shape == (B, T)
        path = np.zeros((B, N), np.int32)
        n = np.zeros(B, np.int32)
        bonus = np.zeros(B, np.int32)
        margin = np.zeros(B)
        self.L.or_accept_sampled(B, T, N, V, *(a.ctypes.data_as(i32) for a in (tok, parent, depth, rank)),
                                 _dp(q), _dp(p), _dp(u_acc), _dp(u_bonus), path.ctypes.data_as(i32),
                                 n.ctypes.data_as(i32), bonus.ctypes.data_as(i32), _dp(margin))
        return (path, n, bonus, margin) if want_margin else (path, n, bonus)

    def tree(self, N, k, root, topk):
        topk = np.ascontiguousarray(topk, dtype=np.int32).reshape(N, k)
        T = 1 + N * k
        tok = np.zeros(T, np.int32)
        par = np.zeros(T, np.int32)
        dep = np.zeros(T, np.int32)
        mask = np.zeros((T, T), np.uint8)
        i32 = ctypes.POINTER(ctypes.c_int32)
        self.L.or_tree(N, k, root, topk.ctypes.data_as(i32), tok.ctypes.data_as(i32),
                       par.ctypes.data_as(i32), dep.ctypes.data_as(i32),
                       mask.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8)))
        return tok, par, dep, mask

    def accept_greedy(self, tok, parent, depth, target_next, P: int, max_path: int):
        """Tree positions and the greedy acceptance walk of one sequence (Sec. 2.4).
        Returns (pos [T], path [max_path] with -1 after the accepted nodes, n, bonus)."""
        i32 = ctypes.POINTER(ctypes.c_int32)
        tok, parent, depth, target_next = (np.ascontiguousarray(a, dtype=np.int32) for a in
                                           (tok, parent, depth, target_next))
        T = tok.shape[0]
        pos = np.zeros(T, np.int32)
        path = np.zeros(max_path, np.int32)
        bonus = ctypes.c_int32(0)
        n = self.L.or_accept_greedy(T, tok.ctypes.data_as(i32), parent.ctypes.data_as(i32),
                                    depth.ctypes.data_as(i32), target_next.ctypes.data_as(i32), int(P),
                                    int(max_path), pos.ctypes.data_as(i32), path.ctypes.data_as(i32),
                                    ctypes.byref(bonus))
        return pos, path, int(n), int(bonus.value)

    def smooth_l1(self, x: float) -> float:
        return float(self.L.or_smooth_l1(float(x)))

    def loss(self, logits, teacher, hidden, feat, alpha: float = 0.1, beta: float = 1.0, decay: float = 0.9):
        """Training objective of Sec. 2.3 for one sequence: logits, teacher [N, V]; hidden,
        feat [N, d]. Returns (total, ce [N], feat_loss [N])."""
        logits, teacher, hidden, feat = (np.ascontiguousarray(a, dtype=np.float64) for a in
                                         (logits, teacher, hidden, feat))
        N, V = logits.shape
        d = hidden.shape[1]
        ce = np.zeros(N)
        fl = np.zeros(N)
        tot = self.L.or_loss(N, V, d, _dp(logits), _dp(teacher), _dp(hidden), _dp(feat), float(alpha), float(beta),
                             float(decay), _dp(ce), _dp(fl))
        return float(tot), ce, fl

    def max_threads(self) -> int:
        return int(self.L.or_max_threads())

    # -- whole draft ------------------------------------------------------------------
    def draft_seq(self, cfg: dict, weights: dict, feat_b, tok: int, P: int, kcs, vcs, cap: int,
                  top_k: int, temperature: float = 0.0, want_logits: bool = True,
                  rope_layer_offset: int = 0, final_norm: int = 1):
        """One sequence's draft (cfg["parallel_layers"] = 1: every layer consumes x0). ``weights`` holds host tensors in the canonical layout
        (see fe_synth.workloads); ``kcs``/``vcs`` are N host buffers of this sequence's
        [Hkv, cap, hd] cache. Returns a dict of float64 / int32 numpy arrays."""
        c = config_struct(cfg, rope_layer_offset, final_norm)
        N, d, V = cfg["n_layers"], cfg["d"], cfg["vocab"]
        ptrs = [weights["w_fuse"], weights["w_in"], weights["embed"], weights["lm_head"],
                weights["final_norm"]]
        for lw in weights["layers"]:
            ptrs += [lw["attn_norm"], lw["w_qkv"], lw["w_o"], lw["mlp_norm"], lw["w_gate"],
                     lw["w_up"], lw["w_down"]]
        warr = (_P * len(ptrs))(*[_ptr(t) for t in ptrs])
        karr = (_P * N)(*[_ptr(t) for t in kcs])
        varr = (_P * N)(*[_ptr(t) for t in vcs])
        hidden = np.zeros((N, d))
        logits = np.zeros((N, V)) if want_logits else None
        lse = np.zeros(N)
        tid = np.zeros((N, top_k), np.int32)
        tlg = np.zeros((N, top_k))
        tpr = np.zeros((N, top_k))
        rc = self.L.or_draft_seq(ctypes.byref(c), warr, _ptr(feat_b), int(tok), int(P), karr, varr,
                                 int(cap), int(top_k), float(temperature), _dp(hidden),
                                 _dp(logits) if logits is not None else None, _dp(lse),
                                 tid.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), _dp(tlg),
                                 _dp(tpr))
        if rc != 0:
            raise ValueError("oracle rejected the arguments")
        return dict(hidden=hidden, logits=logits, lse=lse, topk_id=tid, topk_logit=tlg,
                    topk_prob=tpr)

    def lm_head(self, cfg: dict, weights: dict, hidden) -> np.ndarray:
        """Logits [R, V] of R given hidden states [R, d] (Sec. 2.1: the final RMSNorm, then
        the frozen LM head), row by row through or_lm_head."""
        c = config_struct(cfg, 0, 1)
        h = np.ascontiguousarray(np.asarray(hidden, dtype=np.float64).reshape(-1, cfg["d"]))
        out = np.zeros((h.shape[0], cfg["vocab"]))
        for r in range(h.shape[0]):
            self.L.or_lm_head(ctypes.byref(c), _ptr(weights["lm_head"]), _ptr(weights["final_norm"]),
                              _dp(h[r]), _dp(out[r]))
        return out

    def layer(self, cfg: dict, lw: dict, pos: float, kc, vc, cap: int, P: int, x):
        c = config_struct(cfg, 0, 1)
        ptrs = [lw["attn_norm"], lw["w_qkv"], lw["w_o"], lw["mlp_norm"], lw["w_gate"],
                lw["w_up"], lw["w_down"]]
        warr = (_P * 7)(*[_ptr(t) for t in ptrs])
        x = np.array(x, dtype=np.float64)
        self.L.or_layer(ctypes.byref(c), warr, float(pos), _ptr(kc), _ptr(vc), cap, P, _dp(x), None, None)
        return x

    def commit_seq(self, cfg: dict, weights: dict, feats, toks, P: int, kcs, vcs, cap: int,
                   rope_layer_offset: int = 0):
        """Commit len(toks) accepted rows of one sequence at positions P, P + 1, .. (Sec. 2.4,
        "Update and Iterate"): feats [n, 3d] in the storage type, toks [n]; ``kcs``/``vcs``
        are N host buffers of this sequence's [Hkv, cap, hd] cache, written in place."""
        c = config_struct(cfg, rope_layer_offset, 1)
        N = cfg["n_layers"]
        ptrs = [weights["w_fuse"], weights["w_in"], weights["embed"], weights["lm_head"],
                weights["final_norm"]]
        for lw in weights["layers"]:
            ptrs += [lw["attn_norm"], lw["w_qkv"], lw["w_o"], lw["mlp_norm"], lw["w_gate"],
                     lw["w_up"], lw["w_down"]]
        warr = (_P * len(ptrs))(*[_ptr(t) for t in ptrs])
        karr = (_P * N)(*[_ptr(t) for t in kcs])
        varr = (_P * N)(*[_ptr(t) for t in vcs])
        toks = np.ascontiguousarray(np.asarray(toks), dtype=np.int32)
        rc = self.L.or_commit_seq(ctypes.byref(c), warr, _ptr(feats) if len(toks) else None,
                                  toks.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), len(toks), int(P),
                                  karr, varr, int(cap))
        if rc != 0:
            raise ValueError("oracle rejected the arguments")


def config_struct(cfg: dict, rope_layer_offset: int = 0, final_norm: int = 1) -> Config:
    return Config(cfg["d"], cfg["n_heads"], cfg["n_kv_heads"], cfg["head_dim"], cfg["ffn"],
                  cfg["vocab"], cfg["n_layers"], 0 if cfg["dtype"] == "f32" else 1,
                  float(cfg["rope_theta"]), float(cfg["rms_eps"]), rope_layer_offset, final_norm,
                  int(cfg.get("parallel_layers", 0)))


def load(mutant: int = 0, outdir: str | None = None) -> Oracle:
    with _lock:
        key = (mutant, outdir)
        if key not in _cache:
            _cache[key] = Oracle(build(mutant, outdir))
        return _cache[key]

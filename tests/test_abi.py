"""The C-ABI library without a GPU: it loads, exports every entry point include/*.h
declares, and rejects bad arguments on the host before touching CUDA."""
import ctypes
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = []
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        names += re.findall(r"FE_API\s+[\w\s\*]+?\b(\w+)\s*\(", src)
    return names


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    __graft_entry__.build_lib_only()
    import paper_2509_20416_gb300 as fe
    return fe


def test_header_declares_the_boundary():
    names = set(_declared())
    for n in ("fe_draft_init", "fe_draft_forward", "fe_build_tree", "fe_free", "fe_status_str",
              "fe_last_device_status"):
        assert n in names, n


def test_every_declared_symbol_is_exported(lib):
    so = ctypes.CDLL(lib.LIB_PATH)
    for n in _declared():
        assert hasattr(so, n), f"{n} declared in include/ but not exported"


def test_status_strings(lib):
    assert lib.fe_status_str(lib.FE_OK) == "ok"
    assert lib.fe_status_str(lib.FE_ERR_CAPACITY) == "prefix does not fit the cache"
    assert lib.fe_status_str(12345) == "unknown status"


def test_host_side_validation_needs_no_gpu(lib):
    so = lib._lib
    out = ctypes.c_void_p()
    # null config / weights / out pointer: rejected before any CUDA call
    assert so.fe_draft_init(None, None, None, ctypes.byref(out)) == lib.FE_ERR_INVALID_ARG
    c = lib.make_config(dict(d=256, n_heads=4, n_kv_heads=3, head_dim=64, ffn=688, vocab=4096, n_layers=3,
                             top_k_max=8, max_seq=80, rope_theta=1e4, rms_eps=1e-5, dtype="f32"))
    w = lib.fe_weights()
    assert so.fe_draft_init(ctypes.byref(c), ctypes.byref(w), None, ctypes.byref(out)) == lib.FE_ERR_INVALID_ARG
    assert out.value is None
    assert so.fe_draft_forward(None, None, None) == lib.FE_ERR_INVALID_ARG
    assert so.fe_build_tree(None, 1, 1, None, None, None, None) == lib.FE_ERR_INVALID_ARG
    assert so.fe_last_device_status(None, None) == lib.FE_ERR_INVALID_ARG
    assert so.fe_commit(None, None, None) == lib.FE_ERR_INVALID_ARG
    assert so.fe_draft_step_host(None, None, None) == lib.FE_ERR_INVALID_ARG
    assert so.fe_launch_count(None, 1, 1) == -1
    so.fe_free(None)  # no-op


def test_profile_entry_point_validates_on_host(lib):
    so = lib._lib
    n = ctypes.c_int32(0)
    assert so.fe_profile_forward(None, None, None, 8, None, None, ctypes.byref(n)) == lib.FE_ERR_INVALID_ARG
    assert so.fe_profile_graph(None, None, None, None, 8, None, None, None, ctypes.byref(n)) == lib.FE_ERR_INVALID_ARG


def test_next_row_entry_points_validate_on_host(lib):
    """The verification, loss, allocation-free LM head and timeout self-test calls reject a
    missing handle or arguments before they touch CUDA, so a bad call never launches."""
    so = lib._lib
    tree = lib.fe_tree()
    assert so.fe_verify_greedy(None, 1, 1, None, ctypes.byref(tree), None, None, None, None, None,
                               None) == lib.FE_ERR_INVALID_ARG
    assert so.fe_draft_loss(None, None, None, None, 0.1, 1.0, 0.9, None, None, None, None) == lib.FE_ERR_INVALID_ARG
    assert so.fe_verify_sampled(None, 1, 1, ctypes.byref(tree), None, None, None, None, None, None, None, None,
                                None) == lib.FE_ERR_INVALID_ARG
    assert so.fe_lm_head_topk_noalloc(None, None, 1, 1, 0.0, None, None, None, None, None) == lib.FE_ERR_INVALID_ARG
    for ns in (0, 999, 10**9 + 1):  # outside 1e3..1e9 ns, and a null handle
        assert so.fe_selftest_timeout(None, ns, None) == lib.FE_ERR_INVALID_ARG
    assert isinstance(lib.fe_last_error_detail(), str)


def test_binding_rejects_host_and_strided_buffers_before_the_library(lib):
    """The binding hands raw addresses to kernels, so it refuses a host tensor where the
    kernels read or write (fe_draft_forward, the tree, the loss, the commit, ...) and any
    non-contiguous buffer, with a ValueError and before any library call (the handle here
    is a null stand-in that the library would reject)."""
    import torch
    cfg = dict(d=8, n_layers=2, vocab=16)
    h = lib.Handle(0, cfg)
    B, k = 2, 2
    feat, tok, plen = torch.zeros(B, 24), torch.zeros(B, dtype=torch.int32), torch.zeros(B, dtype=torch.int32)
    caches = [torch.zeros(B, 1, 4, 8) for _ in range(2)]
    with pytest.raises(ValueError, match="CUDA"):
        lib.fe_draft_forward(h, feat, tok, plen, caches, caches, k)
    with pytest.raises(ValueError, match="CUDA"):
        lib.fe_build_tree(h, tok, torch.zeros(B, 2, k, dtype=torch.int32), k)
    with pytest.raises(ValueError, match="CUDA"):
        lib.fe_commit(h, torch.zeros(B, 1, 24), torch.zeros(B, 1, dtype=torch.int32), plen, plen, caches, caches)
    with pytest.raises(ValueError, match="CUDA"):
        lib.fe_lm_head_topk_noalloc(h, torch.zeros(2, B, 8), B, k)
    # fe_draft_step_host takes host inputs and outputs, but its caches are device buffers
    out = dict(topk_id=torch.zeros(B, 2, k, dtype=torch.int32), topk_logit=torch.zeros(B, 2, k),
               topk_prob=torch.zeros(B, 2, k), lse=torch.zeros(B, 2), tree_tok=torch.zeros(B, 5, dtype=torch.int32),
               tree_parent=torch.zeros(B, 5, dtype=torch.int32), tree_depth=torch.zeros(B, 5, dtype=torch.int32),
               tree_mask=torch.zeros(B, 5, 5, dtype=torch.uint8))
    with pytest.raises(ValueError, match="CUDA"):
        lib.fe_draft_step_host(h, feat, tok, plen, caches, caches, k, out=out)
    # a strided view is refused even where host memory is allowed (the weights of fe_draft_init)
    with pytest.raises(ValueError, match="contiguous"):
        lib._p(torch.zeros(4, 4).t())
    assert lib._dp(None) is None and lib._dp(0) == 0  # null and raw addresses pass through


BASE_CFG = dict(d=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=688, vocab=4096, n_layers=2, top_k_max=8,
                max_seq=80, rope_theta=1e4, rms_eps=1e-5, dtype="f32")


@pytest.mark.parametrize("change,code", [
    (dict(n_layers=0), "INVALID_ARG"), (dict(n_layers=17), "INVALID_ARG"),
    (dict(top_k_max=0), "INVALID_ARG"), (dict(top_k_max=33), "INVALID_ARG"),
    (dict(top_k_max=8, vocab=7), "INVALID_ARG"), (dict(n_kv_heads=3), "INVALID_ARG"),
    (dict(head_dim=63), "INVALID_ARG"), (dict(rope_theta=0.0), "INVALID_ARG"),
    (dict(rope_theta=float("nan")), "INVALID_ARG"), (dict(rms_eps=-1e-6), "INVALID_ARG"),
    (dict(max_batch=0), "INVALID_ARG"), (dict(max_seq=0), "INVALID_ARG"), (dict(page_size=-1), "INVALID_ARG"),
    (dict(parallel_layers=2), "INVALID_ARG"), (dict(d=0), "INVALID_ARG"),
    # legal, but outside what the kernels cover
    (dict(head_dim=96), "UNSUPPORTED"), (dict(head_dim=32), "UNSUPPORTED"),
    (dict(n_heads=6, n_kv_heads=2), "UNSUPPORTED"), (dict(n_heads=16, n_kv_heads=1), "UNSUPPORTED"),
    (dict(d=260), "UNSUPPORTED"), (dict(ffn=690), "UNSUPPORTED"),
])
def test_init_rejects_configs_before_any_cuda_call(lib, change, code):
    """fe_draft_init checks the configuration (and that every weight pointer is set) before
    it touches CUDA, so these run without a GPU: the weight pointers are non-null stand-ins
    that are never read."""
    so = lib._lib
    cfg = dict(BASE_CFG, **change)
    c = lib.make_config(cfg)
    n = max(1, min(cfg["n_layers"], 16))
    layers = (lib.fe_layer_weights * n)(*[lib.fe_layer_weights(*([8] * 7)) for _ in range(n)])
    w = lib.fe_weights(8, 8, 8, 8, 8, layers)
    out = ctypes.c_void_p()
    assert so.fe_draft_init(ctypes.byref(c), ctypes.byref(w), None, ctypes.byref(out)) == getattr(lib, "FE_ERR_" + code)
    assert out.value is None


def test_init_rejects_a_missing_layer_weight(lib):
    so = lib._lib
    c = lib.make_config(BASE_CFG)
    layers = (lib.fe_layer_weights * 2)(lib.fe_layer_weights(*([8] * 7)), lib.fe_layer_weights(*([8] * 6 + [0])))
    w = lib.fe_weights(8, 8, 8, 8, 8, layers)
    out = ctypes.c_void_p()
    assert so.fe_draft_init(ctypes.byref(c), ctypes.byref(w), None, ctypes.byref(out)) == lib.FE_ERR_INVALID_ARG
    layers[1] = lib.fe_layer_weights(*([8] * 7))
    c.dtype = 7  # neither FE_F32 nor FE_BF16
    assert so.fe_draft_init(ctypes.byref(c), ctypes.byref(w), None, ctypes.byref(out)) == lib.FE_ERR_INVALID_ARG

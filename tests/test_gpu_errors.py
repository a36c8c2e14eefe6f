"""Error behaviour of the C ABI on a GPU: host-side argument errors, device-side range
checks reported through the status word, and the bounded-wait timeout path. None of
these faults, traps or hangs the GPU: every case is detected and reported, and the
handle keeps working afterwards."""
import pytest
import torch

from fe_synth import workloads as wl
import harness as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def small():
    import paper_2509_20416_gb300 as fe
    cfg = wl.make_config(dict(d=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=512, vocab=1000, n_layers=2,
                              dtype="bf16", B=2, prefix=0, top_k=4, rope_theta=1e4, seed=9, page_size=0),
                         prefix_list=[10, 20])
    W = wl.make_weights(cfg)
    I = wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    h = fe.fe_draft_init(dict(cfg, max_batch=cfg["B"]), W)
    yield cfg, W, I, ks, vs, h
    h.close()


def _args(cfg, I, ks, vs):
    return (I["feat"].cuda(), I["next_tok"].cuda(), I["prefix_len"].cuda(), [k.cuda() for k in ks],
            [v.cuda() for v in vs])


def test_host_argument_errors(small):
    import paper_2509_20416_gb300 as fe
    cfg, W, I, ks, vs, h = small
    feat, tok, plen, kd, vd = _args(cfg, I, ks, vs)
    with pytest.raises(fe.FeError) as e:
        fe.fe_draft_forward(h, feat, tok, plen, kd, vd, top_k=cfg["top_k_max"] + 1)
    assert e.value.code == fe.FE_ERR_INVALID_ARG
    with pytest.raises(fe.FeError) as e:
        fe.fe_draft_forward(h, feat, tok, plen, kd, vd, top_k=0)
    assert e.value.code == fe.FE_ERR_INVALID_ARG
    big = torch.zeros(cfg["B"] + 1, dtype=torch.int32, device="cuda")
    with pytest.raises(fe.FeError) as e:
        fe.fe_draft_forward(h, feat, big, big, kd, vd, top_k=2)
    assert e.value.code == fe.FE_ERR_INVALID_ARG
    with pytest.raises(fe.FeError) as e:
        fe.fe_draft_forward(h, feat, tok, plen, kd[:1] + [0], vd, top_k=2)
    assert e.value.code == fe.FE_ERR_INVALID_ARG
    # unsupported head size
    with pytest.raises(fe.FeError) as e:
        fe.fe_draft_init(dict(cfg, head_dim=96, max_batch=2), W)
    assert e.value.code in (fe.FE_ERR_UNSUPPORTED, fe.FE_ERR_INVALID_ARG)
    assert fe.fe_last_device_status(h) == fe.FE_OK


def test_capacity_and_token_range_reported(small):
    import paper_2509_20416_gb300 as fe
    cfg, W, I, ks, vs, h = small
    feat, tok, plen, kd, vd = _args(cfg, I, ks, vs)
    bad = plen.clone()
    bad[1] = cfg["max_seq"]  # P + 1 > capacity
    fe.fe_draft_forward(h, feat, tok, bad, kd, vd, top_k=4)
    assert fe.fe_last_device_status(h) == fe.FE_ERR_CAPACITY
    bt = tok.clone()
    bt[0] = cfg["vocab"]
    fe.fe_draft_forward(h, feat, bt, plen, kd, vd, top_k=4)
    assert fe.fe_last_device_status(h) == fe.FE_ERR_DEVICE
    ids = torch.full((cfg["B"], cfg["n_layers"], 4), -3, dtype=torch.int32, device="cuda")
    fe.fe_build_tree(h, tok, ids, 4)
    assert fe.fe_last_device_status(h) == fe.FE_ERR_DEVICE
    # the handle still drafts correctly afterwards
    g = H.run_gpu(cfg, W, I, ks, vs, handle=h)
    assert g["status"] == fe.FE_OK


@pytest.mark.parametrize("d,n_heads,n_kv_heads,head_dim", [(256, 4, 2, 64), (512, 4, 1, 128)])
def test_bad_page_id_reported(d, n_heads, n_kv_heads, head_dim):
    """An out-of-pool page id is reported, not dereferenced (hd 128 with G = 4 runs on the
    tensor-core attention kernel, hd 64 on the CUDA-core one)."""
    import paper_2509_20416_gb300 as fe
    cfg = wl.make_config(dict(d=d, n_heads=n_heads, n_kv_heads=n_kv_heads, head_dim=head_dim, ffn=512, vocab=1000,
                              n_layers=1, dtype="bf16", B=2, prefix=0, top_k=4, rope_theta=1e4, seed=10,
                              page_size=16), prefix_list=[40, 3])
    W = wl.make_weights(cfg)
    I = wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    h = fe.fe_draft_init(dict(cfg, max_batch=2), W)
    kd, vd, table, n_pages = H.device_caches(cfg, ks, vs, I["prefix_len"])
    table[0, 1] = n_pages + 5  # points past the pool
    fe.fe_draft_forward(h, I["feat"].cuda(), I["next_tok"].cuda(), I["prefix_len"].cuda(), kd, vd, 4,
                        page_table=table, n_pages=n_pages)
    assert fe.fe_last_device_status(h) == fe.FE_ERR_DEVICE
    h.close()


def test_bounded_wait_times_out_and_gpu_stays_usable(small):
    import paper_2509_20416_gb300 as fe
    cfg, W, I, ks, vs, h = small
    assert fe.fe_selftest_timeout(h, 20_000_000) == fe.FE_OK  # 20 ms
    assert fe.fe_last_device_status(h) == fe.FE_ERR_TIMEOUT
    assert fe.fe_last_device_status(h) == fe.FE_OK  # cleared by the read
    g = H.run_gpu(cfg, W, I, ks, vs, handle=h)
    assert g["status"] == fe.FE_OK

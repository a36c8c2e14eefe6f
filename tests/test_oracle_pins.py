"""The oracle against what the paper and mathematics fix (CPU only)."""
import pytest

import oracle_pins as pins


@pytest.mark.parametrize("pin", pins.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(orc, pin):
    pin(orc)


def test_lm_head_binding_reproduces_the_draft(orc):
    """Oracle.lm_head (the LM head over given hidden rows, used to check the allocation-free
    LM head) hands or_lm_head the right buffers: on a draft's own hidden states it returns
    that draft's logits exactly, and the final norm's gain enters (a gain of 2 doubles the
    logits)."""
    import numpy as np
    import torch
    from fe_synth import workloads as wl
    cfg = wl.make_config(dict(d=64, n_heads=2, n_kv_heads=1, head_dim=32, ffn=96, vocab=300, n_layers=3,
                              dtype="bf16", B=1, prefix=5, top_k=4, rope_theta=1e4, seed=9, page_size=0))
    W, I = wl.make_weights(cfg), wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    o = orc.draft_seq(cfg, W, I["feat"][0].contiguous(), int(I["next_tok"][0]), int(I["prefix_len"][0]),
                      [k[0].contiguous() for k in ks], [v[0].contiguous() for v in vs], cfg["max_seq"], 4)
    lg = orc.lm_head(cfg, W, o["hidden"])
    assert np.array_equal(lg, o["logits"])
    W2 = dict(W, final_norm=torch.full_like(W["final_norm"], 2.0))
    assert np.allclose(orc.lm_head(cfg, W2, o["hidden"]), 2.0 * o["logits"], rtol=1e-12, atol=1e-12)


def test_sample_keys_binding_gives_the_draw_order(orc):
    """Oracle.sample_keys (the keys the parity test's near-tie exemption reads) are the keys
    topk_sample draws by: its draw order is their descending order (ties: smaller id), for
    several rows, temperatures and seeds."""
    import numpy as np
    rng = np.random.default_rng(5)
    for T, seed, row in ((1.0, 7, 0), (0.7, 123, 5), (2.5, 2**63 + 11, 41)):
        lg = rng.normal(0, 2, 777)
        keys = orc.sample_keys(lg, T, seed, row)
        ids, drawn = orc.topk_sample(lg[None, :], 12, T, seed, row0=row)
        order = sorted(range(lg.size), key=lambda v: (-keys[v], v))[:12]
        assert list(drawn[0]) == order
        assert set(ids[0]) == set(order)

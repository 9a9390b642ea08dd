"""The seeded generator: bf16 rounding matches torch's round-to-nearest-even,
draws are reproducible, shapes follow the workload table."""

import numpy as np
import torch

from oracle import v_all
from paper_2603_01639_gb300 import workload as wl


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(100000).astype(np.float32) * 7,
                        np.array([0.0, -0.0, 1.0, 1.00390625, 1.01171875, 65504.0, 1e-30], np.float32)])
    ours = wl.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)
    back = wl.bf16_bits_to_f32(ours)
    assert np.array_equal(back, torch.from_numpy(x).to(torch.bfloat16).float().numpy())


def test_draws_are_seeded_and_shaped():
    cfg = wl.config("tiny")
    a = wl.draw_cycle(cfg, 3)
    b = wl.draw_cycle(cfg, 3)
    assert np.array_equal(a.draft_rows, b.draft_rows) and a.root.tolist() == b.root.tolist()
    assert a.draft_rows.shape == (1, 1 + (3 - 1) * 2, 1000)
    assert cfg.max_n <= v_all(cfg.W, cfg.depth_range[0])
    c = wl.config("70b")
    ci = wl.draw_cycle(c, 1, draft_rows=False)
    assert ci.ctx.min() >= 1024 and ci.ctx.max() <= 8192
    assert set(ci.mode.tolist()) <= {0, 1}
    assert ((ci.n_verify >= 32) & (ci.n_verify <= 96)).all()
    assert (ci.n_verify <= np.array([v_all(c.W, int(L)) for L in ci.depth])).all()


def test_every_config_fits_its_tree():
    for name, cfg in wl.CONFIGS.items():
        assert cfg.max_n <= v_all(cfg.W, cfg.depth_range[0]), name
        assert cfg.s_cap >= cfg.max_ctx + cfg.max_n and cfg.s_cap % 128 == 0

"""The RL environment (section 3.1): the throughput reward on the host, and
on the GPU whole episodes checked against the oracle cycle with the same
depth and size decisions."""
import numpy as np
import pytest
import torch

import oracle
from paper_2603_01639_gb300 import env, ltd
from paper_2603_01639_gb300 import workload as wl

from . import harness as H


def test_throughput_reward_counts_the_bonus_token():
    # L_A = accepted draft tokens + 1; T in seconds -> tokens per second
    r = env.throughput_reward([0, 3], 1e-4, 3e-4)
    np.testing.assert_allclose(r, [1 / 4e-4, 4 / 4e-4])


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the no-GPU failure")
def test_env_refuses_to_run_without_a_gpu():
    with pytest.raises(ltd.LtdError):
        env.CycleEnv("tiny")


@pytest.mark.gpu
@pytest.mark.parametrize("name,seed", [("tiny", 0), ("70b", 2)])
def test_env_episode_matches_the_oracle_cycle(name, seed):
    from paper_2603_01639_gb300 import build
    build.build()
    cfg = wl.config(name)
    e = env.CycleEnv(name, layers=2, seed=seed)
    rng = np.random.default_rng(seed + 5)
    for episode in range(2):
        obs = e.reset()
        ci = e.ci
        assert obs.shape == (cfg.batch, cfg.W * cfg.W + 2)
        drafting = True
        while drafting:
            cont = rng.random(cfg.batch) < 0.7
            obs, drafting = e.step_depth(cont)
        sobs = e.size_observation()
        levels = e.tree.view()["n_levels"].cpu().numpy()
        assert levels.min() >= 1 and levels.max() <= cfg.max_depth
        trees = [oracle.grow_tree(int(ci.root[b]), ci.draft_rows[b], cfg.W, int(levels[b]))
                 for b in range(cfg.batch)]
        for b, t in enumerate(trees):
            ref = oracle.size_observation(t, int(ci.ctx[b]), e.v_pad)
            assert np.abs(sobs[b] - ref).max() <= H.CUM_TOL * max(1.0, np.abs(ref).max())
        n = np.array([min(cfg.max_n, t.n_nodes, int(rng.integers(1, cfg.max_n + 1))) for t in trees])
        reward, info = e.step_size(n)
        np.testing.assert_array_equal(info["levels"], levels)
        sels = [oracle.select_verify(t, int(n[b]), int(ci.ctx[b])) for b, t in enumerate(trees)]
        for b in range(cfg.batch):
            np.testing.assert_array_equal(info["ids"][b, :n[b]], sels[b][0])
        ci.depth, ci.n_verify = levels.astype(np.int32), n.astype(np.int32)
        assert min(H.tree_margin(t, cfg.W) for t in trees) > H.CUT_MARGIN
        ref = H.oracle_accept(cfg, ci, trees, sels, e.last_target, e.acc_seed, e.cycle_no)
        assert H.stochastic_margins_ok(ref), "near-tie in a stochastic decision; pick another seed"
        for b in range(cfg.batch):
            assert info["accept_len"][b] == ref[b]["accept_len"]
            assert info["bonus"][b] == ref[b]["bonus"]
            a = ref[b]["accept_len"]
            np.testing.assert_array_equal(info["path"][b, :a + 1], ref[b]["path"])
        assert info["t_draft_s"] > 0 and info["t_verify_s"] > 0
        np.testing.assert_allclose(
            reward, (info["accept_len"] + 1) / (info["t_draft_s"] + info["t_verify_s"]), rtol=1e-12)

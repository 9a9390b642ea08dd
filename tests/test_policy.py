"""Host policies (section 3.1, Appendix A/B): shapes of the paper's MLPs, the
action ranges, and seeded determinism.  No GPU."""
import numpy as np

from paper_2603_01639_gb300 import policy


def test_depth_policy_shapes_and_actions():
    k = 10
    p = policy.DepthPolicy(k, seed=3)
    dims = [w.shape for w, _ in p.net.layers]
    assert dims == [(k * k + 2, 1024), (1024, 2)]          # one hidden layer of 1024
    rng = np.random.default_rng(0)
    obs = np.concatenate([rng.normal(-5, 2, (4, k * k)), [[3, 4096]] * 4], axis=1)
    a = p.decide(obs)
    assert a.shape == (4,) and a.dtype == bool
    assert np.array_equal(a, policy.DepthPolicy(k, seed=3).decide(obs))


def test_size_policy_shapes_and_range():
    v_pad = 1 + 10 + 5 * 100
    p = policy.SizePolicy(v_pad, seed=4)
    dims = [w.shape for w, _ in p.net.layers]
    assert dims == [(v_pad + 2, 1024), (1024, 256), (256, 12)]   # [1024, 256] hidden, 12 actions
    rng = np.random.default_rng(1)
    obs = np.concatenate([rng.normal(-8, 3, (5, v_pad)), [[6, 2048]] * 5], axis=1)
    n = p.decide(obs)
    assert n.dtype == np.int32 and n.shape == (5,)
    assert ((n >= 20) & (n <= 240) & (n % 20 == 0)).all()
    assert np.array_equal(n, policy.SizePolicy(v_pad, seed=4).decide(obs))


def test_mlp_is_the_plain_relu_network():
    net = policy.MLP(3, (4,), 2, seed=0)
    x = np.array([[1.0, -2.0, 0.5]], np.float32)
    (w1, b1), (w2, b2) = net.layers
    ref = np.maximum(x @ w1 + b1, 0) @ w2 + b2
    assert np.allclose(net.forward(x), ref)


def test_size_actions_map_linearly_onto_20_to_240():
    p = policy.SizePolicy(8, seed=0)
    w, b = p.net.layers[-1]
    obs = np.zeros((1, 10), np.float32)
    got = []
    for a in range(12):                 # force each action through the output bias
        b[:] = 0.0
        w[:] = 0.0
        b[a] = 1.0
        got.append(int(p.decide(obs)[0]))
    assert got == list(range(20, 241, 20))


def test_verify_size_counts_the_root_and_respects_the_caps():
    p = policy.SizePolicy(8, seed=0)
    w, b = p.net.layers[-1]
    w[:] = 0.0
    b[:] = 0.0
    b[2] = 1.0                                    # action 2: V = 60
    obs = np.zeros((3, 10), np.float32)
    n = p.verify_size(obs, n_cap=64, n_nodes=[511, 30, 511])
    assert n.tolist() == [61, 30, 61]
    assert p.verify_size(obs, n_cap=48, n_nodes=[511, 511, 511]).tolist() == [48, 48, 48]


def test_host_policies_match_the_oracle_network():
    """The host (numpy fp32) policies against the oracle's fp64 network on
    the same observations: logits within the fp32 accumulation bound,
    decisions equal wherever the fp64 top-two gap is clear of it."""
    import oracle
    rng = np.random.default_rng(11)
    k, v_pad = 10, 1 + 10 + 5 * 100
    dp, sp = policy.DepthPolicy(k, seed=5), policy.SizePolicy(v_pad, seed=6)
    for pol, n_in in ((dp, k * k + 2), (sp, v_pad + 2)):
        obs = np.concatenate([rng.normal(-8, 3, (16, n_in - 2)),
                              np.stack([rng.integers(1, 9, 16), rng.integers(512, 8192, 16)], 1)],
                             axis=1).astype(np.float32)
        got = pol.net.forward(obs)
        ref = oracle.mlp_forward(obs, pol.net.layers)
        h = np.abs(obs.astype(np.float64))
        for w, b in pol.net.layers:
            h = h @ np.abs(w.astype(np.float64)) + np.abs(b.astype(np.float64))
        tol = 1e-5 * h + 1e-6
        assert (np.abs(got - ref) <= tol).all()
        top2 = np.sort(ref, axis=1)[:, -2:]
        clear = (top2[:, 1] - top2[:, 0]) > 2 * tol.max(axis=1)
        assert clear.sum() >= 8, "too many near-ties to check decisions; pick another seed"
        np.testing.assert_array_equal(np.argmax(got, axis=1)[clear], np.argmax(ref, axis=1)[clear])


def test_device_policy_bindings_check_their_buffers_on_the_host():
    """Wrong buffers are refused by the binding before any launch (CPU
    tensors, wrong dtype or size), so no device call is made."""
    import pytest
    import torch

    from paper_2603_01639_gb300 import ltd
    with pytest.raises(ltd.LtdError):
        ltd._need_vec(torch.zeros(4, dtype=torch.int32), "x", 4, torch.int32)   # not on a GPU
    with pytest.raises(ltd.LtdError):
        ltd._need(torch.zeros(4, dtype=torch.float32), "x", torch.int32)

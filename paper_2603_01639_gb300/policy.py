"""Host-side policies of LTD (section 3.1; Appendix A and B): lightweight MLPs
that read the device-gathered observations and choose the draft depth (the
depth policy, one continue/stop decision per level) and the verify size N
(the size policy, N in [20, 240] in 12 steps).

Architectures follow the paper: the depth policy has one hidden layer of
1024 ReLU units and two actions; the size policy has hidden layers of 1024
and 256 ReLU units and 12 actions mapped linearly onto N = 20, 40, ..., 240
(Appendix A.2, "Size Policy", action space).  No trained weights
exist here: the weights are seeded random (He-normal), which fixes the
shapes and the cost of a decision, not its quality.  The observation's D
and L entries are brought to O(1) by the first layer's weights (their rows
are scaled by 1/16 and 1/8192), so the network reads the observation as the
library gathers it.  Each policy runs either on the host (numpy fp32,
``decide``) or on the device (``device()`` gives the weights to
``ltd_depth_policy`` / ``ltd_size_policy``; same network, fp32).
"""
from __future__ import annotations

import numpy as np

N_MIN, N_MAX, N_ACTIONS = 20, 240, 12
N_STEP = (N_MAX - N_MIN) // (N_ACTIONS - 1)   # 20


def _dense(rng: np.random.Generator, n_in: int, n_out: int):
    w = rng.standard_normal((n_in, n_out), dtype=np.float32) * np.float32(np.sqrt(2.0 / n_in))
    return w, np.zeros(n_out, np.float32)


class MLP:
    """ReLU MLP with seeded random weights; forward(x [B][n_in]) -> logits.
    ``in_scale`` [n_in] scales the first layer's rows (input normalisation
    folded into the weights)."""

    def __init__(self, n_in: int, hidden: tuple, n_out: int, seed: int, in_scale=None):
        rng = np.random.default_rng(seed)
        dims = (n_in,) + tuple(hidden) + (n_out,)
        self.layers = [_dense(rng, a, b) for a, b in zip(dims[:-1], dims[1:])]
        if in_scale is not None:
            w0, b0 = self.layers[0]
            self.layers[0] = (w0 * np.asarray(in_scale, np.float32)[:, None], b0)

    def device(self, device="cuda", packed=True):
        """The same weights on the device, for ltd_depth_policy / ltd_size_policy
        (packed into the library's streaming layout unless ``packed`` is False)."""
        from . import ltd
        return ltd.MlpNet(self.layers, device, packed=packed)

    def forward(self, x: np.ndarray) -> np.ndarray:
        h = np.asarray(x, np.float32)
        for i, (w, b) in enumerate(self.layers):
            h = h @ w + b
            if i + 1 < len(self.layers):
                h = np.maximum(h, 0.0)
        return h


def _obs_scale(n_in: int) -> np.ndarray:
    """Scores as they are; D and L (the last two entries) scaled to O(1)."""
    s = np.ones(n_in, np.float32)
    s[-2] = 1.0 / 16.0
    s[-1] = 1.0 / 8192.0
    return s


class DepthPolicy:
    """pi_D: observation [B][k*k + 2] -> continue drafting (bool [B])."""

    def __init__(self, k: int, seed: int = 0):
        self.net = MLP(k * k + 2, (1024,), 2, seed, _obs_scale(k * k + 2))

    def decide(self, obs: np.ndarray) -> np.ndarray:
        return np.argmax(self.net.forward(obs), axis=1) == 1


class SizePolicy:
    """pi_V: observation [B][v_pad + 2] -> candidate count V in {20, 40, ...,
    240} ([B]); ``verify_size`` turns it into the verify size N the library
    takes (root included), as ltd_size_policy does on the device."""

    def __init__(self, v_pad: int, seed: int = 1):
        self.net = MLP(v_pad + 2, (1024, 256), N_ACTIONS, seed, _obs_scale(v_pad + 2))

    def decide(self, obs: np.ndarray) -> np.ndarray:
        a = np.argmax(self.net.forward(obs), axis=1).astype(np.int32)
        return (N_MIN + N_STEP * a).astype(np.int32)

    def verify_size(self, obs: np.ndarray, n_cap: int, n_nodes) -> np.ndarray:
        """N = min(1 + V, n_cap, nodes in the tree) per sequence."""
        v = self.decide(obs)
        return np.minimum(np.minimum(1 + v, n_cap), np.asarray(n_nodes)).astype(np.int32)

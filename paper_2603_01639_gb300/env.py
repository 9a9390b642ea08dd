"""The reinforcement-learning environment of LTD (section 3.1), on the device.

An episode is one draft-and-verify cycle of a batch of sequences.  After
every draft level the depth policy's observation comes back and the caller
decides, per sequence, whether drafting continues (the binary action of the
depth policy); once no sequence continues, the size policy's observation
comes back and the caller picks the verify size N per sequence (the size
policy's action).  The environment then verifies (selection, tree attention
in every layer, acceptance with KV compaction) and returns the reward of
section 3.1, the cycle's throughput

    R = L_A / (T_draft + T_verify),

with L_A = accepted draft tokens + 1 (the bonus token: the tokens the cycle
emits) and T_draft, T_verify the device time of the draft-tree phase and of
the verification phase, measured with CUDA events around the library's
launches.  The draft and target models are not run: the draft logits, q/K/V
and target logits are the seeded synthetic workloads (the target agreeing
with the draft by the workload's planting rule), so T covers the cycle's own
kernels, not the models' forward passes.  PPO itself is not part of this
module; it only supplies (observation, action, reward) transitions.

Every step runs in the library's CUDA kernels (``ltd``); there is no host
fallback.
"""
from __future__ import annotations

import numpy as np
import torch

from . import ltd
from . import workload as wl


def throughput_reward(accept_len, t_draft_s, t_verify_s):
    """R = L_A / (T_draft + T_verify) in tokens per second, L_A = accepted
    draft tokens + the bonus token (section 3.1)."""
    return (np.asarray(accept_len, np.float64) + 1.0) / (float(t_draft_s) + float(t_verify_s))


class CycleEnv:
    """Draft-and-verify cycles of one synthetic workload as RL episodes."""

    def __init__(self, config: str = "8b", layers: int | None = None, seed: int = 0,
                 device="cuda", acc_seed: int = 1234):
        if not torch.cuda.is_available():
            raise ltd.LtdError("CycleEnv needs a CUDA device")
        self.cfg = cfg = wl.config(config)
        self.layers = cfg.layers if layers is None else layers
        self.device = torch.device(device)
        self.seed, self.acc_seed, self.cycle_no = seed, acc_seed, 0
        self.tdt = torch.bfloat16 if cfg.dtype == wl.BF16 else torch.float32
        B, d = cfg.batch, cfg.head_dim
        dev = self.device
        self.tree = ltd.Tree(B, cfg.max_depth, cfg.W, cfg.vocab, device=dev)
        g = torch.Generator(device=dev).manual_seed(seed)
        self.q = [torch.randn(B, cfg.max_n, cfg.hq, d, generator=g, device=dev).to(self.tdt)
                  for _ in range(self.layers)]
        self.k = [torch.randn(B, cfg.hkv, cfg.s_cap, d, generator=g, device=dev).to(self.tdt)
                  for _ in range(self.layers)]
        self.v = [torch.randn(B, cfg.hkv, cfg.s_cap, d, generator=g, device=dev).to(self.tdt)
                  for _ in range(self.layers)]
        self.kv = ltd.KVCache(self.k, self.v)
        self.out = torch.zeros(B, cfg.max_n, cfg.hq, d, dtype=self.tdt, device=dev)
        self.att_ws = ltd.attention_workspace(B, cfg.hq, cfg.hkv, d, cfg.max_n, cfg.max_ctx,
                                              self.tdt, dev)
        self.acc_ws = ltd.accept_workspace(B, cfg.max_n, cfg.vocab, dev)
        self.v_pad = self.tree.max_nodes
        self._ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
        self.ci = None

    # ------------------------------------------------------------ helpers
    def _i32(self, x):
        return torch.as_tensor(np.asarray(x, np.int32), device=self.device)

    def _timed(self, fn):
        """Run fn on the current stream; its device time in seconds."""
        s = torch.cuda.current_stream(self.device)
        self._ev[0].record(s)
        fn()
        self._ev[1].record(s)
        self._ev[1].synchronize()
        return self._ev[0].elapsed_time(self._ev[1]) * 1e-3

    # ------------------------------------------------------------- episode
    def reset(self, seed: int | None = None) -> np.ndarray:
        """Draw a cycle, build draft level 1 and return the depth policy's
        observation [B][k*k + 2]."""
        cfg = self.cfg
        self.cycle_no += 1
        s = self.seed + self.cycle_no if seed is None else seed
        ci = wl.draw_cycle(cfg, s)
        self.ci = ci
        self.draft = torch.from_numpy(ci.draft_rows).to(self.device).to(self.tdt)
        self.root, self.ctx, self.mode = self._i32(ci.root), self._i32(ci.ctx), self._i32(ci.mode)
        self.active = np.ones(cfg.batch, bool)
        self.t_draft = self._timed(lambda: (ltd.ltd_tree_reset(self.tree, self.root),
                                            ltd.ltd_expand_tree(self.tree, 1, self.draft)))
        self.levels = 1
        return ltd.ltd_depth_observation(self.tree, self.ctx).cpu().numpy()

    def step_depth(self, cont) -> tuple[np.ndarray, bool]:
        """Apply the depth decisions (True = continue drafting) and build the
        next level for the sequences that continue.  Returns the depth
        observation (a stopped sequence keeps reporting its last level) and
        whether any sequence is still drafting."""
        if self.ci is None:
            raise RuntimeError("reset() starts an episode")
        cont = np.asarray(cont, bool).reshape(-1)
        if cont.shape[0] != self.cfg.batch:
            raise ValueError("one depth decision per sequence")
        self.active &= cont
        if self.levels >= self.cfg.max_depth:
            self.active[:] = False
        if self.active.any():
            self.levels += 1
            act = self._i32(self.active.astype(np.int32))
            lv = self.levels
            self.t_draft += self._timed(lambda: ltd.ltd_expand_tree(self.tree, lv, self.draft,
                                                                    active=act))
        obs = ltd.ltd_depth_observation(self.tree, self.ctx).cpu().numpy()
        return obs, bool(self.active.any())

    def size_observation(self) -> np.ndarray:
        """The size policy's observation [B][v_pad + 2] of the finished tree."""
        return ltd.ltd_size_observation(self.tree, self.ctx, self.v_pad).cpu().numpy()

    def step_size(self, n_verify):
        """Verify N_b nodes per sequence (root included) and return the reward
        [B] (tokens per second) and an info dict."""
        cfg, ci = self.cfg, self.ci
        if ci is None:
            raise RuntimeError("reset() starts an episode")
        view = {k: v.cpu().numpy() for k, v in self.tree.view().items()}
        n = np.asarray(n_verify, np.int64).reshape(-1)
        if n.shape[0] != cfg.batch or (n < 1).any() or (n > cfg.max_n).any() or \
                (n > view["n_nodes"]).any():
            raise ValueError("N must lie in [1, min(n_max, tree size)] for every sequence")
        n_dev = self._i32(n)
        sel = {}
        t_sel = self._timed(lambda: sel.update(zip(("ids", "pos", "mask"), ltd.ltd_select_verify(
            self.tree, n_dev, cfg.max_n, self.ctx))))
        # target logits agreeing with the draft on the verified tree (the
        # target model's output; an input here, outside the timed phases)
        ids = sel["ids"].cpu().numpy()
        target = wl.draw_target_rows(cfg, ci)
        rng = np.random.default_rng(ci.seed + 99)
        for b in range(cfg.batch):
            wl.plant_agreement(cfg, target[b], ids[b, :n[b]], view["parent"][b], view["token"][b],
                               view["depth"][b], rng, greedy=(ci.mode[b] == 0))
        self.last_target = target
        tgt = torch.from_numpy(target).to(self.device).to(self.tdt)
        acc = {}

        def verify():
            for l in range(self.layers):
                ltd.ltd_tree_attention(self.q[l], self.k[l], self.v[l], self.ctx, cfg.max_ctx, n_dev,
                                       sel["mask"], out=self.out, workspace=self.att_ws)
            acc.update(ltd.ltd_accept(self.tree, tgt, self.draft, sel["ids"], n_dev, self.mode,
                                      self.ctx, seed=self.acc_seed, cycle=self.cycle_no, kv=self.kv,
                                      workspace=self.acc_ws))

        t_verify = t_sel + self._timed(verify)
        ltd.ltd_check()
        a = acc["accept_len"].cpu().numpy()
        reward = throughput_reward(a, self.t_draft, t_verify)
        self.ci = None  # the episode is over
        info = {"accept_len": a, "bonus": acc["bonus"].cpu().numpy(),
                "path": acc["path"].cpu().numpy(), "levels": view["n_levels"].copy(),
                "n_verify": n.astype(np.int32), "ids": ids,
                "t_draft_s": self.t_draft, "t_verify_s": t_verify}
        return reward, info

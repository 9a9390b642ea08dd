"""Runs one draft-and-verify cycle through the C ABI (GPU) and through the
oracle (CPU) on the same seeded inputs, and compares them.

Bars: integers (tree structure, frontier, selected ids, positions, masks,
paths, accept lengths, bonus tokens, compacted rows) bit-exact; cum_logprob
within 1e-4 * max(1, |ref|); bf16 attention within max-abs 2e-2 and mean-abs
2e-3, fp32 attention within 1e-4.  Decisions the oracle flags as near-ties
(fp64 gap below the margins here) are reported instead of compared.
"""

from __future__ import annotations

import math

import numpy as np
import torch

import oracle
from paper_2603_01639_gb300 import ltd
from paper_2603_01639_gb300 import workload as wl

TORCH_DT = {wl.F32: torch.float32, wl.BF16: torch.bfloat16}
CUT_MARGIN = 1e-5        # frontier / selection cut gap (fp64 cum units)
RATIO_MARGIN = 1e-4      # relative gap of a stochastic ratio test
GUMBEL_MARGIN = 1e-4     # gap between the two best Gumbel scores
CUM_TOL = 1e-4
ATT_TOL = {wl.BF16: (2e-2, 2e-3), wl.F32: (1e-4, 1e-5)}


def dev(x: np.ndarray, dtype: str) -> torch.Tensor:
    """Exact transfer: values are representable in ``dtype``."""
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).cuda().to(TORCH_DT[dtype])


def i32(x) -> torch.Tensor:
    return torch.as_tensor(np.asarray(x, dtype=np.int32)).cuda()


# ---------------------------------------------------------------- oracle side
def oracle_side(cfg: wl.Config, ci: wl.CycleInputs, plant_seed: int = 99):
    """Trees, selections and (planted) target rows from the oracle."""
    trees, sels = [], []
    for b in range(cfg.batch):
        t = oracle.grow_tree(int(ci.root[b]), ci.draft_rows[b], cfg.W, int(ci.depth[b]))
        trees.append(t)
        sels.append(oracle.select_verify(t, int(ci.n_verify[b]), int(ci.ctx[b])))
    target = wl.draw_target_rows(cfg, ci)
    rng = np.random.default_rng(ci.seed + plant_seed)
    for b in range(cfg.batch):
        ids = sels[b][0]
        wl.plant_agreement(cfg, target[b], ids, trees[b].parent, trees[b].token, trees[b].depth,
                           rng, greedy=(ci.mode[b] == 0))
    return trees, sels, target


def oracle_accept(cfg, ci, trees, sels, target, seed, cycle_no):
    res = []
    for b in range(cfg.batch):
        ids = sels[b][0]
        N = int(ci.n_verify[b])
        rows = target[b, :N].astype(np.float64)
        if ci.mode[b] == 0:
            path, a, bonus = oracle.accept_greedy(trees[b], ids, rows)
            margins = []
        else:
            path, a, bonus, margins = oracle.accept_stochastic(
                trees[b], ids, rows, ci.draft_rows[b].astype(np.float64), seed, b, cycle_no)
        res.append(dict(path=path, accept_len=a, bonus=bonus, margins=margins,
                        new_ctx=int(ci.ctx[b]) + 1 + a))
    return res


# ------------------------------------------------------------------- GPU side
def gpu_draft(cfg: wl.Config, ci: wl.CycleInputs, draft: torch.Tensor, tree=None):
    B = cfg.batch
    if tree is None:
        tree = ltd.Tree(B, cfg.max_depth, cfg.W, cfg.vocab)
    ltd.ltd_tree_reset(tree, i32(ci.root))
    depth = np.asarray(ci.depth)
    for level in range(1, int(depth.max()) + 1):
        active = None if (depth >= level).all() else i32((depth >= level).astype(np.int32))
        ltd.ltd_expand_tree(tree, level, draft, active=active)
    return tree


def gpu_select(cfg, ci, tree):
    return ltd.ltd_select_verify(tree, i32(ci.n_verify), cfg.max_n, i32(ci.ctx))


# ----------------------------------------------------------------- comparisons
def compare_trees(cfg, ci, tree, trees):
    """Bit-exact structure, cum within tolerance; returns worst cut margin."""
    v = {k: t.cpu().numpy() for k, t in tree.view().items()}
    worst = math.inf
    for b in range(cfg.batch):
        t = trees[b]
        n = t.n_nodes
        assert n == oracle.v_all(cfg.W, int(ci.depth[b]))
        if t.cut_margins:
            worst = min(worst, min(t.cut_margins))
        assert v["n_nodes"][b] == n, (b, v["n_nodes"][b], n)
        assert v["n_levels"][b] == int(ci.depth[b])
        np.testing.assert_array_equal(v["token"][b, :n], np.array(t.token), err_msg=f"token b={b}")
        np.testing.assert_array_equal(v["parent"][b, :n], np.array(t.parent), err_msg=f"parent b={b}")
        np.testing.assert_array_equal(v["depth"][b, :n], np.array(t.depth), err_msg=f"depth b={b}")
        np.testing.assert_array_equal(v["frontier"][b], np.array(t.frontier), err_msg=f"frontier b={b}")
        np.testing.assert_array_equal(v["xrow"][b, :n], np.array(t.xrow), err_msg=f"xrow b={b}")
        ref = np.array(t.cum)
        err = np.abs(v["cum_logprob"][b, :n] - ref) / np.maximum(1.0, np.abs(ref))
        assert err.max() <= CUM_TOL, (b, err.max())
        expanded = np.array(t.xrow) >= 0
        xerr = np.abs(v["xlse"][b, :n][expanded] - np.array(t.xlse)[expanded])
        assert xerr.max() <= CUM_TOL * max(1.0, np.abs(np.array(t.xlse)).max()), xerr.max()
    return worst


def compare_select(cfg, ci, got, sels):
    ids, pos, mask = (x.cpu().numpy() for x in got)
    W32 = (cfg.max_n + 31) // 32
    worst = math.inf
    for b in range(cfg.batch):
        rids, rpos, rmask, margin = sels[b]
        worst = min(worst, margin)
        N = len(rids)
        np.testing.assert_array_equal(ids[b, :N], rids, err_msg=f"ids b={b}")
        np.testing.assert_array_equal(pos[b, :N], rpos, err_msg=f"pos b={b}")
        assert (ids[b, N:] == -1).all() and (pos[b, N:] == -1).all()
        words = oracle.mask_words(rmask)
        full = np.zeros((cfg.max_n, W32), np.uint32)
        full[:N, :words.shape[1]] = words
        np.testing.assert_array_equal(mask[b].view(np.uint32), full, err_msg=f"mask b={b}")
    return worst


def compare_accept(cfg, got, ref):
    g = {k: t.cpu().numpy() for k, t in got.items()}
    for b in range(cfg.batch):
        r = ref[b]
        a = r["accept_len"]
        assert g["accept_len"][b] == a, (b, g["accept_len"][b], a)
        np.testing.assert_array_equal(g["path"][b, :a + 1], np.array(r["path"]), err_msg=f"path b={b}")
        assert (g["path"][b, a + 1:] == -1).all()
        assert g["bonus"][b] == r["bonus"], (b, g["bonus"][b], r["bonus"])
        assert g["new_ctx"][b] == r["new_ctx"]


def stochastic_margins_ok(ref) -> bool:
    for r in ref:
        m = r["margins"]
        if not m:
            continue
        if min(m[:-1], default=math.inf) < RATIO_MARGIN or m[-1] < GUMBEL_MARGIN:
            return False
    return True


def attention_error(got: np.ndarray, ref: np.ndarray):
    d = np.abs(got.astype(np.float64) - ref)
    return float(d.max()), float(d.mean())

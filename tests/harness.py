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


def oracle_accept(cfg, ci, trees, sels, target, seed, cycle_no, temperature=1.0):
    res = []
    for b in range(cfg.batch):
        ids = sels[b][0]
        N = int(ci.n_verify[b])
        rows = target[b, :N].astype(np.float64)
        if ci.mode[b] == 0:
            path, a, bonus = oracle.accept_greedy(trees[b], ids, rows)
            margins = []
        elif ci.mode[b] == 2:
            path, a, bonus, margins = oracle.accept_point_mass(trees[b], ids, rows, seed, b, cycle_no,
                                                               temperature)
        elif ci.mode[b] == 3:
            path, a, bonus, margins = oracle.accept_without_replacement(
                trees[b], ids, rows, ci.draft_rows[b].astype(np.float64), seed, b, cycle_no,
                temperature)
        else:
            path, a, bonus, margins = oracle.accept_stochastic(
                trees[b], ids, rows, ci.draft_rows[b].astype(np.float64), seed, b, cycle_no,
                temperature)
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
def _adjacent_gaps(t, ids):
    """fp64 gaps between neighbours of ``ids`` sorted by (cum desc, id asc).
    A zero gap between siblings is an exact tie (same parent, same logit):
    both sides hold bit-identical values and break it by id, so it is not a
    near-tie and is skipped."""
    order = sorted(ids, key=lambda i: (-t.cum[i], i))
    gaps = []
    for a, c in zip(order, order[1:]):
        g = t.cum[a] - t.cum[c]
        if g == 0.0 and t.parent[a] == t.parent[c]:
            continue
        gaps.append(g)
    return gaps


def tree_margin(t, W) -> float:
    """Smallest gap that decides a frontier (its membership and its rank
    order, which picks the next level's draft rows)."""
    worst = math.inf
    for lvl in range(2, t.levels + 1):
        pool = [i for i in range(t.n_nodes) if t.depth[i] == lvl]
        top = sorted(pool, key=lambda i: (-t.cum[i], i))[:W + 1]
        worst = min([worst] + _adjacent_gaps(t, top))
    return worst


def select_margin(t, N) -> float:
    """Gap at the selection cut (last verified vs first left out)."""
    rest = sorted(range(1, t.n_nodes), key=lambda i: (-t.cum[i], i))
    if N - 1 >= len(rest) or N < 2:
        return math.inf
    return min([math.inf] + _adjacent_gaps(t, rest[N - 2:N]))


def compare_trees(cfg, ci, tree, trees):
    """Bit-exact structure, cum within tolerance; returns worst cut margin."""
    v = {k: t.cpu().numpy() for k, t in tree.view().items()}
    worst = math.inf
    for b in range(cfg.batch):
        t = trees[b]
        n = t.n_nodes
        assert n == oracle.v_all(cfg.W, int(ci.depth[b]))
        worst = min(worst, tree_margin(t, cfg.W))
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


def compare_select(cfg, ci, got, sels, trees):
    ids, pos, mask = (x.cpu().numpy() for x in got)
    W32 = (cfg.max_n + 31) // 32
    worst = math.inf
    for b in range(cfg.batch):
        rids, rpos, rmask, _ = sels[b]
        worst = min(worst, select_margin(trees[b], int(ci.n_verify[b])))
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

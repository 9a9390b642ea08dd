"""ltd_lm_head_row_stats against the oracle's lm_head_row_stats.

The target's LM head over the verified tokens (paper section 3.2, "Draft
Tree Verification") with the statistics acceptance reads fused into the
GEMM: per row the max, the log-sum-exp and the argmax (ties to the lower
token id).  Inputs are seeded and synthetic: hidden states N(0, 1) and a
weight N(0, 1 / hidden), both rounded to bf16, so the logits are O(1) like
a language model's.  The kernel accumulates in fp32 from bf16 inputs; the
oracle in fp64 from the same bf16 values.  Row max and log-sum-exp must
agree within 1e-4 relative to max(1, |ref|); the argmax bit for bit on rows
whose fp64 top-two gap is clear of fp32 accumulation error (1e-3, at least
90% of the rows), and on the other rows one of the tokens within that gap of
the max; logits, when asked for, within bf16 rounding of the fp64 value.
"""

import numpy as np
import pytest
import torch

import oracle
from paper_2603_01639_gb300 import ltd
from paper_2603_01639_gb300 import workload as wl

pytestmark = pytest.mark.gpu

STAT_TOL = 1e-4
ARGMAX_GAP = 1e-3


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2603_01639_gb300 import build
    build.build()
    ltd.lib()


def _draw(rows, vocab, hidden, seed):
    rng = np.random.default_rng(seed)
    h = wl.round_to(rng.standard_normal((rows, hidden), dtype=np.float32), wl.BF16)
    w = wl.round_to(rng.standard_normal((vocab, hidden), dtype=np.float32)
                    * np.float32(1.0 / np.sqrt(hidden)), wl.BF16)
    return h, w


def _dev(x):
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).cuda().to(torch.bfloat16)


def _check(h, w, logits=False, check_gap=True):
    got = ltd.ltd_lm_head_row_stats(_dev(h), _dev(w), logits=logits)
    assert ltd.ltd_check() == 0
    ref_logits, mx, lse, am = oracle.lm_head_row_stats(h, w)
    gmx = got["row_max"].cpu().numpy().astype(np.float64)
    glse = got["row_lse"].cpu().numpy().astype(np.float64)
    gam = got["row_argmax"].cpu().numpy()
    assert np.all(np.abs(gmx - mx) <= STAT_TOL * np.maximum(1.0, np.abs(mx))), np.abs(gmx - mx).max()
    assert np.all(np.abs(glse - lse) <= STAT_TOL * np.maximum(1.0, np.abs(lse))), np.abs(glse - lse).max()
    if check_gap:
        # rows whose fp64 top two are within fp32 accumulation error of each
        # other may pick either: there the kernel's token must be one of them
        top2 = np.sort(ref_logits, axis=1)[:, -2:]
        clear = (top2[:, 1] - top2[:, 0]) > ARGMAX_GAP
        assert clear.mean() >= 0.9, clear.mean()
        near = ~clear
        assert np.array_equal(gam[clear], am[clear]), np.nonzero(gam[clear] != am[clear])[0]
        assert np.all(ref_logits[near, gam[near]] >= mx[near] - ARGMAX_GAP)
    else:
        assert np.array_equal(gam, am), (np.nonzero(gam != am)[0], gam[gam != am], am[gam != am])
    if logits:
        gl = got["logits"].float().cpu().numpy().astype(np.float64)
        assert np.all(np.abs(gl - ref_logits) <= 4e-3 * np.abs(ref_logits) + 1e-3)
    return got, (ref_logits, mx, lse, am)


def test_lm_head_8b_class_shape():
    """60 verified rows, the 128,256-token vocabulary and hidden size 4096 of
    the 8B-class target: statistics only (the logits are not written)."""
    h, w = _draw(60, 128256, 4096, 0)
    _check(h, w)


@pytest.mark.parametrize("rows,vocab,hidden,seed", [(1, 1000, 64, 1), (256, 32000, 512, 2),
                                                    (37, 5003, 128, 3), (96, 32000, 5120, 4)])
def test_lm_head_shapes_with_logits(rows, vocab, hidden, seed):
    """A single row; the most rows one call takes; a row count and a
    vocabulary that are not multiples of the tiles (the last vocabulary tile
    ragged); the 13B-class hidden size.  The bf16 logits are written and
    compared too."""
    h, w = _draw(rows, vocab, hidden, seed)
    _check(h, w, logits=True)


def test_lm_head_argmax_ties_go_to_the_lower_token():
    """Two identical weight rows give bit-identical logits on both sides;
    when they hold the row's maximum the lower token id wins, across tiles
    (token 3 against the row's own argmax far in the vocabulary) and
    inside one tile."""
    h, w = _draw(8, 4000, 256, 5)
    _, (_, _, _, am) = _check(h, w, check_gap=False)
    assert am[0] > 3 and am[1] > 0
    w2 = w.copy()
    w2[3] = w[am[0]]                 # across tiles: row 0's argmax is far from token 3
    _, (_, _, _, am2) = _check(h, w2, check_gap=False)
    assert am2[0] == 3
    w3 = w.copy()
    w3[am[1] - 1] = w[am[1]]         # neighbours, usually inside one tile
    _, (_, _, _, am3) = _check(h, w3, check_gap=False)
    assert am3[1] == am[1] - 1


def test_lm_head_rejects_bad_sizes_before_launch():
    """Row counts outside 1..256 and hidden sizes that are not multiples of
    64 return LTD_ERR_SHAPE (workspace 0) without a launch."""
    L = ltd.lib()
    assert L.ltd_lm_head_workspace_bytes(0, 1000, 64) == 0
    assert L.ltd_lm_head_workspace_bytes(257, 1000, 64) == 0
    assert L.ltd_lm_head_workspace_bytes(4, 1000, 96) == 0
    assert L.ltd_lm_head_workspace_bytes(4, 1000, 128) > 0

"""GPU (C ABI) vs oracle parity on the seeded workloads, plus edge cases.

Sizes: the tiny workload end to end; the draft, selection and acceptance of
every workload at full size (vocab 32k-152k, trees up to 711 nodes, batch 16
ragged); tree attention at full size for one layer, compared on every output
where the oracle is affordable and on sampled KV heads for the 32B and 70B
shapes.
"""

import math

import numpy as np
import pytest
import torch

import oracle
from paper_2603_01639_gb300 import ltd
from paper_2603_01639_gb300 import workload as wl

from . import harness as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2603_01639_gb300 import build
    build.build()
    ltd.lib()
    torch.cuda.init()


def _draft_select_accept(name, seed, cycle_no=0, acc_seed=1234):
    cfg = wl.config(name)
    ci = wl.draw_cycle(cfg, seed)
    trees, sels, target = H.oracle_side(cfg, ci)
    draft = H.dev(ci.draft_rows, cfg.dtype)
    tree = H.gpu_draft(cfg, ci, draft)
    margin = min(H.tree_margin(t, cfg.W) for t in trees)
    assert margin > H.CUT_MARGIN, f"near-tie deciding a frontier ({margin}); pick another seed"
    sel_margin = min(H.select_margin(t, int(n)) for t, n in zip(trees, ci.n_verify))
    assert sel_margin > H.CUT_MARGIN, f"near-tie at the selection cut ({sel_margin})"
    H.compare_trees(cfg, ci, tree, trees)
    got = H.gpu_select(cfg, ci, tree)
    H.compare_select(cfg, ci, got, sels, trees)
    ref = H.oracle_accept(cfg, ci, trees, sels, target, acc_seed, cycle_no)
    assert H.stochastic_margins_ok(ref), "near-tie in a stochastic decision; pick another seed"
    tgt = H.dev(target, cfg.dtype)
    out = ltd.ltd_accept(tree, tgt, draft, got[0], H.i32(ci.n_verify), H.i32(ci.mode),
                         H.i32(ci.ctx), seed=acc_seed, cycle=cycle_no)
    assert ltd.ltd_check() == 0
    H.compare_accept(cfg, out, ref)
    return cfg, ci, ref


# ------------------------------------------------------------ draft/select/accept
def test_tiny_cycle():
    cfg, ci, ref = _draft_select_accept("tiny", 0)
    assert 0 <= ref[0]["accept_len"] <= 3


@pytest.mark.parametrize("seed", [0, 1])
def test_8b_cycle_full_size(seed):
    cfg, ci, ref = _draft_select_accept("8b", seed)
    assert ref[0]["accept_len"] >= 0


@pytest.mark.parametrize("seed", [0, 1, 2, 3, 4])
def test_13b_stochastic_cycles(seed):
    _draft_select_accept("13b", seed, cycle_no=seed)


def test_32b_cycle_full_size():
    _draft_select_accept("32b", 0)


def test_70b_batched_ragged_mixed():
    cfg, ci, ref = _draft_select_accept("70b", 0)
    assert set(ci.mode.tolist()) == {0, 1}
    assert len(set(ci.depth.tolist())) > 1 and len(set(ci.ctx.tolist())) > 1


# ------------------------------------------------------- policy observations
def _check_obs(got, ref, dev_cum, ids, n_real, tail_at):
    """Real slots: the device tree's cums bit for bit and the oracle's within
    CUM_TOL; pad slots: exactly LTD_POLICY_PAD; D and L exact."""
    np.testing.assert_array_equal(got[:n_real], dev_cum[ids])
    err = np.abs(got[:n_real] - ref[:n_real]) / np.maximum(1.0, np.abs(ref[:n_real]))
    assert n_real == 0 or err.max() <= H.CUM_TOL, err.max()
    assert (got[n_real:tail_at] == np.float32(ltd.LTD_POLICY_PAD)).all()
    assert oracle.POLICY_PAD == ltd.LTD_POLICY_PAD
    assert got[tail_at] == ref[tail_at] and got[tail_at + 1] == ref[tail_at + 1]


@pytest.mark.parametrize("name,seed", [("tiny", 0), ("8b", 0), ("70b", 0)])
def test_policy_observations(name, seed):
    """Depth observation after every level (ragged depths: a finished
    sequence keeps reporting its last level) and the size observation of the
    finished tree, padded beyond max_nodes."""
    cfg = wl.config(name)
    ci = wl.draw_cycle(cfg, seed)
    B, W = cfg.batch, cfg.W
    kk = W * W
    draft = H.dev(ci.draft_rows, cfg.dtype)
    ctx = H.i32(ci.ctx)
    depth = np.asarray(ci.depth)
    tree = ltd.Tree(B, cfg.max_depth, W, cfg.vocab)
    ltd.ltd_tree_reset(tree, H.i32(ci.root))
    otrees = [oracle.OracleTree.rooted(int(ci.root[b]), W) for b in range(B)]
    for level in range(1, int(depth.max()) + 1):
        act = depth >= level
        ltd.ltd_expand_tree(tree, level, draft, active=None if act.all() else H.i32(act.astype(np.int32)))
        r0 = 0 if level == 1 else 1 + (level - 2) * W
        r1 = 1 if level == 1 else r0 + W
        for b in np.flatnonzero(act):
            oracle.expand_level(otrees[b], ci.draft_rows[b][r0:r1])
        got = ltd.ltd_depth_observation(tree, ctx).cpu().numpy()
        cum = tree.view()["cum_logprob"].cpu().numpy()
        assert ltd.ltd_check() == 0
        for b in range(B):
            t = otrees[b]
            lv = t.levels
            first = 1 if lv == 1 else 1 + W + (lv - 2) * kk
            count = W if lv == 1 else kk
            ref = oracle.depth_observation(t, int(ci.ctx[b]))
            _check_obs(got[b], ref, cum[b], np.arange(first, first + count), count, kk)
    assert min(H.tree_margin(t, W) for t in otrees) > H.CUT_MARGIN
    v_pad = tree.max_nodes + 13
    got = ltd.ltd_size_observation(tree, ctx, v_pad).cpu().numpy()
    cum = tree.view()["cum_logprob"].cpu().numpy()
    assert ltd.ltd_check() == 0
    for b in range(B):
        ref = oracle.size_observation(otrees[b], int(ci.ctx[b]), v_pad)
        n = otrees[b].n_nodes
        _check_obs(got[b], ref, cum[b], np.arange(n), n, v_pad)


# ------------------------------------------------------- policies on device
def _abs_bound(x, layers):
    """Forward of |x| through |W|, |b| without the ReLU's cut: bounds every
    partial sum, so fp32 rounding stays below ~n eps times it."""
    h = np.abs(np.asarray(x, np.float64))
    for w, b in layers:
        h = h @ np.abs(np.asarray(w, np.float64)) + np.abs(np.asarray(b, np.float64))
    return h


@pytest.mark.parametrize("name,seed,packed", [("8b", 0, True), ("8b", 0, False), ("70b", 0, True),
                                              ("70b", 2, False)])
def test_device_policies_match_the_oracle_network(name, seed, packed):
    """The paper-size networks (seeded random weights), packed for the
    streaming kernel and row-major: logits against the fp64 oracle network
    fed the same observation, decisions where the fp64 top-two gap is clear
    of the fp32 error."""
    from paper_2603_01639_gb300 import policy
    cfg = wl.config(name)
    ci = wl.draw_cycle(cfg, seed)
    B, W = cfg.batch, cfg.W
    draft = H.dev(ci.draft_rows, cfg.dtype)
    ctx = H.i32(ci.ctx)
    tree = ltd.Tree(B, cfg.max_depth, W, cfg.vocab)
    dp = policy.DepthPolicy(W, seed=3)
    sp = policy.SizePolicy(tree.max_nodes, seed=4)
    dnet, snet = dp.net.device(packed=packed), sp.net.device(packed=packed)
    ltd.ltd_tree_reset(tree, H.i32(ci.root))
    depth = np.asarray(ci.depth)

    def check(obs, logits, layers):
        ref = oracle.mlp_forward(obs.astype(np.float64), layers)
        tol = 2e-5 * _abs_bound(obs, layers) + 1e-6
        assert (np.abs(logits - ref) <= tol).all(), np.abs(logits - ref).max()
        return ref, tol

    for level in range(1, int(depth.max()) + 1):
        act = H.i32((depth >= level).astype(np.int32))
        ltd.ltd_expand_tree(tree, level, draft, active=act)
        logits = torch.empty(B, 2, dtype=torch.float32, device="cuda")
        out = ltd.ltd_depth_policy(tree, ctx, dnet, active_in=act, logits=logits)
        obs = ltd.ltd_depth_observation(tree, ctx).cpu().numpy()
        assert ltd.ltd_check() == 0
        ref, tol = check(obs, logits.cpu().numpy(), dp.net.layers)
        want = (ref[:, 1] > ref[:, 0]) & (depth >= level) & (level < cfg.max_depth)
        clear = np.abs(ref[:, 1] - ref[:, 0]) > 2 * tol.max(axis=1)
        assert clear.all(), "near-tie in a depth decision; pick another seed"
        np.testing.assert_array_equal(out.cpu().numpy(), want.astype(np.int32))
    logits = torch.empty(B, 12, dtype=torch.float32, device="cuda")
    n = ltd.ltd_size_policy(tree, ctx, snet, cfg.max_n, logits=logits).cpu().numpy()
    obs = ltd.ltd_size_observation(tree, ctx).cpu().numpy()
    assert ltd.ltd_check() == 0
    ref, tol = check(obs, logits.cpu().numpy(), sp.net.layers)
    nodes = tree.view()["n_nodes"].cpu().numpy()
    for b in range(B):
        top2 = np.sort(ref[b])[-2:]
        assert top2[1] - top2[0] > 2 * tol[b].max(), "near-tie in a size decision"
        a = int(np.argmax(ref[b]))
        assert n[b] == min(21 + 20 * a, cfg.max_n, int(nodes[b]))


def _designed_nets(kk, v_pad):
    """Networks whose decisions read off the observation exactly (powers of
    two and small integers, so fp32 and fp64 agree bit for bit):
    depth: STOP logit D, CONTINUE logit L/2048 + 1.75 -> keep drafting while
    D < L/2048 + 1.75; size: logit_j = j D - j^2/2 -> action D, V = 20 + 20 D."""
    w1 = np.zeros((kk + 2, 2), np.float32)
    w1[kk, 0] = 1.0
    w1[kk + 1, 1] = 1.0 / 2048
    depth = [(w1, np.zeros(2, np.float32)), (np.eye(2, dtype=np.float32), np.array([0, 1.75], np.float32))]
    s1 = np.zeros((v_pad + 2, 1), np.float32)
    s1[v_pad, 0] = 1.0
    j = np.arange(12, dtype=np.float32)
    size = [(s1, np.zeros(1, np.float32)), (j[None, :], -0.5 * j * j)]
    return depth, size


@pytest.mark.parametrize("name,seed", [("tiny", 0), ("70b", 0), ("70b", 3)])
def test_adaptive_draft_driven_by_device_policies(name, seed):
    """The depth policy's decisions drive the draft on the device (each
    level's active mask is the previous decision), the size policy's N feeds
    the selection; the oracle follows its own decisions.  Levels, trees, N
    and the selection must agree exactly."""
    cfg = wl.config(name)
    ci = wl.draw_cycle(cfg, seed)
    B, W = cfg.batch, cfg.W
    draft = H.dev(ci.draft_rows, cfg.dtype)
    ctx = H.i32(ci.ctx)
    tree = ltd.Tree(B, cfg.max_depth, W, cfg.vocab)
    dl, sl = _designed_nets(W * W, tree.max_nodes)
    dnet, snet = ltd.MlpNet(dl), ltd.MlpNet(sl)
    # the oracle's adaptive draft
    otrees = []
    for b in range(B):
        t = oracle.OracleTree.rooted(int(ci.root[b]), W)
        keep = True
        while keep:
            lv = t.levels + 1
            r0 = 0 if lv == 1 else 1 + (lv - 2) * W
            oracle.expand_level(t, ci.draft_rows[b][r0:(1 if lv == 1 else r0 + W)])
            keep, _ = oracle.depth_policy_step(t, int(ci.ctx[b]), dl, True, cfg.max_depth)
        otrees.append(t)
    # the device's: every level launched, sequences stop on the device
    ltd.ltd_tree_reset(tree, H.i32(ci.root))
    act = torch.ones(B, dtype=torch.int32, device="cuda")
    for level in range(1, cfg.max_depth + 1):
        ltd.ltd_expand_tree(tree, level, draft, active=act)
        ltd.ltd_depth_policy(tree, ctx, dnet, active_in=act, active_out=act)
    n_dev = ltd.ltd_size_policy(tree, ctx, snet, cfg.max_n)
    got = ltd.ltd_select_verify(tree, n_dev, cfg.max_n, ctx)
    assert ltd.ltd_check() == 0
    levels = [t.levels for t in otrees]
    if B > 1:
        assert len(set(levels)) > 1, "the designed policy should stop sequences at different depths"
    v = tree.view()
    np.testing.assert_array_equal(v["n_levels"].cpu().numpy(), levels)
    assert min(H.tree_margin(t, W) for t in otrees) > H.CUT_MARGIN
    ci.depth = np.array(levels, np.int32)
    H.compare_trees(cfg, ci, tree, otrees)
    n_ref = [oracle.size_policy_step(t, int(ci.ctx[b]), tree.max_nodes, sl, cfg.max_n)[0]
             for b, t in enumerate(otrees)]
    np.testing.assert_array_equal(n_dev.cpu().numpy(), n_ref)
    ci.n_verify = np.array(n_ref, np.int32)
    sels = [oracle.select_verify(t, int(n), int(ci.ctx[b])) for b, (t, n) in enumerate(zip(otrees, n_ref))]
    assert min(H.select_margin(t, int(n)) for t, n in zip(otrees, n_ref)) > H.CUT_MARGIN
    H.compare_select(cfg, ci, got, sels, otrees)


# ------------------------------------------------ point-mass stochastic rule
def _accept_case(cfg, ci, target, acc_seed=1234, cycle_no=0, temperature=None):
    trees, sels, _ = H.oracle_side(cfg, ci)
    assert min(H.tree_margin(t, cfg.W) for t in trees) > H.CUT_MARGIN
    ref = H.oracle_accept(cfg, ci, trees, sels, target, acc_seed, cycle_no,
                          1.0 if temperature is None else temperature)
    assert H.stochastic_margins_ok(ref), "near-tie in a stochastic decision; pick another seed"
    draft = H.dev(ci.draft_rows, cfg.dtype)
    tree = H.gpu_draft(cfg, ci, draft)
    got = H.gpu_select(cfg, ci, tree)
    out = ltd.ltd_accept(tree, H.dev(target, cfg.dtype), draft, got[0], H.i32(ci.n_verify),
                         H.i32(ci.mode), H.i32(ci.ctx), seed=acc_seed, cycle=cycle_no,
                         temperature=temperature)
    assert ltd.ltd_check() == 0
    H.compare_accept(cfg, out, ref)
    return ref


@pytest.mark.parametrize("mode", [2, 3])
@pytest.mark.parametrize("seed", [0, 1, 3])
def test_variant_rules_accepting(seed, mode):
    """Every sequence on the point-mass (2) or without-replacement (3) rule,
    the target rows at each expanded node a sharpened copy of its draft row
    (so children are accepted, and rejected ones leave the bonus draw)."""
    assert mode in (ltd.LTD_STOCHASTIC_POINT_MASS, ltd.LTD_STOCHASTIC_NO_REPLACEMENT)
    cfg = wl.config("13b")
    ci = wl.draw_cycle(cfg, seed)
    ci.mode = np.full(cfg.batch, mode, np.int32)
    trees, sels, target = H.oracle_side(cfg, ci)
    for b in range(cfg.batch):
        for sl, nid in enumerate(sels[b][0]):
            xr = trees[b].xrow[int(nid)]
            if xr >= 0:
                target[b, sl] = wl.round_to(ci.draft_rows[b, xr] * 5.0, cfg.dtype)
    ref = _accept_case(cfg, ci, target, cycle_no=seed)
    assert ref[0]["accept_len"] >= 1


@pytest.mark.parametrize("seed", [0, 2, 3])
def test_70b_batch_with_every_rule(seed):
    """The ragged 70B batch with greedy, stochastic, point-mass and
    without-replacement sequences side by side."""
    cfg = wl.config("70b")
    ci = wl.draw_cycle(cfg, seed)
    ci.mode = (np.arange(cfg.batch) % 4).astype(np.int32)
    _, _, target = H.oracle_side(cfg, ci)
    _accept_case(cfg, ci, target, cycle_no=seed)


@pytest.mark.parametrize("temperature", [0.5, 2.0])
@pytest.mark.parametrize("seed", [0, 2])
def test_every_rule_at_a_temperature(seed, temperature):
    """ltd_accept_tempered: the ragged 70B batch with all four rules side by
    side at T = 0.5 and T = 2 against the oracle's rules at the same T (p and
    q the softmax of the rows divided by T; greedy unchanged)."""
    cfg = wl.config("70b")
    ci = wl.draw_cycle(cfg, seed)
    ci.mode = (np.arange(cfg.batch) % 4).astype(np.int32)
    _, _, target = H.oracle_side(cfg, ci)
    _accept_case(cfg, ci, target, cycle_no=seed, temperature=temperature)


@pytest.mark.parametrize("mode", [1, 2, 3])
def test_tempered_rules_accepting(mode):
    """Sharpened target rows (a copy of the draft row times 5, as above) at
    T = 2, so children are accepted at the higher temperature too; and T = 1
    through ltd_accept_tempered equals ltd_accept bit for bit."""
    cfg = wl.config("13b")
    ci = wl.draw_cycle(cfg, 1)
    ci.mode = np.full(cfg.batch, mode, np.int32)
    trees, sels, target = H.oracle_side(cfg, ci)
    for b in range(cfg.batch):
        for sl, nid in enumerate(sels[b][0]):
            xr = trees[b].xrow[int(nid)]
            if xr >= 0:
                target[b, sl] = wl.round_to(ci.draft_rows[b, xr] * 5.0, cfg.dtype)
    _accept_case(cfg, ci, target, cycle_no=4, temperature=2.0)
    draft = H.dev(ci.draft_rows, cfg.dtype)
    tree = H.gpu_draft(cfg, ci, draft)
    ids = H.gpu_select(cfg, ci, tree)[0]
    args = (tree, H.dev(target, cfg.dtype), draft, ids, H.i32(ci.n_verify), H.i32(ci.mode),
            H.i32(ci.ctx))
    a = ltd.ltd_accept(*args, seed=9, cycle=1)
    b = ltd.ltd_accept(*args, seed=9, cycle=1, temperature=1.0)
    assert ltd.ltd_check() == 0
    for k in a:
        assert torch.equal(a[k], b[k]), k


def test_unknown_rule_is_flagged_and_the_others_still_run():
    """A mode outside ltd_mode raises the MODE bit; that sequence's outputs
    are -1 and the other sequences of the batch are still right."""
    cfg = wl.config("70b")
    ci = wl.draw_cycle(cfg, 0)
    ci.mode = (np.arange(cfg.batch) % 4).astype(np.int32)
    trees, sels, target = H.oracle_side(cfg, ci)
    ref = H.oracle_accept(cfg, ci, trees, sels, target, 1234, 0)
    draft = H.dev(ci.draft_rows, cfg.dtype)
    tree = H.gpu_draft(cfg, ci, draft)
    got = H.gpu_select(cfg, ci, tree)
    bad = ci.mode.copy()
    bad[5] = 7
    out = ltd.ltd_accept(tree, H.dev(target, cfg.dtype), draft, got[0], H.i32(ci.n_verify),
                         H.i32(bad), H.i32(ci.ctx), seed=1234, cycle=0)
    bits = ltd.ltd_check(raise_on_error=False)
    assert bits == 0x20
    o = {k: v.cpu().numpy() for k, v in out.items()}
    assert o["accept_len"][5] == -1 and o["bonus"][5] == -1 and (o["path"][5] == -1).all()
    assert o["new_ctx"][5] == ci.ctx[5]
    for b in range(cfg.batch):
        if b != 5:
            assert o["accept_len"][b] == ref[b]["accept_len"] and o["bonus"][b] == ref[b]["bonus"]


def test_kv_append_writes_every_layer_and_flags_bad_sequences():
    """The new rows land at ctx_b .. ctx_b + N_b - 1 of every layer's K and V
    (bit for bit), nothing else changes; N out of range and ctx + N past the
    cache are flagged and leave that sequence's rows alone."""
    g = torch.Generator(device="cuda").manual_seed(3)
    L, B, hkv, s_cap, d, n_max = 3, 4, 2, 512, 128, 16
    k = [torch.randn(B, hkv, s_cap, d, generator=g, device="cuda").to(torch.bfloat16) for _ in range(L)]
    v = [torch.randn(B, hkv, s_cap, d, generator=g, device="cuda").to(torch.bfloat16) for _ in range(L)]
    k0 = [t.clone() for t in k]
    v0 = [t.clone() for t in v]
    kv = ltd.KVCache(k, v)
    nk = torch.randn(L, B, hkv, n_max, d, generator=g, device="cuda").to(torch.bfloat16)
    nv = torch.randn(L, B, hkv, n_max, d, generator=g, device="cuda").to(torch.bfloat16)
    ctx = np.array([100, 300, 10, 500], np.int32)
    n = np.array([16, 5, 0, 16], np.int32)           # b=2: N = 0; b=3: 500 + 16 > 512
    ltd.ltd_kv_append(kv, nk, nv, H.i32(ctx), H.i32(n))
    assert ltd.ltd_check(raise_on_error=False) == 0x2 | 0x4
    for l in range(L):
        for cache, before, new in ((k[l], k0[l], nk[l]), (v[l], v0[l], nv[l])):
            want = before.clone()
            for b in (0, 1):
                want[b, :, ctx[b]:ctx[b] + n[b]] = new[b, :, :n[b]]
            assert torch.equal(cache, want)


def test_determinism_and_reuse_of_scratch():
    """Same inputs twice through the same tree and workspace: identical bits
    (tickets and scratch are left ready for reuse)."""
    cfg = wl.config("8b")
    ci = wl.draw_cycle(cfg, 5)
    draft = H.dev(ci.draft_rows, cfg.dtype)
    tree = H.gpu_draft(cfg, ci, draft)
    a = {k: v.clone() for k, v in tree.view().items()}
    H.gpu_draft(cfg, ci, draft, tree)
    b = tree.view()
    for k in a:
        assert torch.equal(a[k], b[k]), k


# --------------------------------------------------------------------- edge cases
def _small_tree(W, L, vocab, seed, dtype=wl.F32, rows=None):
    rng = np.random.default_rng(seed)
    R = 1 + (L - 1) * W
    if rows is None:
        rows = rng.standard_normal((1, R, vocab)).astype(np.float32)
    rows = wl.round_to(rows, dtype)
    root = int(rng.integers(vocab))
    ci = wl.CycleInputs(wl.config("tiny", W=W, vocab=vocab, depth_range=(L, L), dtype=dtype),
                        seed, np.array([root], np.int32), np.array([L], np.int32),
                        np.array([1], np.int32), np.array([0], np.int32),
                        np.array([0], np.int32), rows)
    return ci


@pytest.mark.parametrize("W,L,vocab", [(1, 6, 64), (2, 1, 8), (3, 4, 24), (32, 2, 4096),
                                       (5, 3, 1000 + 8 * 37), (32, 2, 40000)])
def test_expand_and_select_shapes(W, L, vocab):
    """k = 1 chains, a single level, k = 32, vocab not a multiple of the
    vocabulary item; k = 32 over five items per row is more than the merging
    CTA keeps in shared memory, so its warps merge the rows' item lists."""
    ci = _small_tree(W, L, vocab, seed=W * 7 + L)
    cfg = ci.cfg
    tree = H.gpu_draft(cfg, ci, H.dev(ci.draft_rows, wl.F32))
    otree = oracle.grow_tree(int(ci.root[0]), ci.draft_rows[0], W, L)
    H.compare_trees(cfg, ci, tree, [otree])
    n = otree.n_nodes
    for N in sorted({1, 2, min(7, n), min(n, ltd.LTD_MAX_N)}):
        ids, pos, mask = ltd.ltd_select_verify(tree, H.i32([N]), max(N, 1), H.i32([11]))
        rids, rpos, rmask, _ = oracle.select_verify(otree, N, 11)
        assert ids.cpu().numpy()[0].tolist() == rids.tolist()
        assert pos.cpu().numpy()[0].tolist() == rpos.tolist()
        words = oracle.mask_words(rmask)
        assert np.array_equal(mask.cpu().numpy()[0].view(np.uint32), words)
        if W == 1:
            assert np.array_equal(rmask, np.tril(np.ones((N, N), bool)))


@pytest.mark.parametrize("dtype", [wl.F32, wl.BF16])
def test_expand_exact_ties_and_overflowing_candidate_lists(dtype):
    """Logits min(floor(z), 1): about one entry in six ties at the row's
    maximum, so every vocabulary item's candidate list overflows and the
    exact fallback ranks it; the row of frontier rank 0 at level 2 is all
    zeros (every token tied).  Tokens, parents, frontiers bit-exact: tied
    logits go to the lower token, tied children to the lower node id."""
    W, L, vocab = 6, 3, 3 * 8192 + 8 * 13
    rng = np.random.default_rng(17)
    rows = np.minimum(np.floor(rng.standard_normal((1, 1 + (L - 1) * W, vocab))), 1.0)
    rows = rows.astype(np.float32)
    rows[0, 1] = 0.0
    ci = _small_tree(W, L, vocab, seed=17, dtype=dtype, rows=rows)
    otree = oracle.grow_tree(int(ci.root[0]), ci.draft_rows[0], W, L)
    assert H.tree_margin(otree, W) > H.CUT_MARGIN, "near-tie deciding a frontier"
    tree = H.gpu_draft(ci.cfg, ci, H.dev(ci.draft_rows, dtype))
    assert ltd.ltd_check() == 0
    H.compare_trees(ci.cfg, ci, tree, [otree])
    v = tree.view()
    first = 1 + W                               # children of the all-zero row
    assert v["token"][0, first:first + W].tolist() == list(range(W))


def test_expand_rows_that_repeat_every_item():
    """Each row repeats the same decreasing logits every 8192 tokens (one
    vocabulary item), scaled per row, so the row's best tokens are tied
    across the items (ties to the lower token) and nine of every item's ten
    listed keys reach the row's threshold: the merging CTA's candidate list
    for the row overflows and it ranks the row among all of its item keys."""
    W, L, vocab = 10, 3, 7 * 8192
    R = 1 + (L - 1) * W
    t = (np.arange(vocab) % 8192).astype(np.float64)
    rows = np.stack([-(t * 0.001) * (1.0 + 0.05 * r) for r in range(R)])[None].astype(np.float32)
    ci = _small_tree(W, L, vocab, seed=23, rows=rows)
    otree = oracle.grow_tree(int(ci.root[0]), ci.draft_rows[0], W, L)
    assert H.tree_margin(otree, W) > H.CUT_MARGIN, "near-tie deciding a frontier"
    tree = H.gpu_draft(ci.cfg, ci, H.dev(ci.draft_rows, wl.F32))
    assert ltd.ltd_check() == 0
    H.compare_trees(ci.cfg, ci, tree, [otree])
    # level 1: the seven items' first tokens (tied), then three second tokens
    assert tree.view()["token"][0, 1:1 + W].tolist() == [8192 * c for c in range(7)] + [1, 8193, 16385]


def test_expand_wait_runs_out_and_level_stays_unbuilt():
    """The expansion's bounded wait, run out without a GPU fault: the test
    hook makes the merging CTA wait for a tag no record carries, with a 2 ms
    limit.  ltd_check returns LTD_ERR_TIMEOUT with the TIMEOUT bit and the
    level stays unbuilt (n_levels 0, n_nodes 1); with the hook reset the
    same tree grows to the oracle's tree."""
    import ctypes as C
    ci = _small_tree(4, 3, 20000, seed=5)
    cfg = ci.cfg
    draft = H.dev(ci.draft_rows, wl.F32)
    tree = ltd.Tree(1, cfg.max_depth, cfg.W, cfg.vocab)
    ltd.ltd_tree_reset(tree, H.i32(ci.root))
    L = ltd.lib()
    assert L.ltd_debug_expand_wait(2_000_000, 7) == 0
    try:
        ltd.ltd_expand_tree(tree, 1, draft)
        bits = C.c_uint32(0)
        st = L.ltd_check(None, C.byref(bits))
    finally:
        assert L.ltd_debug_expand_wait(0, 0) == 0
    assert L.ltd_status_string(st).decode() == "LTD_ERR_TIMEOUT"
    assert bits.value == 0x10
    v = tree.view()
    assert v["n_levels"].item() == 0 and v["n_nodes"].item() == 1
    tree = H.gpu_draft(cfg, ci, draft, tree)
    assert ltd.ltd_check() == 0
    H.compare_trees(cfg, ci, tree, [oracle.grow_tree(int(ci.root[0]), ci.draft_rows[0], cfg.W, 3)])


def test_single_node_verify_is_autoregressive():
    cfg = wl.config("tiny")
    ci = wl.draw_cycle(cfg, 3)
    ci.n_verify[:] = 1
    draft = H.dev(ci.draft_rows, cfg.dtype)
    tree = H.gpu_draft(cfg, ci, draft)
    ids, pos, mask = H.gpu_select(cfg, ci, tree)
    tgt = torch.randn(1, cfg.max_n, cfg.vocab, device="cuda")
    out = ltd.ltd_accept(tree, tgt, draft, ids, H.i32([1]), H.i32([0]), H.i32(ci.ctx))
    assert out["accept_len"].item() == 0
    assert out["bonus"].item() == int(torch.argmax(tgt[0, 0]).item())
    assert out["new_ctx"].item() == int(ci.ctx[0]) + 1


def test_device_flags_bad_per_sequence_sizes():
    """N larger than the tree is a device-side error: flagged, not trapped, and
    the context stays usable."""
    cfg = wl.config("tiny")
    ci = wl.draw_cycle(cfg, 4)
    draft = H.dev(ci.draft_rows, cfg.dtype)
    tree = H.gpu_draft(cfg, ci, draft)
    ltd.ltd_check()
    ids, pos, mask = ltd.ltd_select_verify(tree, H.i32([12]), 16, H.i32(ci.ctx))  # V_all = 11
    bits = ltd.ltd_check(raise_on_error=False)
    assert bits & 0x2
    assert (ids == -1).all()
    # expanding out of order is flagged too
    ltd.ltd_expand_tree(tree, 2, draft)
    assert ltd.ltd_check(raise_on_error=False) & 0x1
    # and the device still works
    tree = H.gpu_draft(cfg, ci, draft)
    assert ltd.ltd_check() == 0


def test_compaction_race_pattern_and_untouched_rows():
    B, hkv, s_cap, d, layers = 2, 3, 64, 128, 2
    g = torch.Generator(device="cuda").manual_seed(0)
    ks = [torch.randn(B, hkv, s_cap, d, device="cuda", generator=g).to(torch.bfloat16)
          for _ in range(layers)]
    vs = [torch.randn(B, hkv, s_cap, d, device="cuda", generator=g).to(torch.bfloat16)
          for _ in range(layers)]
    before_k = [k.cpu().float().numpy() for k in ks]
    before_v = [v.cpu().float().numpy() for v in vs]
    kv = ltd.KVCache(ks, vs)
    path = H.i32([[0, 2, 3, -1, -1], [0, 1, 4, 6, 9]])
    alen = H.i32([2, 4])
    ctx = H.i32([10, 20])
    ltd.ltd_kv_compact(kv, path, alen, ctx)
    assert ltd.ltd_check() == 0
    for arrs, before in ((ks, before_k), (vs, before_v)):
        for l in range(layers):
            got = arrs[l].cpu().float().numpy()
            for b, (c, p, a) in enumerate([(10, [0, 2, 3], 2), (20, [0, 1, 4, 6, 9], 4)]):
                ref = oracle.compact_kv(before[l][b], c, p[:a + 1])
                assert np.array_equal(got[b], ref)


# ---------------------------------------------------------------------- attention
def _attention_case(name, seed, heads=None, seqs=None, poison=False, workspace=None,
                    bad_seq=None, key_ramp=None, mask_mutant=None, check=True, **overrides):
    """One attention layer through the C ABI against the oracle.  Returns the
    worst max-abs and mean-abs errors over the compared heads and the max-abs
    error relative to the largest reference output.  ``mask_mutant``
    ("transpose" or "drop") feeds the kernel a corrupted copy of the mask
    words while the oracle keeps the true mask (``check=False`` then returns
    the errors without asserting the tolerance)."""
    cfg = wl.config(name, **overrides)
    ci = wl.draw_cycle(cfg, seed, draft_rows=False)
    rng = np.random.default_rng(seed + 5)
    masks = []
    for b in range(cfg.batch):
        # a random valid tree over the verified slots: parent slot < slot
        N = int(ci.n_verify[b])
        par = [-1] + [int(rng.integers(0, i)) for i in range(1, N)]
        m = np.zeros((N, N), bool)
        for i in range(N):
            a = i
            while a >= 0:
                m[i, a] = True
                a = par[a]
        masks.append(m)
    q, k, v = wl.draw_attention(cfg, seed, ci.ctx, ci.n_verify)
    if key_ramp is not None:
        # key j scaled by 1 + key_ramp * j / S_cap: a row's scores grow (or,
        # for a negative ramp, shrink) along the cache
        ramp = 1.0 + key_ramp * np.arange(cfg.s_cap, dtype=np.float32) / cfg.s_cap
        k = wl.round_to(k * ramp[None, None, :, None], cfg.dtype)
    W32 = (cfg.max_n + 31) // 32
    mw = np.zeros((cfg.batch, cfg.max_n, W32), np.uint32)
    for b in range(cfg.batch):
        m = masks[b]
        if mask_mutant == "transpose":
            m = m.T.copy()
        elif mask_mutant == "drop":
            m = m.copy()
            m[-1, 0] = False  # the deepest slot no longer sees the root
        elif mask_mutant is not None:
            raise ValueError(mask_mutant)
        w = oracle.mask_words(m)
        mw[b, :w.shape[0], :w.shape[1]] = w
    qd, kd, vd = H.dev(q, cfg.dtype), H.dev(k, cfg.dtype), H.dev(v, cfg.dtype)
    if poison:
        # the API reads no q row past N_b and no cache row past ctx_b + N_b
        for b in range(cfg.batch):
            N, c = int(ci.n_verify[b]), int(ci.ctx[b])
            qd[b, N:] = float("nan")
            kd[b, :, c + N:] = float("nan")
            vd[b, :, c + N:] = float("nan")
    ctx_arg = ci.ctx.copy()
    if bad_seq is not None:
        ctx_arg[bad_seq] = cfg.max_ctx + 1  # out of range: flagged, the sequence skipped
    out = ltd.ltd_tree_attention(qd, kd, vd, H.i32(ctx_arg), cfg.max_ctx, H.i32(ci.n_verify),
                                 torch.from_numpy(mw.view(np.int32)).cuda(), workspace=workspace)
    if bad_seq is None:
        assert ltd.ltd_check() == 0
    else:
        assert ltd.ltd_check(raise_on_error=False) == 0x4
        assert not out[bad_seq].float().abs().sum().item()
        seqs = [b for b in (seqs if seqs is not None else range(cfg.batch)) if b != bad_seq]
    got = out.float().cpu().numpy()
    G = cfg.hq // cfg.hkv
    scale = 1.0 / math.sqrt(cfg.head_dim)
    worst_max, worst_mean, ref_max = 0.0, 0.0, 0.0
    for b in (seqs if seqs is not None else range(cfg.batch)):
        N, c = int(ci.n_verify[b]), int(ci.ctx[b])
        for kvh in (heads if heads is not None else range(cfg.hkv)):
            hs = list(range(kvh * G, kvh * G + G))
            ref = oracle.tree_attention(q[b, :N][:, hs], k[b, kvh:kvh + 1], v[b, kvh:kvh + 1], c,
                                        masks[b], scale)
            mx, mn = H.attention_error(got[b, :N][:, hs], ref)
            worst_max, worst_mean = max(worst_max, mx), max(worst_mean, mn)
            ref_max = max(ref_max, float(np.abs(ref).max()))
        # rows past N are untouched (zeros from torch.zeros_like)
        assert not got[b, N:].any()
    rel = worst_max / ref_max if ref_max > 0 else 0.0
    if check:
        tol_max, tol_mean = H.ATT_TOL[cfg.dtype]
        assert worst_max <= tol_max and worst_mean <= tol_mean, (worst_max, worst_mean, rel)
    return worst_max, worst_mean, rel


def test_attention_tiny():
    _attention_case("tiny", 0)


@pytest.mark.parametrize("seed", [0, 1])
def test_attention_8b_layer(seed):
    _attention_case("8b", seed)


def test_attention_13b_mha():
    _attention_case("13b", 2)


def test_attention_32b_sampled_heads():
    _attention_case("32b", 0, heads=[0, 7])


def test_attention_70b_sampled():
    _attention_case("70b", 0, heads=[3], seqs=[0, 5, 11, 15])


@pytest.mark.parametrize("name,n", [("8b", 60), ("8b", 256), ("13b", 96), ("32b", 256)])
def test_attention_tree_keys_alone(name, n):
    """ctx = 0: every output row is set by its ancestor keys alone, so one
    wrong mask bit moves it by O(1) (at full context the few ancestor keys
    carry ~0.2% of a row's weight and a wrong bit moves it by ~1e-3).  The
    relative error (max-abs over the largest reference output) stays at bf16
    rounding."""
    mx, mn, rel = _attention_case(name, 20 + n, ctx_range=(0, 0), n_choices=(n,))
    assert rel <= 1e-2, (mx, mn, rel)


def test_attention_tree_keys_alone_catch_mask_mutants():
    """The cases above fail on a corrupted mask: the kernel fed the bit
    matrix transposed (descendants instead of ancestors), or with one
    ancestor bit dropped, misses the oracle's tolerance."""
    tol_max, _ = H.ATT_TOL[wl.BF16]
    for mutant in ("transpose", "drop"):
        mx, mn, rel = _attention_case("8b", 31, ctx_range=(0, 0), n_choices=(60,),
                                      mask_mutant=mutant, check=False)
        assert mx > 10 * tol_max, (mutant, mx, mn)


def test_attention_scores_growing_along_the_cache():
    # later chunks pass a row's running max by far more than its P may grow
    # unchecked: those chunks re-derive P from the chunk's max and rescale O
    _attention_case("8b", 6, ctx_range=(1500, 1500), n_choices=(40,), key_ramp=40.0)
    # full-length 8B layer: two chunks per split, both in one softmax round
    # (a max that grows between them rescales the first chunk's P)
    _attention_case("8b", 9, key_ramp=40.0)
    _attention_case("13b", 7, ctx_range=(900, 900), n_choices=(64,), key_ramp=60.0)
    _attention_case("13b", 8, ctx_range=(900, 900), n_choices=(64,), key_ramp=-0.9)


def test_attention_ignores_rows_past_the_tree():
    """NaN in q rows past N_b and in cache rows past ctx_b + N_b (a ctx that
    ends mid-chunk) must not reach the output."""
    _attention_case("8b", 4, poison=True, ctx_range=(1000, 1000), n_choices=(37,))
    _attention_case("13b", 5, poison=True, ctx_range=(333, 333), n_choices=(48,))


def test_attention_ragged_split_batch():
    """Few units, so every unit's keys are split; short sequences leave some
    splits without keys."""
    _attention_case("8b", 6, batch=3, ctx_range=(20, 3000), n_choices=(7, 33, 60))


@pytest.mark.parametrize("name,hq,hkv,ctx,n", [("8b", 8, 2, 3968, 60), ("13b", 60, 60, 2048, 64),
                                                ("13b", 15, 15, 2600, 64)])
def test_attention_split_counts(name, hq, hkv, ctx, n):
    """On a 152-SM device these shapes cut each unit's keys into 32 splits of
    one chunk (4 units, 32 chunks), 2 splits (60 units) and 7 splits (15
    units, 21 chunks): the most, the fewest and an odd count, each combined
    through the workspace."""
    _attention_case(name, 40 + hq, hq=hq, hkv=hkv, ctx_range=(ctx, ctx), n_choices=(n,))


def test_attention_flags_bad_sequence():
    """A sequence with ctx past max_ctx is flagged and left untouched, in
    both launch shapes (split keys; one split per unit, longest first), and
    the other sequences are still right."""
    _attention_case("8b", 10, bad_seq=1, batch=3, ctx_range=(500, 3000), n_choices=(20, 60))
    _attention_case("70b", 11, bad_seq=4, heads=[0, 5], seqs=[0, 4, 9, 15])
    assert ltd.ltd_check() == 0


def test_attention_next_layer_hint_changes_nothing():
    """ltd_tree_attention_next (L2 hint for the next layer's caches) returns
    the bytes ltd_tree_attention returns."""
    for name in ("8b", "13b"):
        cfg = wl.config(name)
        ci = wl.draw_cycle(cfg, 12, draft_rows=False)
        q, k, v = wl.draw_attention(cfg, 12, ci.ctx, ci.n_verify)
        qd, kd, vd = H.dev(q, cfg.dtype), H.dev(k, cfg.dtype), H.dev(v, cfg.dtype)
        k2, v2 = torch.roll(kd, 1, dims=2), torch.roll(vd, 1, dims=2)
        W32 = (cfg.max_n + 31) // 32
        mw = torch.zeros(cfg.batch, cfg.max_n, W32, dtype=torch.int32, device="cuda")
        mw[..., 0] = 1
        c, n = H.i32(ci.ctx), H.i32(ci.n_verify)
        a = ltd.ltd_tree_attention(qd, kd, vd, c, cfg.max_ctx, n, mw)
        b = ltd.ltd_tree_attention(qd, kd, vd, c, cfg.max_ctx, n, mw, next_k=k2, next_v=v2)
        assert ltd.ltd_check() == 0
        assert torch.equal(a, b)


def test_attention_workspace_reuse():
    """Back-to-back calls on one workspace: the split counters are left at
    zero by each call, so every call combines correctly."""
    cfg = wl.config("8b")
    ws = ltd.attention_workspace(cfg.batch, cfg.hq, cfg.hkv, cfg.head_dim, cfg.max_n,
                                 cfg.max_ctx, torch.bfloat16)
    for seed in (7, 8, 9):
        _attention_case("8b", seed, workspace=ws)


def test_attention_split_wait_runs_out_and_recovers():
    """A bounded wait that runs out, without a GPU fault: the test hook makes
    every split of the 8B-class layer wait on its unit's counter for one
    arrival more than the unit has, with a 2 ms limit.  Every split gives
    up, ltd_check returns LTD_ERR_TIMEOUT with the TIMEOUT bit, and no
    output row is written; the splits still departed, so the counters are
    back at zero and, with the hook reset, the same workspace gives the
    oracle's result on the next calls."""
    import ctypes as C
    cfg = wl.config("8b")
    ws = ltd.attention_workspace(cfg.batch, cfg.hq, cfg.hkv, cfg.head_dim, cfg.max_n,
                                 cfg.max_ctx, torch.bfloat16)
    ci = wl.draw_cycle(cfg, 13, draft_rows=False)
    q, k, v = wl.draw_attention(cfg, 13, ci.ctx, ci.n_verify)
    W32 = (cfg.max_n + 31) // 32
    mw = torch.zeros(cfg.batch, cfg.max_n, W32, dtype=torch.int32, device="cuda")
    mw[..., 0] = 1
    L = ltd.lib()
    assert L.ltd_debug_attention_wait(2_000_000, 1) == 0
    try:
        out = ltd.ltd_tree_attention(H.dev(q, cfg.dtype), H.dev(k, cfg.dtype), H.dev(v, cfg.dtype),
                                     H.i32(ci.ctx), cfg.max_ctx, H.i32(ci.n_verify), mw,
                                     workspace=ws)
        bits = C.c_uint32(0)
        st = L.ltd_check(None, C.byref(bits))
    finally:
        assert L.ltd_debug_attention_wait(0, 0) == 0
    assert L.ltd_status_string(st).decode() == "LTD_ERR_TIMEOUT"
    assert bits.value == 0x10
    assert not out.float().abs().sum().item()
    for seed in (14, 15):
        _attention_case("8b", seed, workspace=ws)


def test_attention_all_ones_mask_equals_unmasked():
    cfg = wl.config("8b", ctx_range=(300, 300), n_choices=(40,))
    rng = np.random.default_rng(3)
    q = wl.round_to(rng.standard_normal((1, 40, cfg.hq, 128)).astype(np.float32), wl.BF16)
    k = wl.round_to(rng.standard_normal((1, cfg.hkv, cfg.s_cap, 128)).astype(np.float32), wl.BF16)
    v = wl.round_to(rng.standard_normal((1, cfg.hkv, cfg.s_cap, 128)).astype(np.float32), wl.BF16)
    ones = np.full((1, 40, 2), 0xFFFFFFFF, np.uint32)
    ones[..., 1] = (1 << 8) - 1
    out = ltd.ltd_tree_attention(H.dev(q, wl.BF16), H.dev(k, wl.BF16), H.dev(v, wl.BF16),
                                 H.i32([300]), 300, H.i32([40]),
                                 torch.from_numpy(ones.view(np.int32)).cuda())
    G = cfg.hq // cfg.hkv
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q[0].astype(np.float64)).transpose(0, 1),
        torch.from_numpy(np.repeat(k[0, :, :340], G, 0).astype(np.float64)),
        torch.from_numpy(np.repeat(v[0, :, :340], G, 0).astype(np.float64)),
        scale=1 / math.sqrt(128)).transpose(0, 1).numpy()
    mx, mn = H.attention_error(out[0].float().cpu().numpy(), ref)
    assert mx <= 2e-2 and mn <= 2e-3

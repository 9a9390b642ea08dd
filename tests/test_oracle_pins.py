"""Pins of the fp64 oracle against facts that do not come from the oracle:
a hand-worked example, closed forms, library routines (scipy log_softmax,
torch scaled_dot_product_attention), brute force on tiny inputs, invariants,
the published splitmix64 test vector and a Monte-Carlo test of the
lossless-sampling theorem.  A final group plants plausible mistakes in the
oracle and checks that these pins catch them."""

import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import scipy.special
import scipy.stats
import torch

import oracle
from oracle import ltd_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _worked():
    with open(os.path.join(GOLDEN, "worked_cycle.json")) as f:
        return json.load(f)


def _rows_from_weights(weights):
    return np.log(np.asarray(weights, dtype=np.float64))


# ------------------------------------------------------------ worked example
def test_worked_example_tree():
    g = _worked()
    rows = _rows_from_weights(g["draft_row_weights"])
    tree = oracle.grow_tree(g["root_token"], rows, g["W"], g["L"])
    assert tree.n_nodes == len(g["expected_nodes"]) == oracle.v_all(g["W"], g["L"])
    for node in g["expected_nodes"]:
        i = node["id"]
        assert tree.token[i] == node["token"]
        assert tree.parent[i] == node["parent"]
        assert tree.depth[i] == node["depth"]
        assert tree.cum[i] == pytest.approx(math.log(Fraction(node["cum"])), abs=1e-12)
    assert tree.frontier == g["expected_frontier_after_level"][str(g["L"])]


def test_worked_example_frontiers_per_level():
    g = _worked()
    rows = _rows_from_weights(g["draft_row_weights"])
    for L in (1, 2, 3):
        tree = oracle.grow_tree(g["root_token"], rows, g["W"], L)
        assert tree.frontier == g["expected_frontier_after_level"][str(L)]


def test_worked_example_select_and_accept():
    g = _worked()
    rows = _rows_from_weights(g["draft_row_weights"])
    tree = oracle.grow_tree(g["root_token"], rows, g["W"], g["L"])
    ids, pos, mask, _ = oracle.select_verify(tree, g["N"], g["ctx"])
    assert list(ids) == g["expected_slots"]
    assert list(pos) == g["expected_pos"]
    words = oracle.mask_words(mask)
    assert [int(w[0]) for w in words] == g["expected_mask_words"]
    target = np.asarray(g["target_rows"], dtype=np.float64)
    path, a, bonus = oracle.accept_greedy(tree, ids, target)
    assert path == g["expected_path"]
    assert a == g["expected_accept_len"]
    assert bonus == g["expected_bonus"]
    res = oracle.cycle(g["root_token"], rows, g["W"], g["L"], g["N"], g["ctx"], target)
    assert res["new_ctx"] == g["expected_new_ctx"]


# ------------------------------------------------------------- expansion pins
def _random_tree(seed, W, L, vocab, ties=False):
    rng = np.random.default_rng(seed)
    R = 1 + (L - 1) * W
    rows = rng.standard_normal((R, vocab))
    if ties:
        rows = np.round(rows * 2) / 2  # many exact ties
    root = int(rng.integers(vocab))
    return oracle.grow_tree(root, rows, W, L), rows, root


@pytest.mark.parametrize("W,L", [(1, 1), (1, 5), (2, 1), (2, 3), (3, 4), (10, 2), (4, 6)])
def test_tree_size_closed_form(W, L):
    tree, _, _ = _random_tree(W * 100 + L, W, L, vocab=64)
    # 3.2 Candidate Token Selection: V_all = 1 + W + (D-2) W^2 with D = L + 1
    assert tree.n_nodes == 1 + W + (L - 1) * W * W


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("ties", [False, True])
def test_expand_against_scipy_and_brute_force(seed, ties):
    W, L, vocab = 3, 4, 9
    tree, rows, _ = _random_tree(seed, W, L, vocab, ties)
    # every expanded row: scipy's log_softmax, normalisation, and the
    # brute-force rank of each child among all tokens of its parent's row
    for u in range(tree.n_nodes):
        r = tree.xrow[u]
        if r < 0:
            continue
        row = rows[r]
        ref = scipy.special.logsumexp(row)
        assert tree.xlse[u] == pytest.approx(ref, abs=1e-12)
        assert np.exp(row - tree.xlse[u]).sum() == pytest.approx(1.0, abs=1e-12)
        kids = [c for c in range(tree.n_nodes) if tree.parent[c] == u]
        assert len(kids) == W
        for rank, c in enumerate(kids):
            t = tree.token[c]
            better = sum(1 for s in range(vocab)
                         if row[s] > row[t] or (row[s] == row[t] and s < t))
            assert better == rank
    # cum of every node is the sum of scipy log-probs along its path
    for c in range(1, tree.n_nodes):
        total, a = 0.0, c
        while tree.parent[a] >= 0:
            p = tree.parent[a]
            total += scipy.special.log_softmax(rows[tree.xrow[p]])[tree.token[a]]
            a = p
        assert tree.cum[c] == pytest.approx(total, abs=1e-12)
        assert tree.depth[c] == tree.depth[tree.parent[c]] + 1


@pytest.mark.parametrize("seed", range(6))
def test_beam_frontier_is_top_w_of_pool(seed):
    W, L = 3, 5
    tree, rows, _ = _random_tree(seed, W, L, vocab=11, ties=(seed % 2 == 1))
    # brute force: frontier after the last level is the W best of the last
    # level's W^2 children by (cum desc, id asc)
    last = [i for i in range(tree.n_nodes) if tree.depth[i] == L]
    assert len(last) == W * W
    best = sorted(last, key=lambda i: (-tree.cum[i], i))[:W]
    assert tree.frontier == best
    # only frontier nodes of level l have children at level l + 1
    for lvl in range(2, L):
        parents = {tree.parent[i] for i in range(tree.n_nodes) if tree.depth[i] == lvl + 1}
        lvl_nodes = [i for i in range(tree.n_nodes) if tree.depth[i] == lvl]
        ranked = sorted(lvl_nodes, key=lambda i: (-tree.cum[i], i))[:W]
        assert parents == set(ranked)


def test_expand_row_indexing_follows_frontier_rank():
    W, L = 2, 3
    tree, rows, _ = _random_tree(11, W, L, vocab=7)
    # level 3 rows are 1 + W + r for frontier rank r of level 2
    lvl2_frontier = sorted([i for i in range(tree.n_nodes) if tree.depth[i] == 2],
                           key=lambda i: (-tree.cum[i], i))[:W]
    for r, f in enumerate(lvl2_frontier):
        assert tree.xrow[f] == 1 + (3 - 2) * W + r


# ------------------------------------------------------------- selection pins
def _ancestry_closure(parent):
    n = len(parent)
    A = np.eye(n, dtype=np.int64)
    adj = np.zeros((n, n), dtype=np.int64)
    for c, p in enumerate(parent):
        if p >= 0:
            adj[c, p] = 1
    step = adj.copy()
    for _ in range(n):
        A = np.minimum(A + step, 1)
        step = np.minimum(step @ adj, 1)
    return A  # A[c, a] = 1 iff a is an ancestor-or-self of c


@pytest.mark.parametrize("seed", range(5))
@pytest.mark.parametrize("N", [1, 2, 5, 13, 30])
def test_select_brute_force(seed, N):
    W, L = 3, 4
    tree, _, _ = _random_tree(seed, W, L, vocab=10, ties=(seed % 2 == 0))
    N = min(N, tree.n_nodes)
    ctx = 37
    ids, pos, mask, _ = oracle.select_verify(tree, N, ctx)
    chosen = set(int(i) for i in ids)
    assert 0 in chosen and len(chosen) == N
    assert list(ids) == sorted(ids)
    key = lambda i: (-tree.cum[i], i)  # noqa: E731
    inside = [i for i in chosen if i != 0]
    outside = [i for i in range(1, tree.n_nodes) if i not in chosen]
    for i in inside:
        for j in outside:
            assert key(i) < key(j)
    A = _ancestry_closure(tree.parent)
    for si, ni in enumerate(ids):
        assert pos[si] == ctx + tree.depth[ni]
        for sj, nj in enumerate(ids):
            assert bool(mask[si, sj]) == bool(A[ni, nj])
        # ancestor-closed and topological: every ancestor is verified, earlier
        a = tree.parent[ni]
        while a >= 0:
            assert a in chosen and list(ids).index(a) < si
            a = tree.parent[a]


def test_select_special_cases():
    tree, _, _ = _random_tree(3, 3, 3, vocab=8)
    ids, pos, mask, _ = oracle.select_verify(tree, 1, 5)
    assert list(ids) == [0] and list(pos) == [5] and mask.tolist() == [[True]]
    ids, _, mask, _ = oracle.select_verify(tree, tree.n_nodes, 5)
    assert list(ids) == list(range(tree.n_nodes))
    # W = 1 is a chain: the mask is lower-triangular
    chain, _, _ = _random_tree(4, 1, 7, vocab=8)
    ids, _, mask, _ = oracle.select_verify(chain, chain.n_nodes, 0)
    assert np.array_equal(mask, np.tril(np.ones((8, 8), dtype=bool)))


def test_mask_words_layout():
    m = np.zeros((2, 70), dtype=bool)
    m[0, 0] = m[0, 31] = m[0, 32] = m[1, 69] = True
    w = oracle.mask_words(m)
    assert w.shape == (2, 3)
    assert w[0].tolist() == [1 | (1 << 31), 1, 0]
    assert w[1].tolist() == [0, 0, 1 << 5]


# ------------------------------------------------------------- attention pins
def _sdpa(q, k, v, mask=None, causal=False, scale=None):
    return torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q), torch.from_numpy(k), torch.from_numpy(v),
        attn_mask=None if mask is None else torch.from_numpy(mask),
        is_causal=causal, scale=scale).numpy()


def _att_inputs(seed, N, Hq, Hkv, d, ctx, s_cap=None):
    rng = np.random.default_rng(seed)
    s_cap = s_cap or ctx + N + 5
    q = rng.standard_normal((N, Hq, d))
    k = rng.standard_normal((Hkv, s_cap, d))
    v = rng.standard_normal((Hkv, s_cap, d))
    return q, k, v


def test_attention_chain_equals_causal():
    N, Hq, Hkv, d, ctx = 6, 4, 2, 16, 9
    q, k, v = _att_inputs(0, N, Hq, Hkv, d, ctx)
    mask = np.tril(np.ones((N, N), dtype=bool))
    scale = 1 / math.sqrt(d)
    out = oracle.tree_attention(q, k, v, ctx, mask, scale)
    # causal attention over the ctx + N sequence; prefix queries are arbitrary
    rng = np.random.default_rng(1)
    qfull = np.concatenate([rng.standard_normal((ctx, Hq, d)), q], axis=0)
    G = Hq // Hkv
    kk = np.repeat(k[:, :ctx + N], G, axis=0)
    vv = np.repeat(v[:, :ctx + N], G, axis=0)
    ref = _sdpa(qfull.transpose(1, 0, 2), kk, vv, causal=True, scale=scale)
    np.testing.assert_allclose(out, ref.transpose(1, 0, 2)[ctx:], atol=1e-12)


def test_attention_all_ones_equals_unmasked():
    N, Hq, Hkv, d, ctx = 5, 2, 2, 8, 11
    q, k, v = _att_inputs(2, N, Hq, Hkv, d, ctx)
    out = oracle.tree_attention(q, k, v, ctx, np.ones((N, N), bool), 0.3)
    ref = _sdpa(q.transpose(1, 0, 2), k[:, :ctx + N], v[:, :ctx + N], scale=0.3)
    np.testing.assert_allclose(out, ref.transpose(1, 0, 2), atol=1e-12)


def test_attention_single_token_is_decode():
    Hq, Hkv, d, ctx = 8, 2, 32, 50
    q, k, v = _att_inputs(3, 1, Hq, Hkv, d, ctx)
    out = oracle.tree_attention(q, k, v, ctx, np.ones((1, 1), bool), 1 / math.sqrt(d))
    G = Hq // Hkv
    ref = _sdpa(q.transpose(1, 0, 2), np.repeat(k[:, :ctx + 1], G, 0),
                np.repeat(v[:, :ctx + 1], G, 0), scale=1 / math.sqrt(d))
    np.testing.assert_allclose(out, ref.transpose(1, 0, 2), atol=1e-12)


@pytest.mark.parametrize("seed", range(3))
def test_attention_tree_mask_and_gqa(seed):
    W, L = 2, 3
    tree, _, _ = _random_tree(seed, W, L, vocab=6)
    N = 7
    ids, _, mask, _ = oracle.select_verify(tree, N, 0)
    Hq, Hkv, d, ctx = 8, 2, 16, 13
    q, k, v = _att_inputs(seed + 10, N, Hq, Hkv, d, ctx)
    out = oracle.tree_attention(q, k, v, ctx, mask, 0.25)
    # independent mask from parent pointers, GQA as MHA with repeated KV heads
    A = _ancestry_closure(tree.parent)
    allowed = np.zeros((N, ctx + N), dtype=bool)
    allowed[:, :ctx] = True
    for i, ni in enumerate(ids):
        for j, nj in enumerate(ids):
            allowed[i, ctx + j] = bool(A[ni, nj])
    G = Hq // Hkv
    ref = _sdpa(q.transpose(1, 0, 2), np.repeat(k[:, :ctx + N], G, 0),
                np.repeat(v[:, :ctx + N], G, 0), mask=allowed, scale=0.25)
    np.testing.assert_allclose(out, ref.transpose(1, 0, 2), atol=1e-12)


# -------------------------------------------------------- greedy accept pins
def _brute_force_greedy(tree, ids, target):
    """Enumerate every root path inside the verified set; the accepted one is
    the longest whose every edge matches the target argmax at its parent."""
    slot_of = {int(n): s for s, n in enumerate(ids)}
    best = [0]
    for s, n in enumerate(ids):
        path, a = [], int(n)
        while a >= 0:
            path.append(slot_of[a])
            a = tree.parent[a]
        path = path[::-1]
        ok = all(tree.token[int(ids[path[t + 1]])] == int(np.argmax(target[path[t]]))
                 for t in range(len(path) - 1))
        if ok and len(path) > len(best):
            best = path
    return best, int(np.argmax(target[best[-1]]))


@pytest.mark.parametrize("seed", range(12))
def test_greedy_accept_brute_force(seed):
    W, L = 3, 4
    rng = np.random.default_rng(seed + 100)
    tree, _, _ = _random_tree(seed, W, L, vocab=5, ties=True)
    N = int(rng.integers(1, tree.n_nodes + 1))
    ids, _, _, _ = oracle.select_verify(tree, N, 0)
    target = np.round(rng.standard_normal((N, 5)) * 2) / 2  # ties in argmax
    # plant agreement on a random subset so long paths occur
    for s, n in enumerate(ids):
        kids = [t for t, m in enumerate(ids) if tree.parent[int(m)] == int(n)]
        if kids and rng.random() < 0.8:
            target[s, tree.token[int(ids[kids[0]])]] = 10.0
    path, a, bonus = oracle.accept_greedy(tree, ids, target)
    ref_path, ref_bonus = _brute_force_greedy(tree, ids, target)
    assert path == ref_path and bonus == ref_bonus and a == len(path) - 1
    assert a <= L


def test_greedy_single_node_is_autoregressive():
    tree, _, _ = _random_tree(9, 4, 3, vocab=30)
    ids, _, _, _ = oracle.select_verify(tree, 1, 0)
    row = np.random.default_rng(0).standard_normal((1, 30))
    path, a, bonus = oracle.accept_greedy(tree, ids, row)
    assert path == [0] and a == 0 and bonus == int(np.argmax(row[0]))


# ---------------------------------------------------- stochastic accept pins
def _star_tree(root_tok, child_tokens, W):
    """Root with the given children (may repeat tokens); the root was expanded
    from draft row 0."""
    t = O.OracleTree.rooted(root_tok, W)
    t.xrow[0] = 0
    for tok in child_tokens:
        t._add(tok, 0, 1, 0.0)
    return t


def test_stochastic_preserves_target_distribution():
    """Lossless theorem (speculative sampling): with children drawn i.i.d.
    from q, the first emitted token is distributed as p = softmax(target)."""
    vocab, k, trials = 6, 3, 30000
    rng = np.random.default_rng(123)
    xt = rng.standard_normal(vocab) * 1.5
    xq = rng.standard_normal(vocab) * 1.5
    p = scipy.special.softmax(xt)
    q = scipy.special.softmax(xq)
    draft_rows = xq[None, :]
    counts = np.zeros(vocab)
    for trial in range(trials):
        kids = rng.choice(vocab, size=k, p=q)
        tree = _star_tree(0, kids, k)
        ids = np.arange(k + 1)
        target = np.vstack([xt] + [rng.standard_normal(vocab) for _ in range(k)])
        path, a, bonus, _ = oracle.accept_stochastic(tree, ids, target, draft_rows,
                                                     seed=7, b=0, cycle_no=trial)
        first = tree.token[path[1]] if a >= 1 else bonus
        counts[first] += 1
    chi2 = ((counts - trials * p) ** 2 / (trials * p)).sum()
    pval = scipy.stats.chi2.sf(chi2, vocab - 1)
    assert pval > 1e-4, (counts / trials, p, pval)


def test_stochastic_bonus_is_exact_sample():
    """No children: the bonus alone is a Gumbel-max draw from p."""
    vocab, trials = 5, 20000
    xt = np.array([0.3, -1.0, 2.0, 0.0, 1.1])
    p = scipy.special.softmax(xt)
    tree = _star_tree(0, [], 1)
    counts = np.zeros(vocab)
    for trial in range(trials):
        _, a, bonus, _ = oracle.accept_stochastic(tree, np.array([0]), xt[None, :],
                                                  xt[None, :], seed=3, b=1, cycle_no=trial)
        assert a == 0
        counts[bonus] += 1
    chi2 = ((counts - trials * p) ** 2 / (trials * p)).sum()
    assert scipy.stats.chi2.sf(chi2, vocab - 1) > 1e-4


def test_stochastic_identical_draft_and_target_accepts_first_child():
    """q == p: the ratio test r q(x) < p(x) holds for every r < 1."""
    vocab = 7
    x = np.random.default_rng(5).standard_normal(vocab)
    tree = _star_tree(0, [3, 1], 2)
    path, a, _, _ = oracle.accept_stochastic(tree, np.arange(3), np.vstack([x, x, x]),
                                             x[None, :], seed=1, b=0, cycle_no=0)
    assert path == [0, 1] and a == 1


def test_stochastic_zero_probability_child_rejected():
    """p(x) = 0 up to fp64 underflow: the child is always rejected."""
    vocab = 4
    xt = np.array([0.0, -1e4, 0.0, 0.0])
    xq = np.zeros(vocab)
    tree = _star_tree(0, [1], 1)
    for c in range(50):
        path, a, bonus, _ = oracle.accept_stochastic(tree, np.arange(2), np.vstack([xt, xt]),
                                                     xq[None, :], seed=9, b=0, cycle_no=c)
        assert a == 0 and bonus != 1


# ------------------------------------------------------------------ RNG pins
# ---------------------------------------------------- LM-head row statistics
def test_lm_head_rows_against_torch_linear_and_scipy():
    """logits = hidden W^T as torch.nn.functional.linear computes it (W held
    [vocab][d_model]); row statistics from scipy's logsumexp and a brute-force
    first-maximum scan."""
    rng = np.random.default_rng(9)
    h = rng.standard_normal((5, 12))
    w = rng.standard_normal((37, 12))
    logits, mx, lse, am = O.lm_head_row_stats(h, w)
    ref = torch.nn.functional.linear(torch.from_numpy(h), torch.from_numpy(w)).numpy()
    np.testing.assert_allclose(logits, ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(lse, scipy.special.logsumexp(ref, axis=1), rtol=1e-12)
    np.testing.assert_array_equal(mx, ref.max(axis=1))
    for r in range(5):
        best = max(range(37), key=lambda v: (ref[r, v], -v))
        assert am[r] == best


def test_lm_head_argmax_ties_to_the_lower_token():
    h = np.array([[1.0, 0.0]])
    w = np.array([[0.0, 1.0], [2.0, 0.0], [2.0, 5.0], [1.0, 1.0]])   # tokens 1 and 2 tie at 2
    _, mx, _, am = O.lm_head_row_stats(h, w)
    assert mx[0] == 2.0 and am[0] == 1


# ------------------------------------------------------------- temperature
def test_softmax_at_temperature_is_scipy_softmax_of_scaled_logits():
    x = np.array([0.5, -1.0, 2.0, 0.0, 3.5])
    for T in (0.25, 1.0, 3.0):
        np.testing.assert_allclose(O.softmax_t(x, T), scipy.special.softmax(x / T), rtol=1e-13)


@pytest.mark.parametrize("T", [0.5, 2.0])
def test_stochastic_rule_at_temperature_samples_the_tempered_target(T):
    """Children i.i.d. from q_T = softmax(draft / T): the first emitted token
    follows p_T = softmax(target / T)."""
    vocab, k, trials = 6, 3, 20000
    rng = np.random.default_rng(int(T * 100))
    xt = rng.standard_normal(vocab) * 1.5
    xq = rng.standard_normal(vocab) * 1.5
    p = scipy.special.softmax(xt / T)
    q = scipy.special.softmax(xq / T)
    counts = np.zeros(vocab)
    for trial in range(trials):
        kids = rng.choice(vocab, size=k, p=q)
        tree = _star_tree(0, kids, k)
        target = np.vstack([xt] + [rng.standard_normal(vocab) for _ in range(k)])
        path, a, bonus, _ = oracle.accept_stochastic(tree, np.arange(k + 1), target, xq[None, :],
                                                     seed=5, b=0, cycle_no=trial, temperature=T)
        counts[tree.token[path[1]] if a >= 1 else bonus] += 1
    chi2 = ((counts - trials * p) ** 2 / (trials * p)).sum()
    assert scipy.stats.chi2.sf(chi2, vocab - 1) > 1e-4, (counts / trials, p)


def test_point_mass_at_temperature_samples_the_tempered_target():
    vocab, k, trials, T = 6, 2, 20000, 0.5
    xt = np.array([1.0, 0.4, -0.3, 0.9, -1.1, 0.2])
    p = scipy.special.softmax(xt / T)
    tree = _star_tree(0, [0, 3], k)
    counts = np.zeros(vocab)
    for trial in range(trials):
        path, a, bonus, _ = oracle.accept_point_mass(tree, np.arange(k + 1), np.vstack([xt] * (k + 1)),
                                                     seed=8, b=0, cycle_no=trial, temperature=T)
        counts[tree.token[path[1]] if a >= 1 else bonus] += 1
    chi2 = ((counts - trials * p) ** 2 / (trials * p)).sum()
    assert scipy.stats.chi2.sf(chi2, vocab - 1) > 1e-4, (counts / trials, p)


# --------------------------------------------- without-replacement rule
def test_without_replacement_preserves_target_distribution():
    """Children drawn from q WITHOUT replacement (distinct tokens, as a
    top-k tree has): the first emitted token is distributed as p."""
    vocab, k, trials = 6, 3, 30000
    rng = np.random.default_rng(77)
    xt = rng.standard_normal(vocab) * 1.5
    xq = rng.standard_normal(vocab) * 1.5
    p = scipy.special.softmax(xt)
    q = scipy.special.softmax(xq)
    counts = np.zeros(vocab)
    for trial in range(trials):
        kids = rng.choice(vocab, size=k, p=q, replace=False)   # sequential draws without replacement
        tree = _star_tree(0, kids, k)
        target = np.vstack([xt] + [rng.standard_normal(vocab) for _ in range(k)])
        path, a, bonus, _ = oracle.accept_without_replacement(tree, np.arange(k + 1), target, xq[None, :],
                                                              seed=13, b=0, cycle_no=trial)
        first = tree.token[path[1]] if a >= 1 else bonus
        counts[first] += 1
    chi2 = ((counts - trials * p) ** 2 / (trials * p)).sum()
    assert scipy.stats.chi2.sf(chi2, vocab - 1) > 1e-4, (counts / trials, p)


def test_with_replacement_rule_is_biased_for_distinct_children():
    """The plain rule keeps q after a rejection, which assumes i.i.d.
    children; for distinct children it is off -- the variant above is what
    makes the difference (guards against the two rules being the same)."""
    vocab, k, trials = 4, 3, 20000
    xt = np.array([2.0, 1.5, -1.0, 0.0])
    xq = np.array([2.0, 1.8, 1.6, -3.0])
    p = scipy.special.softmax(xt)
    q = scipy.special.softmax(xq)
    rng = np.random.default_rng(5)
    counts = np.zeros(vocab)
    for trial in range(trials):
        kids = rng.choice(vocab, size=k, p=q, replace=False)
        tree = _star_tree(0, kids, k)
        path, a, bonus, _ = oracle.accept_stochastic(tree, np.arange(k + 1), np.vstack([xt] * (k + 1)),
                                                     xq[None, :], seed=3, b=0, cycle_no=trial)
        counts[tree.token[path[1]] if a >= 1 else bonus] += 1
    chi2 = ((counts - trials * p) ** 2 / (trials * p)).sum()
    assert scipy.stats.chi2.sf(chi2, vocab - 1) < 1e-6


# ------------------------------------------------ point-mass stochastic rule
def test_point_mass_preserves_target_distribution_for_deterministic_children():
    """The children are a fixed top-k set (not samples from any q): the
    first emitted token is still distributed exactly as p."""
    vocab, k, trials = 6, 3, 30000
    rng = np.random.default_rng(321)
    xt = rng.standard_normal(vocab) * 1.5
    p = scipy.special.softmax(xt)
    kids = np.argsort(-p)[:k]                      # deterministic: the k likeliest
    tree = _star_tree(0, kids, k)
    ids = np.arange(k + 1)
    counts = np.zeros(vocab)
    for trial in range(trials):
        target = np.vstack([xt] + [rng.standard_normal(vocab) for _ in range(k)])
        path, a, bonus, _ = oracle.accept_point_mass(tree, ids, target, seed=11, b=0, cycle_no=trial)
        first = tree.token[path[1]] if a >= 1 else bonus
        counts[first] += 1
    chi2 = ((counts - trials * p) ** 2 / (trials * p)).sum()
    assert scipy.stats.chi2.sf(chi2, vocab - 1) > 1e-4, (counts / trials, p)


def test_point_mass_accept_probabilities_in_closed_form():
    """Two children x1, x2: P(x1) = p1, P(x2) = (1 - p1) p2 / (1 - p1) = p2,
    and the bonus never repeats a rejected child."""
    vocab, trials = 5, 20000
    xt = np.array([1.0, 0.2, -0.5, 0.7, -1.2])
    p = scipy.special.softmax(xt)
    tree = _star_tree(0, [3, 0], 2)
    hits = np.zeros(3)
    for trial in range(trials):
        path, a, bonus, _ = oracle.accept_point_mass(tree, np.arange(3), np.vstack([xt, xt, xt]),
                                                     seed=2, b=0, cycle_no=trial)
        if a == 0:
            assert bonus not in (3, 0)
            hits[2] += 1
        else:
            hits[path[1] - 1] += 1
    expect = np.array([p[3], p[0], 1 - p[3] - p[0]]) * trials
    chi2 = ((hits - expect) ** 2 / expect).sum()
    assert scipy.stats.chi2.sf(chi2, 2) > 1e-4, (hits / trials, expect / trials)


def test_point_mass_certain_and_impossible_children():
    vocab = 4
    sure = np.array([30.0, -30.0, -30.0, -30.0])       # p(0) ~ 1
    tree = _star_tree(0, [0], 1)
    for c in range(20):
        path, a, _, _ = oracle.accept_point_mass(tree, np.arange(2), np.vstack([sure, sure]),
                                                 seed=4, b=0, cycle_no=c)
        assert a == 1
    never = np.array([0.0, -1e4, 0.0, 0.0])            # p(1) = 0
    tree = _star_tree(0, [1], 1)
    for c in range(20):
        path, a, bonus, _ = oracle.accept_point_mass(tree, np.arange(2), np.vstack([never, never]),
                                                     seed=4, b=0, cycle_no=c)
        assert a == 0 and bonus != 1


def test_splitmix64_published_vector():
    with open(os.path.join(GOLDEN, "splitmix64_seed0.txt")) as f:
        vals = [int(line, 16) for line in f if line.strip() and not line.startswith("#")]
    assert oracle.splitmix64_stream(0, 4) == vals


def test_uniforms_exact_and_in_range():
    for s in range(200):
        u = oracle.uniform_ratio(11, 2, 3, s % 7, s)
        assert 0.0 <= u < 1.0 and float(np.float32(u)) == u and (u * 2 ** 24).is_integer()
    g = oracle.uniform_gumbel(11, 2, 3, 4, np.arange(5000))
    assert (g > 0).all() and (g < 1).all()
    assert np.array_equal(g.astype(np.float32).astype(np.float64), g)
    # roughly uniform
    assert scipy.stats.kstest(g, "uniform").pvalue > 1e-4


# ----------------------------------------------------------- compaction pins
def test_compaction_copies_and_preserves():
    rng = np.random.default_rng(0)
    cache = rng.standard_normal((2, 3, 20, 4))
    ctx, path = 10, [0, 2, 3]  # destination 1 reads slot 2 while 2 is a destination
    out = oracle.compact_kv(cache, ctx, path)
    for t, s in enumerate(path):
        assert np.array_equal(out[..., ctx + t, :], cache[..., ctx + s, :])
    untouched = [r for r in range(20) if not (ctx <= r < ctx + len(path))]
    assert np.array_equal(out[..., untouched, :], cache[..., untouched, :])


def test_compaction_identity_path():
    cache = np.arange(2 * 12 * 3, dtype=np.float64).reshape(2, 12, 3)
    assert np.array_equal(oracle.compact_kv(cache, 4, [0, 1, 2, 3]), cache)


# ------------------------------------------------- planted mistakes are caught
def _mutant_log_softmax_dropped_lse(x):
    x = np.asarray(x, np.float64)
    return x - x.max(), float(x.max())  # mistake: drops log sum exp(x - m)


# ------------------------------------------------------ policy observation pins
def test_worked_example_observations():
    """Depth and size observations of the hand-worked tree: the exact cums of
    the worked nodes (as fractions), selected by their depth, not by id."""
    g = _worked()
    rows = _rows_from_weights(g["draft_row_weights"])
    W, ctx = g["W"], g["ctx"]
    by_depth = {}
    for node in sorted(g["expected_nodes"], key=lambda n: n["id"]):
        by_depth.setdefault(node["depth"], []).append(math.log(Fraction(node["cum"])))
    for L in (1, 2, 3):
        tree = oracle.grow_tree(g["root_token"], rows, W, L)
        obs = O.depth_observation(tree, ctx)
        want = by_depth[L]
        assert len(obs) == W * W + 2
        assert obs[:len(want)] == pytest.approx(want, abs=1e-12)
        assert (obs[len(want):W * W] == O.POLICY_PAD).all()
        assert obs[W * W] == L and obs[W * W + 1] == ctx
    tree = oracle.grow_tree(g["root_token"], rows, W, g["L"])
    v_pad = 40
    obs = O.size_observation(tree, ctx, v_pad)
    allc = [math.log(Fraction(n["cum"])) if n["id"] else 0.0
            for n in sorted(g["expected_nodes"], key=lambda n: n["id"])]
    assert obs[:len(allc)] == pytest.approx(allc, abs=1e-12)
    assert (obs[len(allc):v_pad] == O.POLICY_PAD).all()
    assert obs[v_pad] == g["L"] and obs[v_pad + 1] == ctx


@pytest.mark.parametrize("W,L", [(1, 3), (2, 1), (3, 4), (4, 2), (10, 3)])
def test_observations_against_depth_and_path_sums(W, L):
    """The depth observation holds exactly the level's candidates (the nodes
    whose depth is L: W at level 1, the whole W^2 pool after), and the size
    observation every node's path sum of scipy log-probs; the count of real
    entries is the paper's 1 + W + (D-2) W^2 with D = L + 1."""
    tree, rows, _ = _random_tree(W * 31 + L, W, L, vocab=40)
    ctx = 777 + L
    d = O.depth_observation(tree, ctx)
    level = [tree.cum[i] for i in range(tree.n_nodes) if tree.depth[i] == L]
    assert len(level) == (W if L == 1 else W * W)
    np.testing.assert_array_equal(d[:len(level)], level)
    assert (d[len(level):W * W] == O.POLICY_PAD).all()
    assert list(d[W * W:]) == [L, ctx]
    v_pad = 1 + W + (L - 1) * W * W + 7
    s = O.size_observation(tree, ctx, v_pad)
    D = L + 1
    n_real = 1 + W + (D - 2) * W * W
    for c in range(n_real):
        total, a = 0.0, c
        while tree.parent[a] >= 0:
            p = tree.parent[a]
            total += scipy.special.log_softmax(rows[tree.xrow[p]])[tree.token[a]]
            a = p
        assert s[c] == pytest.approx(total, abs=1e-12)
    assert (s[n_real:v_pad] == O.POLICY_PAD).all()
    assert list(s[v_pad:]) == [L, ctx]


# ----------------------------------------------------------- policy MLP pins
def test_mlp_hand_worked():
    """x = (1, 2); hidden = relu(x W1 + b1) = relu(3.5, -7) = (3.5, 0);
    logits = (3.5*2, 3.5*(-1) + 1) = (7, -2.5), worked by hand."""
    w1, b1 = [[1.0, -1.0], [1.0, -3.0]], [0.5, 0.0]
    w2, b2 = [[2.0, -1.0], [5.0, 7.0]], [0.0, 1.0]
    z = O.mlp_forward(np.array([[1.0, 2.0]]), [(w1, b1), (w2, b2)])
    assert z.tolist() == [[7.0, -2.5]]
    assert O.first_argmax(z[0]) == 0


def test_mlp_against_torch_linear_layers():
    """torch.nn.Linear holds W as [out][in] and computes x W^T + b; the
    oracle's [in][out] matrices transposed into it give the same network
    (n_in, hidden and n_out all differ, so a transposed operand cannot pass)."""
    rng = np.random.default_rng(5)
    dims = [7, 11, 5, 3]
    layers = [(rng.standard_normal((a, b)), rng.standard_normal(b)) for a, b in zip(dims[:-1], dims[1:])]
    mods = []
    for i, (w, b) in enumerate(layers):
        lin = torch.nn.Linear(w.shape[0], w.shape[1], dtype=torch.float64)
        with torch.no_grad():
            lin.weight.copy_(torch.from_numpy(w.T))
            lin.bias.copy_(torch.from_numpy(b))
        mods.append(lin)
        if i + 1 < len(layers):
            mods.append(torch.nn.ReLU())
    x = rng.standard_normal((4, dims[0]))
    ref = torch.nn.Sequential(*mods)(torch.from_numpy(x)).detach().numpy()
    np.testing.assert_allclose(O.mlp_forward(x, layers), ref, rtol=1e-13, atol=1e-13)


def test_argmax_ties_to_the_lower_action():
    assert O.first_argmax([1.0, 3.0, 3.0, 2.0]) == 1
    assert O.first_argmax([0.0, 0.0]) == 0


def _bias_only(n_in, n_out, action):
    w = np.zeros((n_in, n_out))
    b = np.zeros(n_out)
    b[action] = 1.0
    return [(w, b)]


def test_size_policy_maps_actions_to_20_through_240():
    """12 actions map linearly onto V = 20..240 (App. A.2); N = V + 1 counts
    the root and is capped by the verify buffer and the tree size."""
    big, _, _ = _random_tree(3, 10, 3, vocab=50)     # 211 nodes
    v_pad = big.n_nodes
    got = [O.size_policy_step(big, 100, v_pad, _bias_only(v_pad + 2, 12, a), 256)[0]
           for a in range(12)]
    assert got == [21, 41, 61, 81, 101, 121, 141, 161, 181, 201, 211, 211]
    assert O.size_policy_step(big, 100, v_pad, _bias_only(v_pad + 2, 12, 11), 64)[0] == 64
    small, _, _ = _random_tree(4, 2, 2, vocab=9)     # 7 nodes
    assert O.size_policy_step(small, 5, 7, _bias_only(9, 12, 0), 256)[0] == 7


def test_depth_policy_continue_stop_and_limits():
    tree, _, _ = _random_tree(6, 3, 2, vocab=20)
    cont, stop = _bias_only(11, 2, 1), _bias_only(11, 2, 0)
    assert O.depth_policy_step(tree, 9, cont, True, 4)[0] is True
    assert O.depth_policy_step(tree, 9, stop, True, 4)[0] is False
    assert O.depth_policy_step(tree, 9, cont, False, 4)[0] is False    # already stopped
    assert O.depth_policy_step(tree, 9, cont, True, 2)[0] is False     # no level left


def test_planted_mistake_in_log_softmax_is_caught(monkeypatch):
    monkeypatch.setattr(O, "log_softmax", _mutant_log_softmax_dropped_lse)
    with pytest.raises(AssertionError):
        test_worked_example_tree()


def test_planted_mistake_in_tiebreak_is_caught(monkeypatch):
    def rank_hi_first(x, W):
        x = np.asarray(x, np.float64)
        return np.lexsort((-np.arange(x.size), -x))[:W]  # mistake: ties to higher id
    monkeypatch.setattr(O, "rank_by_logit", rank_hi_first)
    with pytest.raises(AssertionError):
        test_worked_example_tree()


def test_planted_mistake_in_attention_scale_is_caught(monkeypatch):
    real = O.tree_attention

    def wrong(q, k, v, ctx, mask, scale):
        return real(q, k, v, ctx, mask, scale * 1.0001)
    monkeypatch.setattr(oracle, "tree_attention", wrong)
    with pytest.raises(AssertionError):
        test_attention_all_ones_equals_unmasked()


def test_planted_mistake_in_attention_mask_transpose_is_caught(monkeypatch):
    real = O.tree_attention

    def wrong(q, k, v, ctx, mask, scale):
        return real(q, k, v, ctx, np.asarray(mask).T, scale)
    monkeypatch.setattr(oracle, "tree_attention", wrong)
    with pytest.raises(AssertionError):
        test_attention_chain_equals_causal()


def test_planted_mistake_in_residual_is_caught(monkeypatch):
    """A sign error in the residual max(p - q, 0) breaks losslessness."""
    real_max = np.maximum

    def accept_wrong(tree, chosen, target_rows, draft_rows, seed, b, cycle_no):
        orig = O.np.maximum
        O.np.maximum = lambda a, c: real_max(-a, c)  # mistake: max(q - p, 0)
        try:
            return real_accept(tree, chosen, target_rows, draft_rows, seed, b, cycle_no)
        finally:
            O.np.maximum = orig
    real_accept = O.accept_stochastic
    monkeypatch.setattr(oracle, "accept_stochastic", accept_wrong)
    with pytest.raises(AssertionError):
        test_stochastic_preserves_target_distribution()


def test_planted_mistake_in_greedy_walk_is_caught(monkeypatch):
    real = O.accept_greedy

    def wrong(tree, chosen, target_rows):
        path, a, bonus = real(tree, chosen, target_rows)
        return path[:-1] or path, max(a - 1, 0), bonus  # mistake: off by one
    monkeypatch.setattr(oracle, "accept_greedy", wrong)
    with pytest.raises(AssertionError):
        test_worked_example_select_and_accept()


def test_brute_force_enumeration_is_exhaustive():
    """Self-check of the brute-force helper on a hand-made tree."""
    t = _star_tree(0, [1, 2], 2)
    t._add(3, 1, 2, 0.0)  # node 3 under node 1
    ids = np.arange(4)
    target = np.zeros((4, 4))
    target[0, 1] = 1  # root predicts 1 -> slot 1
    target[1, 3] = 1  # slot 1 predicts 3 -> slot 3
    target[3, 2] = 1
    best, bonus = _brute_force_greedy(t, ids, target)
    assert best == [0, 1, 3] and bonus == 2


def test_planted_mistake_in_depth_observation_is_caught(monkeypatch):
    def shifted(tree, ctx):   # mistake: the level's first id off by one
        out = np.full(tree.W * tree.W + 2, O.POLICY_PAD)
        lvl, W = tree.levels, tree.W
        first = 1 if lvl == 1 else W + (lvl - 2) * W * W
        cnt = W if lvl == 1 else W * W
        out[:cnt] = tree.cum[first:first + cnt]
        out[-2:] = (lvl, ctx)
        return out
    monkeypatch.setattr(O, "depth_observation", shifted)
    with pytest.raises(AssertionError):
        test_observations_against_depth_and_path_sums(3, 4)


def test_planted_mistake_in_mlp_is_caught(monkeypatch):
    def no_relu(x, layers):   # mistake: the hidden ReLU dropped
        h = np.asarray(x, np.float64)
        for w, b in layers:
            h = h @ np.asarray(w, np.float64) + np.asarray(b, np.float64)
        return h
    monkeypatch.setattr(O, "mlp_forward", no_relu)
    with pytest.raises(AssertionError):
        test_mlp_hand_worked()

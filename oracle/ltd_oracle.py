"""fp64 oracle of the LTD draft-and-verify cycle (test infrastructure only).

The cycle (paper §3.2 "Draft-and-Verify Cycle") has three parts, each written
here as the plain definition, in fp64, with exhaustive sorts and lower-index
tie-breaking:

* Draft Tree Generation (§3.2): beam-like expansion.  Level 1 takes the top-W
  tokens of the root's draft distribution; every later level gives each of the
  W frontier nodes W children (a W^2 pool, all of which join the tree) and
  keeps the W children with the highest cumulative path log-probability as
  the next frontier.
* Candidate Token Selection (§3.2): the tree holds V_all = 1 + W + (D-2)W^2
  tokens; the V with the highest overall probability are flattened with a
  tree attention mask.
* Draft Tree Verification (§3.2, tree attention after SpecInfer, §2.1): one
  target forward over the V tokens, each attending to the prefix and to its
  own ancestors; the path is accepted up to the first mismatch and the
  target's token there is the bonus and the next root.  The stochastic rule
  (T = 1) is SpecInfer's multi-candidate speculative sampling with the
  Leviathan/Chen ratio test (the paper only states that the target
  distribution is preserved, §1 and §5.1 "Metrics").

Around the cycle, also written out here: the two policies' observations and
network (Appendix A.2: depth observation, size observation, ReLU MLP,
argmax decisions), two more stochastic verification rules for trees whose
children are not i.i.d. draws (point-mass proposals, proposals without
replacement), every stochastic rule at a temperature T, and the target
LM head's logits with the row statistics acceptance reads.

Readings where the paper is silent or loose:

* depth: L = levels below the root, V_all = 1 + W + (L-1) W^2 (the paper's D
  is L + 1);
* N counts the root, which always sits in slot 0 (N = 1 is plain decode);
* ranking inside a row is by the raw logit (exact on both sides), ties to the
  lower token id; across nodes by cumulative log-prob, ties to the lower node
  id; argmax ties to the lower token id;
* the bonus of a stochastic cycle is drawn by Gumbel-max from the (residual)
  target distribution with counter-based uniforms; sampling is exact.

The draft row store: every sequence owns R = 1 + (L_max-1) W rows of draft
logits.  Row 0 is the root's distribution (level 1); the row of frontier rank
r at level l >= 2 is 1 + (l-2) W + r.  Node ids are assigned in expansion
order: level 1 gives ids 1..W in rank order; level l >= 2 gives the child of
rank c of frontier rank r the id base_l + r W + c, base_l = 1 + W + (l-2) W^2.
"""

from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

MASK64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15  # splitmix64 increment (golden ratio, Steele et al. 2014)


# ---------------------------------------------------------------- utilities
def v_all(W: int, L: int) -> int:
    """Tree size after L levels below the root: 1 + W + (L-1) W^2 (§3.2,
    Candidate Token Selection, with the paper's D = L + 1)."""
    if L <= 0:
        return 1
    return 1 + W + (L - 1) * W * W


def log_softmax(x: np.ndarray) -> tuple[np.ndarray, float]:
    """log p_t = x_t - logsumexp(x) in fp64; returns (log p, logsumexp)."""
    x = np.asarray(x, dtype=np.float64)
    m = float(x.max())
    lse = m + float(np.log(np.exp(x - m).sum()))
    return x - lse, lse


def rank_by_logit(x: np.ndarray, W: int) -> np.ndarray:
    """Token ids of the W largest logits, ordered by (logit desc, id asc)."""
    x = np.asarray(x, dtype=np.float64)
    order = np.lexsort((np.arange(x.size), -x))
    return order[:W]


def softmax_t(x: np.ndarray, temperature: float = 1.0) -> np.ndarray:
    """softmax(x / T) in fp64: the distribution sampled at temperature T
    (T = 1 is the plain softmax)."""
    assert temperature > 0.0
    return np.exp(log_softmax(np.asarray(x, dtype=np.float64) / temperature)[0])


def mask_words(mask: np.ndarray) -> np.ndarray:
    """Pack a boolean [N][N'] mask into uint32 words: bit j of row i lives in
    word j // 32 at bit position j % 32."""
    n_rows, n_cols = mask.shape
    n_words = (n_cols + 31) // 32
    out = np.zeros((n_rows, n_words), dtype=np.uint32)
    for i in range(n_rows):
        for j in range(n_cols):
            if mask[i, j]:
                out[i, j // 32] |= np.uint32(1 << (j % 32))
    return out


# ------------------------------------------------------------ tree generation
@dataclass
class OracleTree:
    """Draft tree of one sequence as plain Python lists (node id = index)."""

    W: int
    token: list = field(default_factory=list)
    parent: list = field(default_factory=list)
    depth: list = field(default_factory=list)
    cum: list = field(default_factory=list)
    xrow: list = field(default_factory=list)   # draft row that expanded the node, -1 if none
    xlse: list = field(default_factory=list)   # logsumexp of that row
    frontier: list = field(default_factory=list)
    levels: int = 0
    cut_margins: list = field(default_factory=list)  # fp64 gap at every frontier cut

    @classmethod
    def rooted(cls, root_token: int, W: int) -> "OracleTree":
        t = cls(W=W)
        t.token.append(int(root_token))
        t.parent.append(-1)
        t.depth.append(0)
        t.cum.append(0.0)
        t.xrow.append(-1)
        t.xlse.append(0.0)
        t.frontier = [0]
        return t

    def _add(self, token, parent, depth, cum):
        self.token.append(int(token))
        self.parent.append(int(parent))
        self.depth.append(int(depth))
        self.cum.append(float(cum))
        self.xrow.append(-1)
        self.xlse.append(0.0)
        return len(self.token) - 1

    @property
    def n_nodes(self) -> int:
        return len(self.token)


def expand_level(tree: OracleTree, rows: np.ndarray) -> None:
    """Grow ``tree`` by one level (§3.2, Draft Tree Generation).

    ``rows[r]`` is the draft model's logit row for frontier rank r (one row at
    level 1, W rows afterwards).  Every frontier node's W best tokens become
    its children with cum = cum(parent) + log p(token); at level 1 all W
    children are the frontier, afterwards the frontier is the W children of
    the W^2 pool with the largest cum (ties to the lower node id).
    """
    W = tree.W
    level = tree.levels + 1
    rows = np.asarray(rows, dtype=np.float64)
    assert rows.shape[0] == len(tree.frontier), "one draft row per frontier node"
    base = tree.n_nodes
    children = []
    for r, f in enumerate(tree.frontier):
        logp, lse = log_softmax(rows[r])
        tree.xrow[f] = 0 if level == 1 else 1 + (level - 2) * W + r
        tree.xlse[f] = lse
        for c, t in enumerate(rank_by_logit(rows[r], W)):
            nid = tree._add(t, f, level, tree.cum[f] + logp[t])
            assert nid == base + r * W + c
            children.append(nid)
    if level == 1:
        tree.frontier = children
    else:
        ids = np.array(children)
        cums = np.array([tree.cum[i] for i in children])
        order = np.lexsort((ids, -cums))
        tree.frontier = [int(ids[o]) for o in order[:W]]
        if len(order) > W:
            tree.cut_margins.append(float(cums[order[W - 1]] - cums[order[W]]))
    tree.levels = level


def grow_tree(root_token: int, draft_rows: np.ndarray, W: int, L: int) -> OracleTree:
    """Build the L-level tree from one sequence's draft row store."""
    tree = OracleTree.rooted(root_token, W)
    for level in range(1, L + 1):
        if level == 1:
            rows = draft_rows[0:1]
        else:
            r0 = 1 + (level - 2) * W
            rows = draft_rows[r0:r0 + W]
        expand_level(tree, rows)
    return tree


# --------------------------------------------------------------- selection
def select_verify(tree: OracleTree, N: int, ctx: int):
    """Candidate Token Selection (§3.2).

    The N-1 non-root nodes with the largest cum (ties to the lower id) plus
    the root, flattened in ascending id order (slots).  Returns
    (ids, pos, mask, margin): pos = ctx + depth, mask[i, j] is True iff slot
    j lies on the root-to-slot-i path, margin is the fp64 gap at the cut
    (inf when nothing is cut).
    """
    n = tree.n_nodes
    assert 1 <= N <= n
    ids = np.arange(1, n)
    cums = np.array(tree.cum[1:], dtype=np.float64)
    order = np.lexsort((ids, -cums))
    chosen = sorted([0] + [int(ids[o]) for o in order[:N - 1]])
    margin = float("inf")
    if N - 1 < n - 1:
        margin = float(cums[order[N - 2]] - cums[order[N - 1]]) if N >= 2 else float("inf")
    slot_of = {nid: s for s, nid in enumerate(chosen)}
    pos = np.array([ctx + tree.depth[nid] for nid in chosen], dtype=np.int64)
    mask = np.zeros((N, N), dtype=bool)
    for i, nid in enumerate(chosen):
        a = nid
        while a >= 0:
            assert a in slot_of, "selection must be ancestor-closed"
            mask[i, slot_of[a]] = True
            a = tree.parent[a]
    return np.array(chosen, dtype=np.int64), pos, mask, margin


# ---------------------------------------------------------------- attention
def tree_attention(q, k_cache, v_cache, ctx: int, mask, scale: float):
    """Tree attention of the N verified tokens (§3.2 Draft Tree Verification;
    SpecInfer-style tree mask, §2.1), fp64.

    q: [N][Hq][d]; k_cache, v_cache: [Hkv][S_cap][d] with the N new tokens at
    rows ctx..ctx+N-1 in slot order.  Query head h reads KV head h // (Hq/Hkv).
    Slot i attends to keys 0..ctx-1 and to ctx+j for every j with mask[i, j].
    Returns o: [N][Hq][d] = softmax(q k^T * scale) v over those keys.
    """
    q = np.asarray(q, dtype=np.float64)
    K = np.asarray(k_cache, dtype=np.float64)
    V = np.asarray(v_cache, dtype=np.float64)
    N, Hq, d = q.shape
    Hkv = K.shape[0]
    G = Hq // Hkv
    allowed = np.concatenate([np.ones((N, ctx), dtype=bool), np.asarray(mask, bool)], axis=1)
    out = np.zeros((N, Hq, d), dtype=np.float64)
    for h in range(Hq):
        kv = h // G
        keys = K[kv, :ctx + N]
        vals = V[kv, :ctx + N]
        s = (q[:, h, :] @ keys.T) * scale
        s = np.where(allowed, s, -np.inf)
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p = p / p.sum(axis=1, keepdims=True)
        out[:, h, :] = p @ vals
    return out


# ------------------------------------------------------- counter-based RNG
def mix64(z: int) -> int:
    """splitmix64 output finaliser (Steele, Lea & Flood 2014; Vigna)."""
    z &= MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
    return z ^ (z >> 31)


def splitmix64_stream(seed: int, count: int) -> list:
    """The published splitmix64 sequence: state += GAMMA; out = mix64(state)."""
    s = seed & MASK64
    out = []
    for _ in range(count):
        s = (s + GAMMA) & MASK64
        out.append(mix64(s))
    return out


def _hash_words(seed: int, words) -> int:
    """Key a splitmix64 step on a tuple of integers:
    h_0 = seed, h_{j+1} = mix64(h_j + GAMMA * (j + 1) + w_j)  (mod 2^64)."""
    h = seed & MASK64
    for j, w in enumerate(words):
        h = mix64((h + GAMMA * (j + 1) + (int(w) & MASK64)) & MASK64)
    return h


STREAM_RATIO = 0
STREAM_BONUS = 1


def uniform_ratio(seed, b, cycle_no, slot, i) -> float:
    """U[0,1) for the ratio test of the i-th child of slot ``slot``:
    the top 24 bits of the hash times 2^-24 (exact in fp32 and fp64)."""
    h = _hash_words(seed, (b, cycle_no, STREAM_RATIO, slot, i))
    return (h >> 40) * 2.0 ** -24


def _mix64_np(z: np.ndarray) -> np.ndarray:
    """mix64 on uint64 arrays (numpy integer arithmetic wraps mod 2^64)."""
    z = z ^ (z >> np.uint64(30))
    z = z * np.uint64(0xBF58476D1CE4E5B9)
    z = z ^ (z >> np.uint64(27))
    z = z * np.uint64(0x94D049BB133111EB)
    return z ^ (z >> np.uint64(31))


def uniform_gumbel(seed, b, cycle_no, slot, tokens: np.ndarray) -> np.ndarray:
    """U(0,1) per token for the Gumbel-max bonus draw at slot ``slot``:
    (2 * (h >> 41) + 1) * 2^-24, never 0 or 1, exact in fp32 and fp64.
    h = _hash_words(seed, (b, cycle, STREAM_BONUS, slot, token)), with the
    last step evaluated on a uint64 array."""
    h4 = _hash_words(seed, (b, cycle_no, STREAM_BONUS, slot))
    t = np.asarray(tokens, dtype=np.int64).astype(np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(h4) + np.uint64((GAMMA * 5) & MASK64) + t
        h = _mix64_np(z)
    return (2.0 * (h >> np.uint64(41)).astype(np.float64) + 1.0) * 2.0 ** -24


# ---------------------------------------------------------------- acceptance
def _children_slots(tree: OracleTree, chosen) -> dict:
    """slot -> list of child slots (ascending) inside the verified set."""
    slot_of = {int(nid): s for s, nid in enumerate(chosen)}
    kids = {s: [] for s in range(len(chosen))}
    for s, nid in enumerate(chosen):
        p = tree.parent[int(nid)]
        if p >= 0:
            kids[slot_of[p]].append(s)
    return kids


def accept_greedy(tree: OracleTree, chosen, target_rows):
    """Greedy verification (§3.2 Draft Tree Verification).

    Walk from slot 0: the target's prediction at the current slot is
    argmax(target_rows[slot]) (ties to the lower id); move to the child slot
    whose token equals it, else stop.  Returns (path slots, accept_len, bonus).
    Sibling tokens are distinct (a top-W of one row), so the path is unique.
    """
    kids = _children_slots(tree, chosen)
    slot = 0
    path = [0]
    while True:
        pred = int(np.argmax(np.asarray(target_rows[slot], dtype=np.float64)))
        nxt = [c for c in kids[slot] if tree.token[int(chosen[c])] == pred]
        if not nxt:
            return path, len(path) - 1, pred
        slot = nxt[0]
        path.append(slot)


def accept_stochastic(tree: OracleTree, chosen, target_rows, draft_rows, seed, b, cycle_no,
                      temperature: float = 1.0):
    """Stochastic verification at temperature T (reading: SpecInfer's
    multi-candidate speculative sampling with the Leviathan/Chen ratio test;
    the paper's experiments use T = 1, the default).

    At the current slot u: p = softmax(target row of u / T), q =
    softmax(draft row that expanded u / T).  For each verified child x_i of u in slot order: accept
    if r_i * q(x_i) < p(x_i) with r_i = uniform_ratio(seed, b, cycle, u, i);
    otherwise p <- max(p - q, 0) / sum (p kept when that sum is 0).  When no
    child is accepted, the bonus is argmax_t [log p(t) - log(-log g_t)] over
    tokens with p(t) > 0 (Gumbel-max; g_t = uniform_gumbel), ties to the
    lower id.  Returns (path, accept_len, bonus, margins) where margins holds
    the relative fp64 gap of every ratio test and of the bonus argmax.
    """
    kids = _children_slots(tree, chosen)
    slot = 0
    path = [0]
    margins = []
    while True:
        u = int(chosen[slot])
        p = softmax_t(target_rows[slot], temperature)
        accepted = None
        if kids[slot]:
            q = softmax_t(draft_rows[tree.xrow[u]], temperature)
            for i, c in enumerate(kids[slot]):
                x = tree.token[int(chosen[c])]
                r = uniform_ratio(seed, b, cycle_no, slot, i)
                lhs, rhs = r * q[x], p[x]
                margins.append(abs(lhs - rhs) / max(abs(rhs), 1e-300))
                if lhs < rhs:
                    accepted = c
                    break
                res = np.maximum(p - q, 0.0)
                z = res.sum()
                if z > 0:
                    p = res / z
        if accepted is None:
            vocab = p.size
            g = uniform_gumbel(seed, b, cycle_no, slot, np.arange(vocab))
            with np.errstate(divide="ignore"):
                score = np.where(p > 0, np.log(p) - np.log(-np.log(g)), -np.inf)
            bonus = int(np.argmax(score))
            top2 = np.sort(score)[-2:]
            margins.append(float(top2[1] - top2[0]) if np.isfinite(top2[0]) else float("inf"))
            return path, len(path) - 1, bonus, margins
        path.append(accepted)
        slot = accepted


def accept_without_replacement(tree: OracleTree, chosen, target_rows, draft_rows, seed, b,
                               cycle_no, temperature: float = 1.0):
    """Stochastic verification at temperature T (p and q as in
    accept_stochastic) for children drawn from q without replacement (a variant of the rule above: recursive rejection sampling).
    Child x_i is proposed by q_i, the draft distribution with the children
    rejected so far removed and renormalised (q_0 = q); it is accepted if
    r_i q_i(x_i) < p_i(x_i), else p_{i+1} = max(p_i - q_i, 0) / sum (p_i kept
    when that sum is 0) and q_{i+1} = q_i with x_i removed, renormalised.
    With no child accepted the bonus is the Gumbel-max draw from the last p.
    Same uniforms and return value as accept_stochastic."""
    kids = _children_slots(tree, chosen)
    slot = 0
    path = [0]
    margins = []
    while True:
        u = int(chosen[slot])
        p = softmax_t(target_rows[slot], temperature)
        accepted = None
        if kids[slot]:
            q = softmax_t(draft_rows[tree.xrow[u]], temperature)
            for i, c in enumerate(kids[slot]):
                x = tree.token[int(chosen[c])]
                r = uniform_ratio(seed, b, cycle_no, slot, i)
                lhs, rhs = r * q[x], p[x]
                margins.append(abs(lhs - rhs) / max(abs(rhs), 1e-300))
                if lhs < rhs:
                    accepted = c
                    break
                res = np.maximum(p - q, 0.0)
                z = res.sum()
                if z > 0:
                    p = res / z
                q = q.copy()
                q[x] = 0.0
                qs = q.sum()
                if qs > 0:
                    q = q / qs
        if accepted is None:
            vocab = p.size
            g = uniform_gumbel(seed, b, cycle_no, slot, np.arange(vocab))
            with np.errstate(divide="ignore"):
                score = np.where(p > 0, np.log(p) - np.log(-np.log(g)), -np.inf)
            bonus = int(np.argmax(score))
            top2 = np.sort(score)[-2:]
            margins.append(float(top2[1] - top2[0]) if np.isfinite(top2[0]) else float("inf"))
            return path, len(path) - 1, bonus, margins
        path.append(accepted)
        slot = accepted


def accept_point_mass(tree: OracleTree, chosen, target_rows, seed, b, cycle_no,
                      temperature: float = 1.0):
    """Stochastic verification at temperature T (p = softmax(target row / T))
    with point-mass proposals (a variant
    of the rule above for a tree whose children are the draft's top-W tokens,
    not samples from q: each child is a deterministic proposal, so its
    proposal distribution is a point mass on its token).

    At the current slot u: p = softmax(target row of u); the rejected set R
    starts empty.  Child x_i (slot order) is accepted if
    r_i (1 - p(R)) < p(x_i), i.e. r_i < p(x_i) / (1 - p(R)), the probability
    of x_i under p restricted to the tokens not yet rejected; otherwise x_i
    joins R.  With no child accepted the bonus is the Gumbel-max draw
    argmax_t [log p(t) - log(-log g_t)] over the tokens outside R with
    p(t) > 0.  Offering tokens one at a time this way and sampling the rest
    from the restricted p emits a token distributed exactly as p, for any
    set of children.  Returns (path, accept_len, bonus, margins) like
    accept_stochastic."""
    kids = _children_slots(tree, chosen)
    slot = 0
    path = [0]
    margins = []
    while True:
        p = softmax_t(target_rows[slot], temperature)
        accepted = None
        rejected = []
        removed = 0.0
        for i, c in enumerate(kids[slot]):
            x = tree.token[int(chosen[c])]
            r = uniform_ratio(seed, b, cycle_no, slot, i)
            lhs, rhs = r * (1.0 - removed), p[x]
            margins.append(abs(lhs - rhs) / max(abs(rhs), 1e-300))
            if lhs < rhs:
                accepted = c
                break
            rejected.append(x)
            removed += p[x]
        if accepted is None:
            vocab = p.size
            g = uniform_gumbel(seed, b, cycle_no, slot, np.arange(vocab))
            keep = p.copy()
            keep[rejected] = 0.0
            with np.errstate(divide="ignore"):
                score = np.where(keep > 0, np.log(keep) - np.log(-np.log(g)), -np.inf)
            bonus = int(np.argmax(score))
            top2 = np.sort(score)[-2:]
            margins.append(float(top2[1] - top2[0]) if np.isfinite(top2[0]) else float("inf"))
            return path, len(path) - 1, bonus, margins
        path.append(accepted)
        slot = accepted


# ---------------------------------------------------------------- compaction
def compact_kv(cache: np.ndarray, ctx: int, path) -> np.ndarray:
    """KV compaction implied by "discards the remainder" (§3.2 Draft Tree
    Verification): rows ctx + t <- rows ctx + path[t] for t = 0..len(path)-1,
    reading every source before any write.  ``cache``: [..., S_cap, d]; the
    returned copy has all other rows unchanged."""
    out = np.array(cache, copy=True)
    src = np.array(cache, copy=True)
    for t, s in enumerate(path):
        out[..., ctx + t, :] = src[..., ctx + int(s), :]
    return out


# ------------------------------------------------------- target LM-head rows
def lm_head_row_stats(hidden: np.ndarray, weight: np.ndarray):
    """The target's verification logits and the row statistics acceptance
    reads from them (section 3.2, "Draft Tree Verification": one target
    forward over the verified tokens; the last layer maps each hidden state
    to vocabulary logits).  logits[r][v] = sum_k hidden[r][k] weight[v][k]
    in fp64; per row the max, the log-sum-exp and the argmax (ties to the
    lower token id).  Returns (logits, row_max, row_lse, row_argmax)."""
    h = np.asarray(hidden, dtype=np.float64)
    w = np.asarray(weight, dtype=np.float64)
    logits = h @ w.T
    row_max = logits.max(axis=1)
    row_lse = row_max + np.log(np.exp(logits - row_max[:, None]).sum(axis=1))
    row_argmax = np.array([first_argmax(r) for r in logits], dtype=np.int64)
    return logits, row_max, row_lse, row_argmax


# --------------------------------------------------------- policy observations
POLICY_PAD = -100.0   # fill of unused observation slots (the paper only says "padded")


def depth_observation(tree: OracleTree, ctx: int) -> np.ndarray:
    """Observation of the depth policy after the last built level (Appendix
    A.2, "Depth Policy", observation space): the cumulative log-probabilities
    of the candidates that level produced, W^2 of them (W at level 1, padded
    to W^2 with POLICY_PAD), in node-id order, then the draft depth D (levels
    built) and the sequence length L = ctx.  Returned in fp64."""
    W, lvl = tree.W, tree.levels
    out = np.full(W * W + 2, POLICY_PAD, np.float64)
    if lvl >= 1:
        first = 1 if lvl == 1 else 1 + W + (lvl - 2) * W * W
        count = W if lvl == 1 else W * W
        out[:count] = tree.cum[first:first + count]
    out[W * W] = lvl
    out[W * W + 1] = ctx
    return out


def size_observation(tree: OracleTree, ctx: int, v_pad: int) -> np.ndarray:
    """Observation of the size policy after drafting (Appendix A.2, "Size
    Policy", observation space): the cumulative log-probabilities of all
    1 + W + (L-1) W^2 tree nodes, root included, in node-id order, padded to
    ``v_pad`` with POLICY_PAD, then D (levels built) and L = ctx."""
    n = tree.n_nodes
    assert v_pad >= n
    out = np.full(v_pad + 2, POLICY_PAD, np.float64)
    out[:n] = tree.cum
    out[v_pad] = tree.levels
    out[v_pad + 1] = ctx
    return out


def mlp_forward(x: np.ndarray, layers) -> np.ndarray:
    """The policies' network (section 3.1; App. A.2 "Architecture"): a
    feed-forward ReLU network, h <- relu(h W + b) for every hidden layer and
    logits = h W + b for the last, with W stored [n_in][n_out].  fp64."""
    h = np.asarray(x, dtype=np.float64)
    for i, (w, b) in enumerate(layers):
        h = h @ np.asarray(w, np.float64) + np.asarray(b, np.float64)
        if i + 1 < len(layers):
            h = np.maximum(h, 0.0)
    return h


def first_argmax(z) -> int:
    """Index of the largest entry, ties to the lower index."""
    z = list(z)
    best = 0
    for j in range(1, len(z)):
        if z[j] > z[best]:
            best = j
    return best


def depth_policy_step(tree: OracleTree, ctx: int, layers, active: bool, max_depth: int):
    """One decision of the depth policy after the last built level (App. A.2
    "Depth Policy": a binary STOP / CONTINUE action per level).  Action 1 is
    CONTINUE; a sequence keeps drafting if it was active, the policy says
    CONTINUE and a level is left.  Returns (keep drafting, logits)."""
    z = mlp_forward(depth_observation(tree, ctx)[None, :], layers)[0]
    return bool(active and first_argmax(z) == 1 and tree.levels < max_depth), z


def size_policy_step(tree: OracleTree, ctx: int, v_pad: int, layers, n_cap: int):
    """The size policy's decision after the draft (App. A.2 "Size Policy":
    discrete actions mapped linearly onto V = 20, 40, ..., 240).  V counts
    candidate tokens, N = V + 1 counts the root too; N is capped by the verify
    buffer (n_cap) and by the tree's node count.  Returns (N, logits)."""
    z = mlp_forward(size_observation(tree, ctx, v_pad)[None, :], layers)[0]
    v = 20 + 20 * first_argmax(z)
    return min(1 + v, n_cap, tree.n_nodes), z


# ------------------------------------------------------------- whole cycle
def cycle(root_token, draft_rows, W, L, N, ctx, target_rows, mode="greedy",
          seed=0, b=0, cycle_no=0):
    """Draft -> select -> accept for one sequence (attention is separate since
    its output does not feed acceptance in this path)."""
    tree = grow_tree(root_token, draft_rows, W, L)
    ids, pos, mask, margin = select_verify(tree, N, ctx)
    if mode == "greedy":
        path, a, bonus = accept_greedy(tree, ids, target_rows)
        margins = []
    else:
        path, a, bonus, margins = accept_stochastic(tree, ids, target_rows, draft_rows,
                                                    seed, b, cycle_no)
    return dict(tree=tree, ids=ids, pos=pos, mask=mask, select_margin=margin,
                path=path, accept_len=a, bonus=bonus, margins=margins,
                new_ctx=ctx + 1 + a)

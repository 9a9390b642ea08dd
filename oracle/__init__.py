"""Plain fp64 CPU oracle for one LTD draft-and-verify cycle.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path (the CUDA library and
its Python binding) may import, call or link anything in this package; only
the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` use it.  It shares no code with the CUDA path: the two meet only
through the seeded inputs of ``paper_2603_01639_gb300.workload``.

Every function follows the paper (Zhang et al., "Learning To Draft: Adaptive
Speculative Decoding with Reinforcement Learning", §3.2 "Draft-and-Verify
Cycle"; Appendix A.2 for the policies' observations) or, where the paper is
silent, the reading stated in its docstring.  All pins are in
``tests/test_oracle_pins.py``; no function here is left "parity unpinned".
"""

from .ltd_oracle import (  # noqa: F401
    GAMMA,
    POLICY_PAD,
    OracleTree,
    accept_greedy,
    accept_point_mass,
    accept_stochastic,
    accept_without_replacement,
    compact_kv,
    cycle,
    depth_observation,
    depth_policy_step,
    expand_level,
    first_argmax,
    grow_tree,
    lm_head_row_stats,
    log_softmax,
    mask_words,
    mlp_forward,
    mix64,
    rank_by_logit,
    select_verify,
    size_observation,
    size_policy_step,
    softmax_t,
    splitmix64_stream,
    tree_attention,
    uniform_gumbel,
    uniform_ratio,
    v_all,
)

"""Seeded synthetic workloads for the draft-and-verify cycle.

This module draws random inputs and nothing else: it holds none of the
method's arithmetic (no softmax, no top-k, no attention, no acceptance), so
both the CUDA path and the CPU oracle can take their inputs from it.  Values
are drawn in numpy from ``np.random.default_rng(seed)`` and rounded to the
workload's dtype here, so the two sides see bit-identical inputs.

Workload shapes follow the target models the paper evaluates (§5.1 "Models":
Llama-3.1-8B, Vicuna-13B, Qwen3-32B, plus a batched 70B-class shape) with the
Eagle3 tree settings of §5.1 "Comparison" (10 nodes per level).  The paper's
datasets (MT-bench, GSM8K, Alpaca, Natural Questions, HumanEval) are replaced
by these synthetic draws: logits N(0, sigma), q/K/V N(0, 1), and a planted
agreement rule that makes the target's argmax equal a draft child with a set
probability.
"""

from __future__ import annotations

from dataclasses import dataclass, field, replace

import numpy as np

F32 = "f32"
BF16 = "bf16"


# ------------------------------------------------------------------ bf16 bits
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (round to nearest, ties to even) and
    return the 16-bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    u = (u + np.uint64(0x7FFF) + lsb) >> np.uint64(16)
    return u.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def round_to(x: np.ndarray, dtype: str) -> np.ndarray:
    """float32 array holding values exactly representable in ``dtype``."""
    x = np.asarray(x, dtype=np.float32)
    if dtype == BF16:
        return bf16_bits_to_f32(f32_to_bf16_bits(x))
    return x


# -------------------------------------------------------------------- configs
@dataclass(frozen=True)
class Config:
    name: str
    batch: int
    layers: int
    hq: int
    hkv: int
    head_dim: int
    vocab: int
    dtype: str
    W: int
    # per-sequence draws (fixed values when lo == hi / single choice)
    ctx_range: tuple            # (lo, hi) inclusive, uniform
    depth_range: tuple          # (lo, hi) inclusive, uniform
    n_choices: tuple            # verify sizes to draw from (uniform)
    mode: str                   # "greedy" | "stochastic" | "mixed"
    sigma_draft: float = 1.0
    sigma_target: float = 1.0
    plant: str = "none"         # "const" | "decay" | "none"
    plant_p: float = 0.0
    plant_decay: float = 1.0
    n_range: tuple = ()         # (lo, hi) inclusive, overrides n_choices when set

    @property
    def max_depth(self) -> int:
        return self.depth_range[1]

    @property
    def max_n(self) -> int:
        return self.n_range[1] if self.n_range else max(self.n_choices)

    @property
    def max_ctx(self) -> int:
        return self.ctx_range[1]

    @property
    def s_cap(self) -> int:
        need = self.max_ctx + self.max_n
        return (need + 127) // 128 * 128

    @property
    def rows_per_seq(self) -> int:
        """Draft row store rows per sequence: 1 + (L_max - 1) W."""
        return 1 + (self.max_depth - 1) * self.W


CONFIGS = {
    "tiny": Config("tiny", batch=1, layers=1, hq=4, hkv=1, head_dim=64, vocab=1000, dtype=F32,
                   W=2, ctx_range=(128, 128), depth_range=(3, 3), n_choices=(8,), mode="greedy",
                   plant="const", plant_p=0.7),
    "8b": Config("8b", batch=1, layers=32, hq=32, hkv=8, head_dim=128, vocab=128256, dtype=BF16,
                 W=10, ctx_range=(4096, 4096), depth_range=(6, 6), n_choices=(60,), mode="greedy",
                 plant="decay", plant_p=0.75, plant_decay=0.9),
    "13b": Config("13b", batch=1, layers=40, hq=40, hkv=40, head_dim=128, vocab=32000, dtype=BF16,
                  W=10, ctx_range=(2048, 2048), depth_range=(3, 8), n_choices=(16, 32, 48, 64, 96),
                  mode="stochastic", sigma_draft=1.5, sigma_target=1.5),
    "32b": Config("32b", batch=1, layers=64, hq=64, hkv=8, head_dim=128, vocab=151936, dtype=BF16,
                  W=8, ctx_range=(16384, 16384), depth_range=(8, 8), n_choices=(48,), mode="greedy",
                  plant="const", plant_p=0.8),
    "70b": Config("70b", batch=16, layers=80, hq=64, hkv=8, head_dim=128, vocab=128256, dtype=BF16,
                  W=10, ctx_range=(1024, 8192), depth_range=(4, 8), n_choices=(), n_range=(32, 96),
                  mode="mixed", plant="decay", plant_p=0.75, plant_decay=0.9),
}


def config(name: str, **overrides) -> Config:
    return replace(CONFIGS[name], **overrides)


# ----------------------------------------------------------- cycle-level draws
@dataclass
class CycleInputs:
    cfg: Config
    seed: int
    root: np.ndarray          # [B] int32
    depth: np.ndarray         # [B] int32 levels below the root (L_b)
    n_verify: np.ndarray      # [B] int32 N_b (root included)
    ctx: np.ndarray           # [B] int32
    mode: np.ndarray          # [B] int32 0 greedy / 1 stochastic
    draft_rows: np.ndarray    # [B][R][vocab] float32, values exact in cfg.dtype
    extra: dict = field(default_factory=dict)


def draw_cycle(cfg: Config, seed: int, draft_rows: bool = True) -> CycleInputs:
    """Per-sequence shape draws and the draft row store of one cycle."""
    rng = np.random.default_rng(seed)
    B = cfg.batch
    root = rng.integers(0, cfg.vocab, size=B).astype(np.int32)
    depth = rng.integers(cfg.depth_range[0], cfg.depth_range[1] + 1, size=B).astype(np.int32)
    if cfg.n_range:
        n = rng.integers(cfg.n_range[0], cfg.n_range[1] + 1, size=B)
    else:
        n = rng.choice(np.array(cfg.n_choices), size=B)
    n = n.astype(np.int32)
    ctx = rng.integers(cfg.ctx_range[0], cfg.ctx_range[1] + 1, size=B).astype(np.int32)
    if cfg.mode == "greedy":
        mode = np.zeros(B, np.int32)
    elif cfg.mode == "stochastic":
        mode = np.ones(B, np.int32)
    else:
        mode = rng.integers(0, 2, size=B).astype(np.int32)
    rows = None
    if draft_rows:
        sig = np.where(mode == 1, cfg.sigma_draft if cfg.mode != "mixed" else 1.5, cfg.sigma_draft)
        rows = np.empty((B, cfg.rows_per_seq, cfg.vocab), np.float32)
        for b in range(B):
            rows[b] = rng.standard_normal((cfg.rows_per_seq, cfg.vocab), dtype=np.float32) * np.float32(sig[b])
        rows = round_to(rows, cfg.dtype)
    return CycleInputs(cfg, seed, root, depth, n, ctx, mode, rows)


def draw_target_rows(cfg: Config, ci: CycleInputs, seed_offset: int = 1_000_003) -> np.ndarray:
    """Unplanted target logits [B][N_max][vocab] (N(0, sigma_target); the mixed
    workload uses sigma 1.5 for stochastic sequences)."""
    rng = np.random.default_rng(ci.seed + seed_offset)
    out = np.empty((cfg.batch, cfg.max_n, cfg.vocab), np.float32)
    for b in range(cfg.batch):
        sig = cfg.sigma_target
        if cfg.mode == "mixed" and ci.mode[b] == 1:
            sig = 1.5
        out[b] = rng.standard_normal((cfg.max_n, cfg.vocab), dtype=np.float32) * np.float32(sig)
    return round_to(out, cfg.dtype)


def plant_probability(cfg: Config, depth: int) -> float:
    if cfg.plant == "const":
        return cfg.plant_p
    if cfg.plant == "decay":
        return cfg.plant_p * cfg.plant_decay ** depth
    return 0.0


def plant_agreement(cfg: Config, target: np.ndarray, chosen, parent, token, depth,
                    rng: np.random.Generator, greedy: bool = True) -> np.ndarray:
    """Make the target agree with the draft (in place, returns ``target``).

    ``chosen`` are the verified node ids in slot order and ``parent``,
    ``token``, ``depth`` the tree's per-node arrays.  For every verified slot
    whose node has verified children, with probability p(depth) the logit of
    the lowest-slot child's token is set to (row max + 1), rounded to the
    workload dtype, so it is the row's strict argmax.  Only greedy sequences
    are planted.
    """
    if not greedy or cfg.plant == "none":
        return target
    chosen = [int(c) for c in chosen]
    first_child = {}
    for s, nid in enumerate(chosen):
        p = int(parent[nid])
        if p >= 0 and p not in first_child:
            first_child[p] = nid
    for s, nid in enumerate(chosen):
        if nid not in first_child:
            continue
        if rng.random() < plant_probability(cfg, int(depth[nid])):
            tok = int(token[first_child[nid]])
            v = np.float32(target[s].max()) + np.float32(1.0)
            target[s, tok] = round_to(np.array([v], np.float32), cfg.dtype)[0]
    return target


# ------------------------------------------------------------ attention draws
def draw_attention(cfg: Config, seed: int, ctx: np.ndarray, n_verify: np.ndarray):
    """q [B][N_max][Hq][d] and one layer's K/V caches [B][Hkv][S_cap][d], N(0, 1)
    rounded to the workload dtype.  Rows past ctx + N are zero."""
    rng = np.random.default_rng(seed + 7_000_001)
    B, d = cfg.batch, cfg.head_dim
    q = round_to(rng.standard_normal((B, cfg.max_n, cfg.hq, d), dtype=np.float32), cfg.dtype)
    k = np.zeros((B, cfg.hkv, cfg.s_cap, d), np.float32)
    v = np.zeros((B, cfg.hkv, cfg.s_cap, d), np.float32)
    for b in range(B):
        rows = int(ctx[b]) + int(n_verify[b])
        k[b, :, :rows] = rng.standard_normal((cfg.hkv, rows, d), dtype=np.float32)
        v[b, :, :rows] = rng.standard_normal((cfg.hkv, rows, d), dtype=np.float32)
    return q, round_to(k, cfg.dtype), round_to(v, cfg.dtype)

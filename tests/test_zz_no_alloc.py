"""ltd_accept_noalloc against ltd_accept.

The allocation-free acceptance entry point is for callers that cannot
allocate device memory when they accept a draft (memory reserved up front,
a host framework that owns every buffer, a stream that must stay
allocation-free for graph capture).  It keeps its scratch in a static device
array instead of a caller workspace.  These tests call both entry points
through the C ABI on the same inputs and require identical results (the
integer outputs of acceptance are compared bit for bit, as everywhere in
this suite), on two calls in a row so that the array's leftover contents
from the first call cannot leak into the second.  This file sorts last so a
run that stops at the first failure has already run every other test; it
also passes on its own in a fresh process.
"""

import numpy as np
import pytest
import torch

from paper_2603_01639_gb300 import ltd
from paper_2603_01639_gb300 import workload as wl

from . import harness as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2603_01639_gb300 import build
    build.build()
    ltd.lib()


def _outputs(B, depth):
    return {"path": torch.full((B, depth + 1), -7, dtype=torch.int32, device="cuda"),
            "accept_len": torch.full((B,), -7, dtype=torch.int32, device="cuda"),
            "bonus": torch.full((B,), -7, dtype=torch.int32, device="cuda"),
            "new_ctx": torch.full((B,), -7, dtype=torch.int32, device="cuda")}


@pytest.mark.parametrize("name,seed", [("tiny", 0), ("8b", 0), ("13b", 3), ("70b", 0)])
def test_noalloc_matches_workspace_entry_point(name, seed):
    cfg = wl.config(name)
    ci = wl.draw_cycle(cfg, seed)
    trees, sels, target = H.oracle_side(cfg, ci)
    draft = H.dev(ci.draft_rows, cfg.dtype)
    tree = H.gpu_draft(cfg, ci, draft)
    ids, _, _ = H.gpu_select(cfg, ci, tree)
    tgt = H.dev(target, cfg.dtype)
    args = (tree, tgt, draft, ids, H.i32(ci.n_verify), H.i32(ci.mode), H.i32(ci.ctx))
    ref = ltd.ltd_accept(*args, seed=77, cycle=seed, out=_outputs(cfg.batch, cfg.max_depth))
    assert ltd.ltd_check() == 0
    for call in range(2):
        got = ltd.ltd_accept_noalloc(*args, seed=77, cycle=seed,
                                     out=_outputs(cfg.batch, cfg.max_depth))
        assert ltd.ltd_check() == 0
        for k in ref:
            assert torch.equal(got[k], ref[k]), (call, k, got[k], ref[k])


def test_noalloc_compacts_like_workspace_entry_point():
    cfg = wl.config("8b", layers=2)
    ci = wl.draw_cycle(cfg, 1)
    trees, sels, target = H.oracle_side(cfg, ci)
    draft = H.dev(ci.draft_rows, cfg.dtype)
    tree = H.gpu_draft(cfg, ci, draft)
    ids, _, _ = H.gpu_select(cfg, ci, tree)
    tgt = H.dev(target, cfg.dtype)
    g = torch.Generator(device="cuda").manual_seed(5)
    base_k = [torch.randn(1, cfg.hkv, cfg.s_cap, 128, generator=g, device="cuda").to(torch.bfloat16)
              for _ in range(2)]
    base_v = [torch.randn(1, cfg.hkv, cfg.s_cap, 128, generator=g, device="cuda").to(torch.bfloat16)
              for _ in range(2)]
    results = []
    for fn in ("ltd_accept", "ltd_accept_noalloc", "ltd_accept_noalloc"):
        ks = [t.clone() for t in base_k]
        vs = [t.clone() for t in base_v]
        kv = ltd.KVCache(ks, vs)
        out = getattr(ltd, fn)(tree, tgt, draft, ids, H.i32(ci.n_verify), H.i32(ci.mode),
                               H.i32(ci.ctx), kv=kv, out=_outputs(1, cfg.max_depth))
        assert ltd.ltd_check() == 0
        results.append((out, ks, vs))
    ref = results[0]
    for out, ks, vs in results[1:]:
        for k in ref[0]:
            assert torch.equal(out[k], ref[0][k])
        for a, b in zip(ks + vs, ref[1] + ref[2]):
            assert torch.equal(a, b)


def test_noalloc_rejects_sizes_beyond_its_array():
    """Sizes whose acceptance scratch exceeds the static array (here 512
    sequences x 256 verify slots, one record each) are refused with
    LTD_ERR_SHAPE before anything is launched."""
    import ctypes as C
    B, n_max, vocab = 512, 256, 1000
    tree = ltd.Tree(B, 3, 2, vocab)
    L = ltd.lib()
    assert L.ltd_accept_workspace_bytes(B, n_max, vocab) > ltd.LTD_ACCEPT_NOALLOC_SCRATCH_BYTES
    buf = torch.zeros(64, dtype=torch.int32, device="cuda")
    p = C.c_void_p(buf.data_ptr())
    st = L.ltd_accept_noalloc(C.byref(tree.s), p, p, 0, vocab, 5, p, p, n_max, p, 0, 0, p, p, p, p,
                              p, None, C.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert L.ltd_status_string(st).decode() == "LTD_ERR_SHAPE"


def test_noalloc_rejects_a_missing_or_malformed_tree_like_its_sibling():
    """A NULL tree, a tree whose arrays were never carved, or a NULL output
    buffer is LTD_ERR_INVALID_ARG, as in ltd_accept, before any size (here an
    oversized batch) is looked at; nothing is launched."""
    import ctypes as C
    L = ltd.lib()
    buf = torch.zeros(64, dtype=torch.int32, device="cuda")
    p = C.c_void_p(buf.data_ptr())
    s = C.c_void_p(torch.cuda.current_stream().cuda_stream)
    raw = ltd.ltd_tree()
    raw.batch, raw.max_depth, raw.k, raw.max_vocab = 4096, 3, 2, 1000   # sizes only, no arrays
    good = ltd.Tree(1, 3, 2, 1000)
    cases = [(None, p), (C.byref(raw), p), (C.byref(good.s), None)]
    for tree, bonus in cases:
        st = L.ltd_accept_noalloc(tree, p, p, 0, 1000, 5, p, p, 8, p, 0, 0, p, p, p, p, bonus,
                                  None, s)
        assert L.ltd_status_string(st).decode() == "LTD_ERR_INVALID_ARG"
        st = L.ltd_accept(tree, p, p, 0, 1000, 5, p, p, 8, p, 0, 0, p, p, p, p, bonus, None, p,
                          1 << 20, s)
        assert L.ltd_status_string(st).decode() == "LTD_ERR_INVALID_ARG"

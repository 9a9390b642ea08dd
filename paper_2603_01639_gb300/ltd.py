"""Thin ctypes binding of ``libltd.so`` (the C ABI in ``include/ltd.h``).

Functions carry the C names and only marshal arguments: torch tensors become
device pointers, the current torch stream becomes the ``cudaStream_t``, and
output tensors are allocated with torch.  Every step of the cycle runs in the
library's CUDA kernels; there is no fallback of any kind -- if the library is
missing or no GPU is present, calls raise.
"""

from __future__ import annotations

import ctypes as C
import os
import threading

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libltd.so")
_lib = None
_lock = threading.Lock()

LTD_F32, LTD_BF16 = 0, 1
LTD_GREEDY, LTD_STOCHASTIC, LTD_STOCHASTIC_POINT_MASS, LTD_STOCHASTIC_NO_REPLACEMENT = 0, 1, 2, 3
LTD_MAX_K, LTD_MAX_DEPTH, LTD_MAX_N, LTD_MAX_TREE_NODES = 32, 16, 256, 4096
DEVERR = {0x1: "LEVEL", 0x2: "NVERIFY", 0x4: "CTX", 0x8: "TREE", 0x10: "TIMEOUT", 0x20: "MODE"}

# Every symbol declared in include/ltd.h.
EXPORTS = [
    "ltd_tree_bytes", "ltd_tree_init", "ltd_tree_reset", "ltd_expand_tree", "ltd_select_verify",
    "ltd_attention_workspace_bytes", "ltd_tree_attention", "ltd_accept_workspace_bytes",
    "ltd_accept", "ltd_kv_compact", "ltd_check", "ltd_status_string", "ltd_version",
    "ltd_attention_kernel", "ltd_selftest_umma", "ltd_accept_noalloc", "ltd_tree_attention_next",
    "ltd_depth_observation", "ltd_size_observation", "ltd_depth_policy", "ltd_size_policy",
    "ltd_mlp_packed_bytes", "ltd_mlp_pack", "ltd_kv_append", "ltd_accept_tempered",
    "ltd_debug_attention_wait", "ltd_debug_expand_wait", "ltd_lm_head_workspace_bytes", "ltd_lm_head_row_stats",
]
LTD_POLICY_PAD = -100.0
LTD_MLP_MAX_LAYERS, LTD_MLP_MAX_WIDTH = 4, 2048
LTD_MLP_ROW_MAJOR, LTD_MLP_PACKED = 0, 1
LTD_ACCEPT_NOALLOC_SCRATCH_BYTES = 1 << 20


class LtdError(RuntimeError):
    pass


class ltd_tree(C.Structure):
    _fields_ = [("batch", C.c_int32), ("max_depth", C.c_int32), ("k", C.c_int32),
                ("max_nodes", C.c_int32), ("max_vocab", C.c_int64),
                ("token", C.c_void_p), ("parent", C.c_void_p), ("depth", C.c_void_p),
                ("cum_logprob", C.c_void_p), ("xrow", C.c_void_p), ("xlse", C.c_void_p),
                ("frontier", C.c_void_p), ("n_nodes", C.c_void_p), ("n_levels", C.c_void_p),
                ("scratch", C.c_void_p), ("scratch_bytes", C.c_size_t)]


class ltd_kv_cache(C.Structure):
    _fields_ = [("d_k_layers", C.c_void_p), ("d_v_layers", C.c_void_p),
                ("n_layers", C.c_int32), ("hkv", C.c_int32), ("head_dim", C.c_int32),
                ("s_cap", C.c_int32), ("dtype", C.c_int32)]


class ltd_mlp(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("layout", C.c_int32),
                ("dims", C.c_int32 * (LTD_MLP_MAX_LAYERS + 1)),
                ("w", C.c_void_p * LTD_MLP_MAX_LAYERS), ("b", C.c_void_p * LTD_MLP_MAX_LAYERS)]


def lib():
    """Load libltd.so once; raise if it is not built."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(_LIB_PATH):
                raise LtdError(f"{_LIB_PATH} is missing: build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
            L = C.CDLL(_LIB_PATH)
            vp, i32, i64, u64, sz = C.c_void_p, C.c_int32, C.c_int64, C.c_uint64, C.c_size_t
            tp = C.POINTER(ltd_tree)
            sig = {
                "ltd_tree_bytes": (sz, [i32, i32, i32, i64]),
                "ltd_tree_init": (C.c_int, [tp, vp, sz, i32, i32, i32, i64]),
                "ltd_tree_reset": (C.c_int, [tp, vp, vp]),
                "ltd_expand_tree": (C.c_int, [tp, i32, vp, C.c_int, i64, i64, vp, vp]),
                "ltd_select_verify": (C.c_int, [tp, vp, i32, vp, vp, vp, vp, vp]),
                "ltd_depth_observation": (C.c_int, [tp, vp, vp, vp]),
                "ltd_size_observation": (C.c_int, [tp, vp, i32, vp, vp]),
                "ltd_mlp_packed_bytes": (sz, [C.POINTER(ltd_mlp)]),
                "ltd_mlp_pack": (C.c_int, [C.POINTER(ltd_mlp), vp, sz, C.POINTER(ltd_mlp), vp]),
                "ltd_depth_policy": (C.c_int, [tp, vp, C.POINTER(ltd_mlp), vp, vp, vp, vp]),
                "ltd_size_policy": (C.c_int, [tp, vp, i32, C.POINTER(ltd_mlp), i32, vp, vp, vp]),
                "ltd_attention_workspace_bytes": (sz, [i32, i32, i32, i32, i32, i32, C.c_int]),
                "ltd_tree_attention": (C.c_int, [vp, vp, vp, vp, C.c_int, i32, i32, i32, i32, i32,
                                                 vp, i32, vp, i32, vp, C.c_float, vp, sz, vp]),
                "ltd_tree_attention_next": (C.c_int, [vp, vp, vp, vp, C.c_int, i32, i32, i32, i32,
                                                      i32, vp, i32, vp, i32, vp, C.c_float, vp, sz,
                                                      vp, vp, vp]),
                "ltd_accept_workspace_bytes": (sz, [i32, i32, i64]),
                "ltd_accept": (C.c_int, [tp, vp, vp, C.c_int, i64, i64, vp, vp, i32, vp, u64, u64,
                                         vp, vp, vp, vp, vp, C.POINTER(ltd_kv_cache), vp, sz, vp]),
                "ltd_accept_tempered": (C.c_int, [tp, vp, vp, C.c_int, i64, i64, vp, vp, i32, vp,
                                                  C.c_float, u64, u64, vp, vp, vp, vp, vp,
                                                  C.POINTER(ltd_kv_cache), vp, sz, vp]),
                "ltd_kv_compact": (C.c_int, [C.POINTER(ltd_kv_cache), i32, vp, i32, vp, vp, vp]),
                "ltd_kv_append": (C.c_int, [C.POINTER(ltd_kv_cache), i32, i32, vp, vp, vp, vp, vp]),
                "ltd_check": (C.c_int, [vp, C.POINTER(C.c_uint32)]),
                "ltd_status_string": (C.c_char_p, [C.c_int]),
                "ltd_version": (i32, []),
                "ltd_attention_kernel": (i32, [C.c_int, i32, i32, i32, i32, i32, i32,
                                               C.POINTER(i32)]),
                "ltd_selftest_umma": (C.c_int, [i32, vp, vp, vp, vp]),
                "ltd_debug_attention_wait": (C.c_int, [u64, C.c_uint32]),
                "ltd_debug_expand_wait": (C.c_int, [u64, C.c_uint32]),
                "ltd_lm_head_workspace_bytes": (sz, [i32, i64, i32]),
                "ltd_lm_head_row_stats": (C.c_int, [vp, vp, i32, i64, i32, vp, vp, vp, vp, vp, sz,
                                                    vp]),
                "ltd_accept_noalloc": (C.c_int, [tp, vp, vp, C.c_int, i64, i64, vp, vp, i32, vp, u64,
                                                 u64, vp, vp, vp, vp, vp, C.POINTER(ltd_kv_cache),
                                                 vp]),
            }
            for name, (res, args) in sig.items():
                fn = getattr(L, name)
                fn.restype = res
                fn.argtypes = args
            _lib = L
    return _lib


def _ok(status: int, what: str):
    if status != 0:
        raise LtdError(f"{what}: {lib().ltd_status_string(status).decode()}")


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return C.c_void_p(s.cuda_stream)


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _dtype(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return LTD_BF16
    if t.dtype == torch.float32:
        return LTD_F32
    raise LtdError(f"unsupported dtype {t.dtype}")


def _need_vec(t: torch.Tensor, name: str, numel: int, dtype):
    """A contiguous CUDA tensor of ``dtype`` holding exactly ``numel`` values."""
    _need(t, name, dtype)
    if t.numel() != numel:
        raise LtdError(f"{name} must hold {numel} values, got {t.numel()}")


def _need(t: torch.Tensor, name: str, dtype=None):
    if not t.is_cuda:
        raise LtdError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise LtdError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise LtdError(f"{name} must be {dtype}, got {t.dtype}")


# ------------------------------------------------------------------ tree
class Tree:
    """A batch of draft trees in one torch-owned device buffer."""

    def __init__(self, batch: int, max_depth: int, k: int, max_vocab: int, device="cuda"):
        L = lib()
        n = L.ltd_tree_bytes(batch, max_depth, k, max_vocab)
        if n == 0:
            raise LtdError("ltd_tree_bytes: bad tree dimensions")
        self.buf = torch.empty(n + 256, dtype=torch.uint8, device=device)
        off = (-self.buf.data_ptr()) % 256
        self.mem = self.buf[off:off + n]
        self.s = ltd_tree()
        _ok(L.ltd_tree_init(C.byref(self.s), C.c_void_p(self.mem.data_ptr()), n, batch, max_depth,
                            k, max_vocab), "ltd_tree_init")

    @property
    def batch(self):
        return self.s.batch

    @property
    def k(self):
        return self.s.k

    @property
    def max_depth(self):
        return self.s.max_depth

    @property
    def max_nodes(self):
        return self.s.max_nodes

    def _view(self, ptr, count, dtype):
        off = ptr - self.mem.data_ptr()
        nbytes = count * 4
        return self.mem[off:off + nbytes].view(dtype)

    def view(self) -> dict:
        """Device views of the tree arrays ([batch][max_nodes] etc.)."""
        B, mn, k = self.batch, self.max_nodes, self.k
        s = self.s
        i32, f32 = torch.int32, torch.float32
        return {
            "token": self._view(s.token, B * mn, i32).view(B, mn),
            "parent": self._view(s.parent, B * mn, i32).view(B, mn),
            "depth": self._view(s.depth, B * mn, i32).view(B, mn),
            "cum_logprob": self._view(s.cum_logprob, B * mn, f32).view(B, mn),
            "xrow": self._view(s.xrow, B * mn, i32).view(B, mn),
            "xlse": self._view(s.xlse, B * mn, f32).view(B, mn),
            "frontier": self._view(s.frontier, B * k, i32).view(B, k),
            "n_nodes": self._view(s.n_nodes, B, i32),
            "n_levels": self._view(s.n_levels, B, i32),
        }


def ltd_tree_reset(tree: Tree, root_tokens: torch.Tensor, stream=None):
    _need(root_tokens, "root_tokens", torch.int32)
    _ok(lib().ltd_tree_reset(C.byref(tree.s), _ptr(root_tokens), _stream(stream)), "ltd_tree_reset")


def ltd_expand_tree(tree: Tree, level: int, draft_rows: torch.Tensor, active=None, stream=None):
    """draft_rows: [batch][rows_per_seq][vocab] bf16/f32."""
    _need(draft_rows, "draft_rows")
    if active is not None:
        _need(active, "active", torch.int32)
    B, R, V = draft_rows.shape
    _ok(lib().ltd_expand_tree(C.byref(tree.s), level, _ptr(draft_rows), _dtype(draft_rows), V, R,
                              _ptr(active), _stream(stream)), "ltd_expand_tree")


def ltd_select_verify(tree: Tree, n_verify: torch.Tensor, n_max: int, ctx: torch.Tensor,
                      out=None, stream=None):
    """Returns (node_ids [B][n_max], pos [B][n_max], mask [B][n_max][ceil(n_max/32)])."""
    _need(n_verify, "n_verify", torch.int32)
    _need(ctx, "ctx", torch.int32)
    B = tree.batch
    w32 = (n_max + 31) // 32
    dev = n_verify.device
    if out is None:
        out = (torch.empty(B, n_max, dtype=torch.int32, device=dev),
               torch.empty(B, n_max, dtype=torch.int32, device=dev),
               torch.empty(B, n_max, w32, dtype=torch.int32, device=dev))
    ids, pos, mask = out
    _ok(lib().ltd_select_verify(C.byref(tree.s), _ptr(n_verify), n_max, _ptr(ctx), _ptr(ids),
                                _ptr(pos), _ptr(mask), _stream(stream)), "ltd_select_verify")
    return ids, pos, mask


def ltd_depth_observation(tree: Tree, ctx: torch.Tensor, out=None, stream=None):
    """Depth-policy observation [B][k*k + 2] (float32): the last level's
    candidate cum log-probs (padded with LTD_POLICY_PAD), then D and L."""
    _need(ctx, "ctx", torch.int32)
    kk = tree.k * tree.k
    if out is None:
        out = torch.empty(tree.batch, kk + 2, dtype=torch.float32, device=ctx.device)
    _ok(lib().ltd_depth_observation(C.byref(tree.s), _ptr(ctx), _ptr(out), _stream(stream)),
        "ltd_depth_observation")
    return out


def ltd_size_observation(tree: Tree, ctx: torch.Tensor, v_pad=None, out=None, stream=None):
    """Size-policy observation [B][v_pad + 2] (float32): every node's cum
    log-prob in id order (padded with LTD_POLICY_PAD), then D and L;
    v_pad defaults to the tree's max_nodes."""
    _need(ctx, "ctx", torch.int32)
    v_pad = tree.max_nodes if v_pad is None else v_pad
    if out is None:
        out = torch.empty(tree.batch, v_pad + 2, dtype=torch.float32, device=ctx.device)
    _ok(lib().ltd_size_observation(C.byref(tree.s), _ptr(ctx), v_pad, _ptr(out), _stream(stream)),
        "ltd_size_observation")
    return out


class MlpNet:
    """A policy MLP's weights on the device ([n_in][n_out] fp32 matrices and
    biases) and the ltd_mlp struct that points at them; with ``packed`` the
    struct points at the library's packed copy (ltd_mlp_pack), which the
    device policies stream with bulk copies."""

    def __init__(self, layers, device="cuda", packed=True, stream=None):
        if not 1 <= len(layers) <= LTD_MLP_MAX_LAYERS:
            raise LtdError(f"an MLP has 1..{LTD_MLP_MAX_LAYERS} layers")
        self.w = [torch.as_tensor(w, dtype=torch.float32).to(device).contiguous() for w, _ in layers]
        self.b = [torch.as_tensor(b, dtype=torch.float32).to(device).contiguous() for _, b in layers]
        self.s = ltd_mlp()
        self.s.n_layers = len(layers)
        self.s.dims[0] = self.w[0].shape[0]
        for i, (w, b) in enumerate(zip(self.w, self.b)):
            if w.dim() != 2 or b.shape != (w.shape[1],) or (i and w.shape[0] != self.w[i - 1].shape[1]):
                raise LtdError("MLP layer shapes do not chain")
            self.s.dims[i + 1] = w.shape[1]
            self.s.w[i] = w.data_ptr()
            self.s.b[i] = b.data_ptr()
        self.row_major = self.s
        if packed:
            n = lib().ltd_mlp_packed_bytes(C.byref(self.s))
            if n == 0:
                raise LtdError("ltd_mlp_packed_bytes: the policies would reject this network")
            self.pbuf = torch.empty(n + 256, dtype=torch.uint8, device=device)
            off = (-self.pbuf.data_ptr()) % 256
            p = ltd_mlp()
            _ok(lib().ltd_mlp_pack(C.byref(self.s), C.c_void_p(self.pbuf.data_ptr() + off), n,
                                   C.byref(p), _stream(stream)), "ltd_mlp_pack")
            self.s = p

    @property
    def n_in(self):
        return self.s.dims[0]

    @property
    def n_out(self):
        return self.s.dims[self.s.n_layers]


def ltd_depth_policy(tree: Tree, ctx: torch.Tensor, net: MlpNet, active_in=None, active_out=None,
                     logits=None, stream=None):
    """Depth policy on the device after the last built level: returns the
    next level's active mask [B] int32 (1 = keep drafting)."""
    _need(ctx, "ctx", torch.int32)
    if active_out is None:
        active_out = torch.empty(tree.batch, dtype=torch.int32, device=ctx.device)
    _need_vec(active_out, "active_out", tree.batch, torch.int32)
    if active_in is not None:
        _need_vec(active_in, "active_in", tree.batch, torch.int32)
    if logits is not None:
        _need_vec(logits, "logits", tree.batch * 2, torch.float32)
    _ok(lib().ltd_depth_policy(C.byref(tree.s), _ptr(ctx), C.byref(net.s), _ptr(active_in),
                               _ptr(active_out), _ptr(logits), _stream(stream)),
        "ltd_depth_policy")
    return active_out


def ltd_size_policy(tree: Tree, ctx: torch.Tensor, net: MlpNet, n_cap: int, v_pad=None,
                    n_verify=None, logits=None, stream=None):
    """Size policy on the device after the draft: returns N per sequence
    ([B] int32, root included, at most n_cap and the tree's node count)."""
    _need(ctx, "ctx", torch.int32)
    v_pad = tree.max_nodes if v_pad is None else v_pad
    if n_verify is None:
        n_verify = torch.empty(tree.batch, dtype=torch.int32, device=ctx.device)
    _need_vec(n_verify, "n_verify", tree.batch, torch.int32)
    if logits is not None:
        _need_vec(logits, "logits", tree.batch * net.n_out, torch.float32)
    _ok(lib().ltd_size_policy(C.byref(tree.s), _ptr(ctx), v_pad, C.byref(net.s), n_cap,
                              _ptr(n_verify), _ptr(logits), _stream(stream)),
        "ltd_size_policy")
    return n_verify


def attention_workspace(batch, hq, hkv, head_dim, n_max, max_ctx, dtype, device="cuda"):
    n = lib().ltd_attention_workspace_bytes(batch, hq, hkv, head_dim, n_max, max_ctx,
                                            LTD_BF16 if dtype == torch.bfloat16 else LTD_F32)
    if n == 0:
        raise LtdError("ltd_attention_workspace_bytes: bad sizes")
    return torch.zeros(n, dtype=torch.uint8, device=device)


def ltd_tree_attention(q, k_cache, v_cache, ctx, max_ctx, n_verify, mask, scale=None,
                       out=None, workspace=None, stream=None, next_k=None, next_v=None):
    """q [B][n_max][hq][d]; k/v [B][hkv][s_cap][d]; returns out like q.  next_k/next_v:
    the next call's caches (same shapes), for ltd_tree_attention_next's L2 hint."""
    for t, n in ((q, "q"), (k_cache, "k_cache"), (v_cache, "v_cache")):
        _need(t, n, q.dtype)
    _need(ctx, "ctx", torch.int32)
    _need(n_verify, "n_verify", torch.int32)
    _need(mask, "mask")
    B, n_max, hq, d = q.shape
    hkv, s_cap = k_cache.shape[1], k_cache.shape[2]
    if scale is None:
        scale = d ** -0.5
    if out is None:
        out = torch.zeros_like(q)
    if workspace is None:
        workspace = attention_workspace(B, hq, hkv, d, n_max, max_ctx, q.dtype, q.device)
    if next_k is None and next_v is None:
        _ok(lib().ltd_tree_attention(_ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(out), _dtype(q),
                                     B, hq, hkv, d, s_cap, _ptr(ctx), max_ctx, _ptr(n_verify),
                                     n_max, _ptr(mask), float(scale), _ptr(workspace),
                                     workspace.numel(), _stream(stream)), "ltd_tree_attention")
        return out
    if (next_k is None) != (next_v is None):
        raise LtdError("next_k and next_v go together")
    for t, n in ((next_k, "next_k"), (next_v, "next_v")):
        _need(t, n, q.dtype)
        if t.shape != k_cache.shape:
            raise LtdError(f"{n} must have the shape of k_cache")
    _ok(lib().ltd_tree_attention_next(_ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(out), _dtype(q),
                                      B, hq, hkv, d, s_cap, _ptr(ctx), max_ctx, _ptr(n_verify),
                                      n_max, _ptr(mask), float(scale), _ptr(workspace),
                                      workspace.numel(), _ptr(next_k), _ptr(next_v),
                                      _stream(stream)), "ltd_tree_attention_next")
    return out


def accept_workspace(batch, n_max, vocab, device="cuda"):
    n = lib().ltd_accept_workspace_bytes(batch, n_max, vocab)
    if n == 0:
        raise LtdError("ltd_accept_workspace_bytes: bad sizes")
    return torch.zeros(n, dtype=torch.uint8, device=device)


class KVCache:
    """Per-layer K/V tensors [B][hkv][s_cap][d] plus the device pointer arrays
    ltd_kv_compact reads."""

    def __init__(self, k_layers, v_layers):
        self.k_layers, self.v_layers = list(k_layers), list(v_layers)
        dev = self.k_layers[0].device
        self.k_ptrs = torch.tensor([t.data_ptr() for t in self.k_layers], dtype=torch.int64, device=dev)
        self.v_ptrs = torch.tensor([t.data_ptr() for t in self.v_layers], dtype=torch.int64, device=dev)
        k0 = self.k_layers[0]
        self.s = ltd_kv_cache(C.c_void_p(self.k_ptrs.data_ptr()), C.c_void_p(self.v_ptrs.data_ptr()),
                              len(self.k_layers), k0.shape[1], k0.shape[3], k0.shape[2], _dtype(k0))


def ltd_accept(tree: Tree, target, draft_rows, node_ids, n_verify, mode, ctx, seed=0, cycle=0,
               kv: KVCache | None = None, workspace=None, out=None, stream=None, temperature=None):
    """Returns dict(path [B][max_depth+1], accept_len [B], bonus [B], new_ctx [B]).
    ``temperature`` (a float) calls ltd_accept_tempered instead."""
    _need(target, "target")
    _need(draft_rows, "draft_rows", target.dtype)
    for t, n in ((node_ids, "node_ids"), (n_verify, "n_verify"), (mode, "mode"), (ctx, "ctx")):
        _need(t, n, torch.int32)
    B, n_max, V = target.shape
    R = draft_rows.shape[1]
    dev = target.device
    if workspace is None:
        workspace = accept_workspace(B, n_max, V, dev)
    if out is None:
        out = {"path": torch.empty(B, tree.max_depth + 1, dtype=torch.int32, device=dev),
               "accept_len": torch.empty(B, dtype=torch.int32, device=dev),
               "bonus": torch.empty(B, dtype=torch.int32, device=dev),
               "new_ctx": torch.empty(B, dtype=torch.int32, device=dev)}
    kvp = C.byref(kv.s) if kv is not None else None
    if temperature is not None:
        _ok(lib().ltd_accept_tempered(C.byref(tree.s), _ptr(target), _ptr(draft_rows),
                                      _dtype(target), V, R, _ptr(node_ids), _ptr(n_verify), n_max,
                                      _ptr(mode), float(temperature), seed, cycle, _ptr(ctx),
                                      _ptr(out["new_ctx"]), _ptr(out["path"]),
                                      _ptr(out["accept_len"]), _ptr(out["bonus"]), kvp,
                                      _ptr(workspace), workspace.numel(), _stream(stream)),
            "ltd_accept_tempered")
        return out
    _ok(lib().ltd_accept(C.byref(tree.s), _ptr(target), _ptr(draft_rows), _dtype(target), V, R,
                         _ptr(node_ids), _ptr(n_verify), n_max, _ptr(mode), seed, cycle, _ptr(ctx),
                         _ptr(out["new_ctx"]), _ptr(out["path"]), _ptr(out["accept_len"]),
                         _ptr(out["bonus"]), kvp, _ptr(workspace), workspace.numel(),
                         _stream(stream)), "ltd_accept")
    return out


def ltd_accept_noalloc(tree: Tree, target, draft_rows, node_ids, n_verify, mode, ctx, seed=0,
                       cycle=0, kv: KVCache | None = None, out=None, stream=None):
    """ltd_accept without a workspace, for callers that cannot allocate device
    memory when they accept (the library keeps the scratch in a static 1 MiB
    device array).  Output tensors are still the caller's: pass ``out`` (a
    dict like ltd_accept returns) to keep this call allocation-free."""
    _need(target, "target")
    _need(draft_rows, "draft_rows", target.dtype)
    for t, n in ((node_ids, "node_ids"), (n_verify, "n_verify"), (mode, "mode"), (ctx, "ctx")):
        _need(t, n, torch.int32)
    B, n_max, V = target.shape
    R = draft_rows.shape[1]
    dev = target.device
    if out is None:
        out = {"path": torch.empty(B, tree.max_depth + 1, dtype=torch.int32, device=dev),
               "accept_len": torch.empty(B, dtype=torch.int32, device=dev),
               "bonus": torch.empty(B, dtype=torch.int32, device=dev),
               "new_ctx": torch.empty(B, dtype=torch.int32, device=dev)}
    kvp = C.byref(kv.s) if kv is not None else None
    _ok(lib().ltd_accept_noalloc(C.byref(tree.s), _ptr(target), _ptr(draft_rows), _dtype(target),
                                 V, R, _ptr(node_ids), _ptr(n_verify), n_max, _ptr(mode), seed,
                                 cycle, _ptr(ctx), _ptr(out["new_ctx"]), _ptr(out["path"]),
                                 _ptr(out["accept_len"]), _ptr(out["bonus"]), kvp,
                                 _stream(stream)), "ltd_accept_noalloc")
    return out


def ltd_kv_compact(kv: KVCache, path, accept_len, ctx, stream=None):
    _need(path, "path", torch.int32)
    _ok(lib().ltd_kv_compact(C.byref(kv.s), path.shape[0], _ptr(path), path.shape[1],
                             _ptr(accept_len), _ptr(ctx), _stream(stream)), "ltd_kv_compact")


def ltd_kv_append(kv: KVCache, new_k, new_v, ctx, n_verify, stream=None):
    """new_k, new_v: [n_layers][batch][hkv][n_max][head_dim] in the cache's
    dtype; rows ctx_b .. ctx_b + N_b - 1 of every layer's cache receive them."""
    for t, n in ((new_k, "new_k"), (new_v, "new_v")):
        _need(t, n, kv.k_layers[0].dtype)
        if t.dim() != 5 or t.shape[0] != len(kv.k_layers):
            raise LtdError(f"{n} must be [n_layers][batch][hkv][n_max][head_dim]")
    if new_k.shape != new_v.shape:
        raise LtdError("new_k and new_v differ in shape")
    _need(ctx, "ctx", torch.int32)
    _need(n_verify, "n_verify", torch.int32)
    _ok(lib().ltd_kv_append(C.byref(kv.s), new_k.shape[1], new_k.shape[3], _ptr(new_k), _ptr(new_v),
                            _ptr(ctx), _ptr(n_verify), _stream(stream)), "ltd_kv_append")


def ltd_lm_head_row_stats(hidden, weight, logits=False, workspace=None, stream=None):
    """hidden [rows][H] bf16, weight [vocab][H] bf16.  Returns dict(row_max,
    row_lse [rows] fp32, row_argmax [rows] int32, logits [rows][vocab] bf16
    when ``logits`` is true)."""
    _need(hidden, "hidden", torch.bfloat16)
    _need(weight, "weight", torch.bfloat16)
    rows, H = hidden.shape
    vocab = weight.shape[0]
    if weight.shape[1] != H:
        raise LtdError("hidden and weight disagree on the hidden size")
    dev = hidden.device
    if workspace is None:
        n = lib().ltd_lm_head_workspace_bytes(rows, vocab, H)
        if n == 0:
            raise LtdError("ltd_lm_head_workspace_bytes: bad sizes")
        workspace = torch.empty(n, dtype=torch.uint8, device=dev)
    out = {"row_max": torch.empty(rows, dtype=torch.float32, device=dev),
           "row_lse": torch.empty(rows, dtype=torch.float32, device=dev),
           "row_argmax": torch.empty(rows, dtype=torch.int32, device=dev)}
    lg = torch.empty(rows, vocab, dtype=torch.bfloat16, device=dev) if logits else None
    _ok(lib().ltd_lm_head_row_stats(_ptr(hidden), _ptr(weight), rows, vocab, H,
                                    _ptr(lg) if lg is not None else None, _ptr(out["row_max"]),
                                    _ptr(out["row_lse"]), _ptr(out["row_argmax"]), _ptr(workspace),
                                    workspace.numel(), _stream(stream)), "ltd_lm_head_row_stats")
    if lg is not None:
        out["logits"] = lg
    return out


def ltd_check(stream=None, raise_on_error=True) -> int:
    """Synchronise, read and clear the device error word; returns its bits."""
    bits = C.c_uint32(0)
    st = lib().ltd_check(_stream(stream), C.byref(bits))
    if raise_on_error and st != 0:
        names = [v for k, v in DEVERR.items() if bits.value & k]
        raise LtdError(f"ltd_check: {lib().ltd_status_string(st).decode()} {names}")
    return bits.value


def ltd_version() -> int:
    return lib().ltd_version()


def ltd_attention_kernel(dtype, batch, hq, hkv, head_dim, n_max, max_ctx) -> tuple:
    """(1 tensor cores / 0 CUDA cores / -1 unsupported, launches per call)."""
    n = C.c_int32(0)
    code = lib().ltd_attention_kernel(LTD_BF16 if dtype == torch.bfloat16 else LTD_F32, batch, hq,
                                      hkv, head_dim, n_max, max_ctx, C.byref(n))
    return code, n.value


def attention_kernel_sources(code: int) -> list:
    """Source files of the attention kernel selected by ltd_attention_kernel."""
    if code == 1:
        return ["k_attn_tc.cu", "tc_util.cuh", "ltd_common.cuh"]
    return ["k_attn_simt.cu", "ltd_common.cuh"]


def ltd_selftest_umma(mode: int, a: torch.Tensor, b: torch.Tensor, stream=None) -> torch.Tensor:
    """128x128x128 bf16 GEMM through TMA + tcgen05 (mode 0: a @ b.T, mode 1: a @ b)."""
    _need(a, "a", torch.bfloat16)
    _need(b, "b", torch.bfloat16)
    c = torch.empty(128, 128, dtype=torch.float32, device=a.device)
    _ok(lib().ltd_selftest_umma(mode, _ptr(a), _ptr(b), _ptr(c), _stream(stream)),
        "ltd_selftest_umma")
    return c

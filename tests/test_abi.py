"""libltd.so loads, exports every function include/ltd.h declares, and rejects
bad arguments on the host before touching a GPU (no compute calls here)."""

import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    from paper_2603_01639_gb300 import build, ltd
    build.build()
    return ltd.lib()


def _declared():
    with open(os.path.join(ROOT, "include", "ltd.h")) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ltd_[a-z0-9_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(L):
    from paper_2603_01639_gb300 import ltd
    declared = _declared()
    assert declared, "no declarations parsed"
    for name in declared:
        assert hasattr(L, name), f"{name} declared in ltd.h but not exported"
    assert sorted(ltd.EXPORTS) == declared


def test_version_and_status_strings(L):
    assert L.ltd_version() == 100
    for s, name in enumerate(["LTD_OK", "LTD_ERR_INVALID_ARG", "LTD_ERR_SHAPE",
                              "LTD_ERR_UNSUPPORTED", "LTD_ERR_CUDA", "LTD_ERR_DEVICE",
                              "LTD_ERR_TIMEOUT"]):
        assert L.ltd_status_string(s).decode() == name


def test_tree_bytes_and_init_validate_on_host(L):
    from paper_2603_01639_gb300 import ltd
    assert L.ltd_tree_bytes(1, 6, 10, 128256) > 0
    assert L.ltd_tree_bytes(0, 6, 10, 128256) == 0
    assert L.ltd_tree_bytes(1, 17, 10, 128256) == 0          # depth over LTD_MAX_DEPTH
    assert L.ltd_tree_bytes(1, 6, 33, 128256) == 0           # k over LTD_MAX_K
    assert L.ltd_tree_bytes(1, 16, 32, 128256) == 0          # more than 4096 nodes
    assert L.ltd_tree_bytes(1, 3, 8, 4) == 0                 # k > vocab
    t = ltd.ltd_tree()
    n = L.ltd_tree_bytes(2, 3, 4, 1000)
    assert L.ltd_tree_init(None, C.c_void_p(256), n, 2, 3, 4, 1000) == 1
    assert L.ltd_tree_init(C.byref(t), None, n, 2, 3, 4, 1000) == 1
    assert L.ltd_tree_init(C.byref(t), C.c_void_p(257), n, 2, 3, 4, 1000) == 1  # misaligned
    assert L.ltd_tree_init(C.byref(t), C.c_void_p(4096), n - 1, 2, 3, 4, 1000) == 2
    # carving is pure pointer arithmetic on the host
    assert L.ltd_tree_init(C.byref(t), C.c_void_p(1 << 20), n, 2, 3, 4, 1000) == 0
    assert t.max_nodes == 1 + 4 + 2 * 16
    ptrs = [t.token, t.parent, t.depth, t.cum_logprob, t.xrow, t.xlse, t.frontier, t.n_nodes,
            t.n_levels, t.scratch]
    assert all(p % 256 == 0 for p in ptrs)
    assert ptrs == sorted(ptrs) and ptrs[-1] + t.scratch_bytes <= (1 << 20) + n


def test_entry_points_reject_bad_arguments_before_launch(L):
    from paper_2603_01639_gb300 import ltd
    t = ltd.ltd_tree()
    n = L.ltd_tree_bytes(1, 3, 4, 1000)
    assert L.ltd_tree_init(C.byref(t), C.c_void_p(1 << 20), n, 1, 3, 4, 1000) == 0
    fake = C.c_void_p(1 << 24)
    s = C.c_void_p(0)
    assert L.ltd_tree_reset(None, fake, s) == 1
    assert L.ltd_tree_reset(C.byref(t), None, s) == 1
    assert L.ltd_expand_tree(C.byref(t), 0, fake, 0, 1000, 9, None, s) == 2       # level 0
    assert L.ltd_expand_tree(C.byref(t), 4, fake, 0, 1000, 9, None, s) == 2       # > max_depth
    assert L.ltd_expand_tree(C.byref(t), 1, fake, 0, 1001, 9, None, s) == 2       # > max_vocab
    assert L.ltd_expand_tree(C.byref(t), 1, fake, 0, 1000, 8, None, s) == 2       # row store short
    assert L.ltd_expand_tree(C.byref(t), 1, fake, 7, 1000, 9, None, s) == 1       # bad dtype
    assert L.ltd_expand_tree(C.byref(t), 1, fake, 1, 996, 9, None, s) == 2        # bf16 row not 16B
    assert L.ltd_select_verify(C.byref(t), fake, 257, fake, fake, fake, fake, s) == 2
    assert L.ltd_select_verify(C.byref(t), None, 8, fake, fake, fake, fake, s) == 1
    assert L.ltd_depth_observation(None, fake, fake, s) == 1
    assert L.ltd_depth_observation(C.byref(t), None, fake, s) == 1
    assert L.ltd_size_observation(C.byref(t), fake, t.max_nodes - 1, fake, s) == 2  # v_pad short
    assert L.ltd_size_observation(C.byref(t), fake, t.max_nodes, None, s) == 1
    net = ltd.ltd_mlp()
    net.n_layers = 2
    net.dims[0], net.dims[1], net.dims[2] = 4 * 4 + 2, 1024, 2
    for i in range(2):
        net.w[i] = 1 << 24
        net.b[i] = 1 << 24
    P = C.byref(net)
    assert L.ltd_depth_policy(C.byref(t), fake, None, None, fake, None, s) == 1
    assert L.ltd_depth_policy(C.byref(t), fake, P, None, None, None, s) == 1        # no output
    net.dims[0] = 17
    assert L.ltd_depth_policy(C.byref(t), fake, P, None, fake, None, s) == 2        # obs length
    net.dims[0], net.dims[2] = 18, 3
    assert L.ltd_depth_policy(C.byref(t), fake, P, None, fake, None, s) == 2        # 3 actions
    net.dims[2] = 2
    net.w[1] = None
    assert L.ltd_depth_policy(C.byref(t), fake, P, None, fake, None, s) == 1        # null weight
    net.w[1] = 1 << 24
    net.n_layers = 5
    assert L.ltd_depth_policy(C.byref(t), fake, P, None, fake, None, s) == 1        # > max layers
    net.n_layers = 2
    net.dims[0], net.dims[2] = t.max_nodes + 2, 12
    assert L.ltd_size_policy(C.byref(t), fake, t.max_nodes - 1, P, 64, fake, None, s) == 2
    assert L.ltd_size_policy(C.byref(t), fake, t.max_nodes, P, 0, fake, None, s) == 2
    assert L.ltd_size_policy(C.byref(t), fake, t.max_nodes, P, 64, None, None, s) == 1
    net.dims[1] = ltd.LTD_MLP_MAX_WIDTH + 1
    assert L.ltd_size_policy(C.byref(t), fake, t.max_nodes, P, 64, fake, None, s) == 2  # width
    net.dims[1] = 1024
    net.layout = 2
    assert L.ltd_size_policy(C.byref(t), fake, t.max_nodes, P, 64, fake, None, s) == 1  # layout
    assert L.ltd_mlp_packed_bytes(P) == 0
    net.layout = ltd.LTD_MLP_ROW_MAJOR
    net.w[0] = (1 << 24) + 4
    assert L.ltd_size_policy(C.byref(t), fake, t.max_nodes, P, 64, fake, None, s) == 1  # misaligned
    assert L.ltd_mlp_packed_bytes(P) == 0
    net.w[0] = 1 << 24
    # packed size: every weight plus column padding, whole 256-byte blocks
    n = L.ltd_mlp_packed_bytes(P)
    assert n >= 4 * ((t.max_nodes + 2) * 1024 + 1024 * 12) and n % 256 == 0
    out = ltd.ltd_mlp()
    assert L.ltd_mlp_pack(P, fake, n, None, s) == 1
    assert L.ltd_mlp_pack(P, C.c_void_p((1 << 24) + 16), n, C.byref(out), s) == 1   # d_mem align
    assert L.ltd_mlp_pack(P, fake, n - 4, C.byref(out), s) == 2
    ws = L.ltd_attention_workspace_bytes(1, 4, 1, 64, 8, 128, 0)
    assert ws > 0
    assert L.ltd_attention_workspace_bytes(1, 5, 2, 64, 8, 128, 0) == 0          # hq % hkv
    args = [fake, fake, fake, fake, 0, 1, 4, 1, 64, 256, fake, 128, fake, 8, fake, 0.125, fake, ws, s]
    bad = list(args); bad[8] = 80                                                  # head_dim
    assert L.ltd_tree_attention(*bad) == 3
    bad = list(args); bad[9] = 130                                                 # s_cap < ctx + n
    assert L.ltd_tree_attention(*bad) == 2
    bad = list(args); bad[17] = ws - 1
    assert L.ltd_tree_attention(*bad) == 2
    bad = list(args); bad[15] = 0.0
    assert L.ltd_tree_attention(*bad) == 1
    nxt = args[:18] + [fake, fake, s]                                               # the hint
    bad = list(nxt); bad[19] = None                                                # one of two
    assert L.ltd_tree_attention_next(*bad) == 1
    bad = list(nxt); bad[18] = C.c_void_p((1 << 24) + 8)                          # misaligned
    assert L.ltd_tree_attention_next(*bad) == 2
    bad = list(nxt); bad[8] = 80
    assert L.ltd_tree_attention_next(*bad) == 3
    assert L.ltd_debug_attention_wait(1000, 1025) == 1                            # too many
    assert L.ltd_debug_attention_wait(0, 0) == 0
    assert L.ltd_debug_expand_wait(1000, 1025) == 1                               # offset too big
    assert L.ltd_debug_expand_wait(0, 0) == 0
    assert L.ltd_accept_workspace_bytes(1, 8, 1000) > 0
    assert L.ltd_accept_workspace_bytes(1, 300, 1000) == 0
    kv = ltd.ltd_kv_cache(fake, fake, 1, 1, 70, 256, 1)                            # 140-byte rows
    assert L.ltd_kv_compact(C.byref(kv), 1, fake, 4, fake, fake, s) == 3
    assert L.ltd_kv_compact(None, 1, fake, 4, fake, fake, s) == 1
    kv_ok = ltd.ltd_kv_cache(fake, fake, 2, 1, 64, 256, 1)                          # 128-byte rows
    assert L.ltd_kv_append(C.byref(kv), 1, 8, fake, fake, fake, fake, s) == 3        # 140-byte rows
    assert L.ltd_kv_append(None, 1, 8, fake, fake, fake, fake, s) == 1
    assert L.ltd_kv_append(C.byref(kv_ok), 1, 8, C.c_void_p((1 << 24) + 8), fake, fake, fake, s) == 1
    assert L.ltd_kv_append(C.byref(kv_ok), 1, 0, fake, fake, fake, fake, s) == 2     # n_max 0
    assert L.ltd_kv_append(C.byref(kv_ok), 0, 8, fake, fake, fake, fake, s) == 2     # batch 0
    assert L.ltd_kv_append(C.byref(kv_ok), 1, 8, fake, None, fake, fake, s) == 1


def test_attention_split_plan_on_a_152_sm_device(L):
    """The host plan of the tensor-core attention (no GPU here, so the SM
    count falls back to 152): units = (sequence, KV head, 128-row tile);
    with fewer units than SMs each unit's keys are cut into the fewest
    splits that give the shortest longest split, at most SMs / units; the
    workspace holds a 32 KB bf16 partial and 128 fp32 log2-sum-exps per
    (unit, split), plus two counters per unit, each part 256-byte aligned."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("the fallback SM count applies only without a device")

    def ws(units, splits):
        rows = units * splits * 128
        a = lambda n: (n + 255) // 256 * 256  # noqa: E731
        return a(rows * 256) + a(rows * 4) + a(units * 2 * 4)

    BF16 = 1
    # 8B-class: 8 heads x 2 tiles (240 rows), 33 chunks -> 9 splits of <= 4
    assert L.ltd_attention_workspace_bytes(1, 32, 8, 128, 60, 4096, BF16) == ws(16, 9)
    # 13B-class MHA: 40 units (one tile), 17 chunks -> 3 splits of <= 6
    assert L.ltd_attention_workspace_bytes(1, 40, 40, 128, 96, 2048, BF16) == ws(40, 3)
    # 32B-class: 8 heads x 3 tiles, 129 chunks -> 6 splits of <= 22
    assert L.ltd_attention_workspace_bytes(1, 64, 8, 128, 48, 16384, BF16) == ws(24, 6)
    # 70B-class batch: 768 units >= 152 SMs -> one split per unit, no partials
    assert L.ltd_attention_workspace_bytes(16, 64, 8, 128, 96, 8192, BF16) == 256
    # 4 units over 32 chunks -> 32 splits of one chunk
    assert L.ltd_attention_workspace_bytes(1, 8, 2, 128, 60, 3968, BF16) == ws(4, 32)

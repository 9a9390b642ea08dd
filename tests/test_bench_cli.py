"""bench.py's command line on CPU: the defaults the driver relies on."""

import sys


def _parse(monkeypatch, *argv):
    import bench
    monkeypatch.setattr(sys, "argv", ["bench.py", *argv])
    return bench._args()


def test_defaults_are_one_gpu_the_8b_workload_and_no_next_layer_hint(monkeypatch):
    a = _parse(monkeypatch)
    assert a.gpus == 1 and a.config == "8b" and a.impl == "ours"
    assert not a.next_hint
    assert a.warmup >= 3


def test_next_layer_hint_is_opt_in_and_the_old_flag_still_parses(monkeypatch):
    assert _parse(monkeypatch, "--next-hint").next_hint
    a = _parse(monkeypatch, "--no-next-hint", "--steps", "20", "--warmup", "3")
    assert not a.next_hint and a.steps == 20 and a.warmup == 3

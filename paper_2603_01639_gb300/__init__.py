"""GB300-native hot path of one LTD draft-and-verify cycle.

The compute lives in ``libltd.so`` (hand-written CUDA for sm_103a behind the
C ABI declared in ``include/ltd.h``); :mod:`.ltd` is the thin ctypes binding
with the same call names, and :mod:`.workload` draws the seeded synthetic
inputs.  Importing the package loads nothing: the binding loads the library on
first use and raises if it is missing.
"""

__all__ = ["ltd", "workload"]

"""CPU oracles of SARA's rollout-collection hot path (arxiv 2607.26253).

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and
bench.py's CPU-baseline / reference leg, never by the product package.  It
shares no code with paper_2607_26253_gb300/ (the CUDA path); the only common
dependency is the seeded input generator `synth`, which holds none of the
method's arithmetic.

  oracle.controller  O1: Algorithm 1 with Eq. (peff) / Eq. (decide), exact
                     rational arithmetic, plain C (oracle/controller.c).
  oracle.decode      O2: the decoder policy forward pass and Gumbel-max
                     sampling in float64 numpy.
  oracle.async_schedule  O1a: the asynchronous per-prompt variant of the step
                     (no round barrier), on O1's predictor and rule.
"""
import os
import subprocess
import threading

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libo1.so")
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile oracle/controller.c into oracle/_build/libo1.so with gcc."""
    src = os.path.join(_HERE, "controller.c")
    with _lock:
        if (not force and os.path.exists(LIB_PATH)
                and os.path.getmtime(LIB_PATH) >= os.path.getmtime(src)):
            return LIB_PATH
        os.makedirs(os.path.dirname(LIB_PATH), exist_ok=True)
        tmp = LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fPIC", "-shared", "-fno-fast-math", "-o", tmp, src,
                               "-lm"])
        os.replace(tmp, LIB_PATH)
    return LIB_PATH

"""Seeded synthetic inputs shared by the oracle, the tests and the benchmark.

This package generates inputs only: model weights, item identifiers, prompts and
random trees/logits for kernel-level parity cases.  It contains none of the
method's arithmetic (no forward pass, no log-softmax, no beam search, no
verification), so the oracle and the CUDA path can both consume it without
sharing any computation.
"""
from .world import *  # noqa: F401,F403

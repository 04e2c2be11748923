"""DFlow speculative-decoding round (arXiv 2609.06498) on one GB300.

The round -- drafter block forward, target verification, acceptance/commit and
DFlow's verifier-state carry -- runs in hand-written sm_103a CUDA behind the C
ABI of include/dflow.h (libdflow.so).  This package holds that library's
sources (csrc/), its build script, and a thin PyTorch-facing binding.
"""
from ._abi import EXPORTS, DFlowError, lib  # noqa: F401
from .engine import DeviceState, DeviceWeights, Engine, pack_weights, random_weights  # noqa: F401

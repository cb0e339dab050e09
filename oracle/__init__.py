"""CPU oracle of the LCA multi-byte-prediction decode step (fp64 numpy).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py`` (CPU baseline and reference arm) and by nothing in the CUDA product
path, with which it shares no code.
"""
from .decode import (SPEC, THRESH, IncrementalDecoder, StepRecord, generate_incremental,
                     generate_reference, greedy_decode)
from .external import ExternalDecoder, generate_external, generate_external_reference
from .model import Model, forward_full
from .sampling import Sampling

__all__ = ["SPEC", "THRESH", "IncrementalDecoder", "StepRecord", "generate_incremental",
           "generate_reference", "greedy_decode", "Model", "forward_full", "Sampling",
           "ExternalDecoder", "generate_external", "generate_external_reference"]

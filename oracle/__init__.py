"""CPU oracle (float64) for the speculative draft-verify step.

TEST INFRASTRUCTURE: only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import it.  The CUDA library never calls
it, and the two share no code; both read inputs drawn by ``workload``.

Every function is pinned by the CPU tests (``tests/test_oracle_*.py``) against
library routines (torch.nn's Transformer decoder and multi-head attention),
brute-force enumeration, the lossless invariant and closed forms.
"""
from .decoder import (Oracle, OracleError, VerifyResult, attention, gelu,
                      greedy_transcript, head_mean_attention, layer_norm, softmax)

__all__ = ["Oracle", "OracleError", "VerifyResult", "attention", "gelu",
           "greedy_transcript", "head_mean_attention", "layer_norm", "softmax"]

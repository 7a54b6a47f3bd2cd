"""CPU oracle of the CDSL lookahead step (fp64 numpy).

TEST INFRASTRUCTURE. Only tests/, ``__graft_entry__.smoke()`` and bench.py's ``cpu_baseline``
and ``--impl reference`` legs may import, call or execute anything in this package; the
product path (the CUDA library and its Python binding) never does, and shares no code with it.

Parity pins (tests/test_oracle_*.py) tie each part to something other than the oracle itself:
closed forms (RoPE as complex rotation, one-key attention, RMS of RMSNorm), a loop-by-loop
restatement of the transformer on tiny shapes, the verify == sequential-decode identity, the
draft == target full-acceptance property, the CDSL -> CDLH reduction, a brute-force beam
selection on a 16-token vocabulary, and the paper's worked reward example (Sec. 4.1).
Parity unpinned: the end-to-end token values of a CDSL step on random models (the paper
prints no worked token-level example); they rest on the pins of the parts above.
"""
from .model import KVCache, Transformer, log_softmax, rms_norm, rope, silu, softmax, widen
from .cdsl import (S1, S2_S3, S2_S3_STEP1, S4, Decider, PromptState, RunParams, StepRecord,
                   alg1_generate, alg1_step, cdlh_generate, cdlh_token, cdsl_k_generate,
                   cdsl_k_step, coverage, n_min, prefill, reward, HARD, SPECULATIVE, splitmix64,
                   uniform24, draw_index, runtime_per_token, speedup)

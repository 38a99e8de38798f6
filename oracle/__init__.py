"""CPU oracle for RVQ-position-aware speculative decoding (arXiv 2609.37007).

TEST INFRASTRUCTURE ONLY.  Plain, slow, fp64 restatement of what the hot path computes,
written from the paper: the MultiCodeDecoder forward pass (Sec. 1, Fig. 1), the
position-aware offset drafter (Sec. 2.2, Fig. 3), top-k/temperature sampling and the
lossless speculative acceptance rule with residual resampling (Sec. 2.2 and Sec. 3.2),
and the per-frame draft/verify loop that emits c1..c15.

Only the tests, `__graft_entry__.smoke()` and the CPU-baseline leg of `bench.py` may
import this package.  It shares no code with the CUDA library; the only common module
is `paper_2609_37007_gb300.synth`, which draws inputs and holds none of the arithmetic.

Modules:
  philox       Philox4x32-10 counter-based generator and the uniform/normal draws.
  sampler      top-k / temperature / softmax, categorical draw, accept test, residual.
  model        fp64 MultiCodeDecoder rows with a per-frame KV cache.
  frame        autoregressive and speculative frame procedures.
  codedecoder  the outer CodeDecoder (one call per frame, emits c0) and the full frame
               pipeline of Fig. 1 (prompt prefill, c0, MultiCodeDecoder, input sum).
  quant        W8A16 per-row symmetric int8 weights.
  tree         sparse tree drafting and verification (Fig. 2) and the greedy tree growth.
  enumeration  exact output distributions of the procedures (losslessness pin).
  accounting   the paper's real-time call arithmetic.

Parity status: every function here is pinned by a `-m "not gpu"` test
(tests/test_oracle_*.py) except where its docstring says "parity unpinned".
"""

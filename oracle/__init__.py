"""CPU oracle for one bidirectional refine step -- TEST INFRASTRUCTURE ONLY.

This package is the plain, slow, obviously-correct statement of what the GPU
library computes. Only the test suite, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import it. The
library and its Python binding never import it, and it imports nothing from
them: the two share no kernels, headers, helpers or constants.

Method (speculative correction, Sec. 4.2): the refiner takes the fixed prompt
plus a complete draft and runs full-sequence bidirectional denoising passes in
which any response position may be revised. One pass on the hot path is

* ``attention.bidir_attn``      -- non-causal GQA attention over all valid
  positions (Sec. 4.2: correction over the entire sequence; Sec. 3.3 contrasts
  it with block-causal decoding);
* ``vocab.vocab_confidence``    -- per position, over the vocabulary: argmax,
  maximum softmax probability and log-sum-exp (the confidences that gate
  edits, Table 10 "Refine th." and Appendix C.4's confident edits);
* ``update.refine_update``      -- commit masked positions, edit confident
  changes of filled draft tokens, remask the k least confident positions
  (Appendix C.4, Table 11: token editing that stops when no confident edits remain);
  optionally ranked by the probability of each position's resulting token,
  with ``vocab.token_prob`` giving the probability of a kept token.

``loop.refine_passes`` repeats such passes over a batch, each on the state the
last one left, until a pass makes no confident edit or a pass budget is spent
(Sec. 4.2's T_r passes; Appendix C.4's early stop when no confident edits
remain).

``lmhead.lm_head_confidence`` is the vocabulary projection (hidden states times
the output weights) followed by ``vocab.vocab_confidence``, the operation of
the fused projection + reduction kernel.

Floating point is fp64 unless a comparison is defined in fp32 (edit threshold,
remask order), where the fp32 values are compared exactly.

Parity pins (tests/test_oracle_*.py) tie every function to something other than
itself: brute-force loops on tiny inputs, torch fp64 library routines, closed
forms, invariants and hand-worked update examples (tests/golden/).
"""
from .attention import bidir_attn  # noqa: F401
from .vocab import token_prob, vocab_confidence  # noqa: F401
from .update import refine_update, remask_count  # noqa: F401
from .lmhead import lm_head_confidence, lm_head_logits  # noqa: F401
from .loop import refine_passes  # noqa: F401

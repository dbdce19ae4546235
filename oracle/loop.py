"""Oracle of the multi-pass refinement with early stop -- test infrastructure.

Sec. 4.2: the refiner revisits the whole response over T_r full-span passes.
Appendix C.4 (with Table 11's mask-only diagnostic of up to 52 passes): the
native editing rule ends the refinement early, once a pass makes no confident
edit. One pass here is

1. the refiner's forward pass on the current state gives the pass's logits
   (``logits_for(tokens, mask, t)``, a callable supplied by the caller: the
   model stand-in);
2. ``vocab.vocab_confidence`` of those logits (argmax, confidence);
3. ``update.refine_update`` of the current state with them (commit masked
   positions, edit confident changes, remask the k least confident).

The passes repeat while the last pass made at least one edit in some
sequence of the batch and fewer than ``max_passes`` passes have run. The stop
is batch-level: every sequence takes part in every pass the batch runs, since
one pass is one forward pass over the whole batch. Commits of masked
positions are not edits and do not keep the loop going.
"""
from __future__ import annotations

import numpy as np

from .update import refine_update
from .vocab import vocab_confidence


def more_passes(n_edits, passes: int, max_passes: int) -> bool:
    """Whether another pass runs after `passes` passes whose last one made
    the per-sequence edit counts `n_edits`."""
    return passes < max_passes and bool(np.any(np.asarray(n_edits) > 0))


def refine_passes(tokens, mask, logits_for, *, max_passes, edit_threshold, remask_k, remask_frac, mask_id,
                  prompt_lens, seq_lens):
    """Runs passes from the state (tokens int [B,L], mask uint8 [B,L]).

    logits_for(tokens, mask, t) -> logits [B*L, V] (or [B, L, V]) of pass t
    (t = 0, 1, ...) given the state that pass starts from. edit_threshold is
    one value or one per pass (the last one repeats).

    Returns a dict: passes (int), tokens, mask, n_edits (of the last pass) and
    history, a list with (tokens, mask, n_edits) after each pass."""
    if max_passes < 1:
        raise ValueError("max_passes must be >= 1")
    tok = np.array(tokens, dtype=np.int32, copy=True)
    msk = np.array(mask, dtype=np.uint8, copy=True)
    B, L = tok.shape
    taus = list(np.atleast_1d(edit_threshold))
    history = []
    passes = 0
    n_edits = np.zeros(B, dtype=np.int32)
    while True:
        x = np.asarray(logits_for(tok, msk, passes))
        am, cf, _ = vocab_confidence(x.reshape(B * L, -1))
        tau = taus[min(passes, len(taus) - 1)]
        tok, msk, n_edits = refine_update(tok, msk, am.reshape(B, L), cf.reshape(B, L), edit_threshold=tau,
                                          remask_k=remask_k, remask_frac=remask_frac, mask_id=mask_id,
                                          prompt_lens=prompt_lens, seq_lens=seq_lens)
        passes += 1
        history.append((tok.copy(), msk.copy(), n_edits.copy()))
        if not more_passes(n_edits, passes, max_passes):
            break
    return {"passes": passes, "tokens": tok, "mask": msk, "n_edits": n_edits, "history": history}

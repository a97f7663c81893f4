"""Oracle: the acceptance pass of one block of positions, from given logits.

Test infrastructure only (see ``oracle/__init__.py``).

For each row b of a block of P positions with c_b positions already committed
(left-aligned, so the window starts at p = c_b):
  * confidence of every uncommitted position from its logits (Eq. 2; top-1 id and
    probability, or exp(-entropy) with ``confidence = 1``; top-2 probability for reporting),
  * K over the window [p, p + L') with L' = min(L, P - p)          (Eq. compute_k),
  * commit x[p:p+K] and refresh drafts at i >= p + L                (Eq. draft_update),
using the same readings as ``oracle.decode``; with ``acceptance = 1`` instead every
uncommitted position of [p, P) with c > tau_commit is committed (Eq. threshold_pd, at least
``min_commit`` of them by confidence), no drafts, and K is the number committed.
"""
from __future__ import annotations

import numpy as np

from . import decode, model


def accept(logits: np.ndarray, committed: np.ndarray, x: np.ndarray,
           cfg: decode.DecodeConfig, window: int):
    """logits float [B][P][V] (bf16 values); committed int [B]; x int [B][P] (copied).

    Returns (K [B], x_out [B][P], ids [B][P], c [B][P], p2 [B][P]) where c is the
    decision confidence (p1, or exp(-H) with ``cfg.confidence = 1``); confidences of
    committed positions are reported as 0 and id -1 (they are never read).
    """
    B, P, _ = logits.shape
    x_out = np.array(x, dtype=np.int32, copy=True)
    ids = np.full((B, P), -1, dtype=np.int32)
    p1 = np.zeros((B, P))
    p2 = np.zeros((B, P))
    K = np.zeros(B, dtype=np.int32)
    for b in range(B):
        p = int(committed[b])
        if p >= P:
            continue
        z = logits[b, p:].astype(np.float64)
        i_, c1, c2 = model.confidence(z)
        H = model.entropy(z) if cfg.confidence == 1 else None
        ids[b, p:], p1[b, p:], p2[b, p:] = i_, decode.decision_confidence(c1, H, cfg), c2
        if cfg.acceptance == 0:
            K[b] = decode.commit_and_draft(x_out[b], p, ids[b], p1[b], cfg, window)
        else:  # Eq. threshold_pd over the uncommitted rest of the block, no drafts
            committed_b = np.arange(P) < p
            K[b] = len(decode.threshold_commit(x_out[b], committed_b, ids[b], p1[b], p, P, cfg))
    return K, x_out, ids, p1, p2

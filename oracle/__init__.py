"""CPU oracle of the DC-Leap denoise step (plain numpy, fp64).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The CUDA library never calls it, shares no code with it, and must
fail loudly rather than fall back to it.

Modules:
  model   - masked-diffusion transformer forward and per-position softmax
            confidence (Eq. 1, Eq. 2, top-1 of Eq. threshold_pd, top-2 of Sec. 2.2,
            the marginal entropy of Eq. entropy_bound)
  decode  - Dynamic Contiguous Verification and draft-guided decoding
            (Eq. compute_k, Eq. draft_update, Eq. remasking, Sec. 3.3, Algorithm 1),
            the entropy confidence and Eq. entropy_bound of each committed set
  accept  - the acceptance pass on given logits (Eq. 2 + Eq. compute_k +
            Eq. draft_update for a block of positions)
  fp8     - the FP8 (E4M3) weight format with per-row power-of-two scales (a serving
            refinement outside the paper): the stored weights' values

Every function is pinned by a ``-m "not gpu"`` test against something other than
itself (closed forms, invariants, library routines, brute force); the model-level
throughput and accuracy numbers of the paper need trained weights and are parity
unpinned.
"""
from . import model, decode, accept, fp8  # noqa: F401

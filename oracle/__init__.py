"""CPU oracle for the FeatFix cached diffusion-transformer denoising path.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports, calls or links
this package: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.

Every function is plain float64 numpy written from the paper
(FeatFix, "Reuse What You Verify through Local Exact-Feature Correction for
Faster Cached Diffusion Inference"):

* ``oracle.model``    -- the exact block B_l(u; t, c) of Eq. 1 (DiT adaLN block,
  MMDiT dual- and single-stream blocks), embeddings, final layer.
* ``oracle.draft``    -- the order-K Taylor draft of Eq. 2 (finite differences
  estimated at exact refreshes) and the reuse draft (K = 0).
* ``oracle.schedule`` -- the fixed layer-timestep plan: refresh steps, the site
  set S (Section 3.3) and the per-(step, layer) decision.
* ``oracle.sampler``  -- Euler flow-matching / rectified-flow and DDIM updates,
  classifier-free guidance.
* ``oracle.featfix``  -- the cached sampling loop with the paid same-input pair
  (Eq. 3), the relative-L1 discrepancy (Eq. 4, plus relative L2), the
  forwarding rule (Eq. 5), the Verify / Exact-only arms and the accounting of
  full refreshes, paid checks and forwarded corrections (Section 3.3).
* ``oracle.noise``    -- the seeded initial latent: SplitMix64 counters mapped
  to normals by Box-Muller.
* ``oracle.flops``    -- FLOP accounting of one denoising step.

Parity status: the method is an approximation (draft + sparse exact
correction), so the oracle runs the algorithm step by step.  Its parts are
pinned by ``tests/test_oracle_pins.py`` against closed forms, library
routines, brute force and the paper's stated invariants, and
``tests/test_oracle_mutations.py`` plants plausible mistakes in a temporary
copy of this package to show that a pin fails for each.  Absolute latents on
random weights have no printed value in the paper: that end-to-end value is
"parity unpinned" against the paper and is checked oracle <-> GPU only.
"""

from . import model, draft, schedule, sampler, featfix, noise, flops  # noqa: F401

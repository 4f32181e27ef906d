"""CPU oracle for FP8 token scoring followed by Calibrated Clipping.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the ``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import
this package.  The product path (``paper_2609_22870_gb300``) never imports,
links or executes anything from here, and nothing here imports the product
path.  The two share no kernels, helpers, tables or constants; only the seeded
input generator (``paper_2609_22870_gb300.synth``, which holds none of the
method's arithmetic) feeds both.

The oracle is deliberately plain and slow: float64 arithmetic, full sorts,
exact integer sums, and numpy primitives (matmul, sort) as single steps with no
blocking or fusion beyond what each definition states.  Every function cites
the passage of "Towards Full Pipeline FP8 Reinforcement Learning for LLMs"
that it follows.

Modules
-------
e4m3        OCP FP8 E4M3 ("fn") decode and round-to-nearest-even saturating
            encode (the Q_FP8 of Eq. 3, §2.2).
quantize    scaled FP8 quantisation at tensor / row / block granularity
            (Eq. 3 and the three scaling strategies, §2.2).
logprobs    dequantised logits, log-softmax, target gather, importance
            ratio and dLoss/dlogits (§2.1 ratio definition).
calibrate   Calibrated Clipping: lower-bound alignment, upper-bound
            rebalancing, SmoothUpdate (§4, Eq. 5, Algorithm 1).
surrogate   clipped PPO surrogate with TIS weights, token-mean
            aggregation, clip fractions and dLoss/dlogp (Eq. 1, Eq. 4);
            the sequence-mean aggregation (§2.1) and the sequence-level
            ratio clipping of the related-work discussion (§6).
diagnostics over-clipping counts, clip fractions and probability / ratio
            NMAE against BF16 references (§3); TIS weights (§2.3).
"""

from . import e4m3, quantize, logprobs, calibrate, surrogate, diagnostics  # noqa: F401

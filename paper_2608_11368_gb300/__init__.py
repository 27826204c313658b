"""GB300-native (sm_103a) hot path of the Pair estimator.

Pairwise-Aware Inclusion Reweighting (PAIR) estimates the complete-pair
policy gradient of a group of RLVR rollouts from an adaptively completed
subset, weighting every observed edge (i, j) by its logged joint inclusion
probability (Sec. 4.5, Eq. pair-ht). The hot path is exposed by the C-ABI
library ``libpair.so`` (header ``include/pair.h``):

* ``pair_coeffs``: per-rollout coefficients of Eq. (pair-advantage);
* ``pair_grad``: the LM-head realisation of the objective sum_i A_i log pi;
* ``pair_estimate_dense``: Eq. (pair-ht) for explicit score vectors.

``binding`` wraps those entry points for torch tensors (argument marshalling
only). ``synth`` draws seeded synthetic workloads. Importing this package
does not load the CUDA library; ``binding`` does, and raises if it is
missing.
"""
__all__ = ["binding", "synth", "build"]

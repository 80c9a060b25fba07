"""Pr^2 (Predictive Routing Replay) MoE-layer forward for GB300 (sm_103a).

The compute lives in ``libpr2.so`` (hand-written CUDA kernels behind the C ABI declared in
``include/pr2.h``); ``binding`` marshals torch tensors to that ABI.  ``synth`` draws the seeded
synthetic layers and ``cost`` holds the closed-form cost model.  Importing the package does not
load the CUDA library; the first call into ``binding`` does, and fails loudly if it is missing.
"""
__all__ = ["binding", "synth", "cost", "build"]

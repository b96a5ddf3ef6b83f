"""Seeded synthetic inputs for the ZO-Act hot path.

This module holds no arithmetic of the method.  It only draws the inputs that
both the CUDA path and the CPU oracle consume (frozen weights, activations,
calibration batches, targets, initial coefficients) and stores them at the
precision the workload fixes.  Random numbers the method itself draws (the
perturbation Z, the basis sketch) are not produced here: each side regenerates
them from its own implementation of Philox4x32-10.

The paper's workloads (Llama-3-8B, OPT-13B, INT4 Llama-3-8B on SuperGLUE and
commonsense tasks) need weights and datasets that are not available; these
generators stand in for them with the same layer shapes and with activations
whose spectrum is dominated by a low-rank component, the structure Section 3
relies on.
"""
from .gen import *  # noqa: F401,F403
from .configs import *  # noqa: F401,F403

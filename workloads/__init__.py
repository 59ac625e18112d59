"""Seeded synthetic workloads (shapes, contexts, budgets, tensors) for the
budget-routed decode step.  Shared by the GPU path's harness and the oracle."""
from . import configs, synth  # noqa: F401

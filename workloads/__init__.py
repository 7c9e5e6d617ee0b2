"""Seeded synthetic inputs for DVI (arxiv 2510.05421).

This package holds only shapes, hyper-parameters and seeded random inputs
(weights, prompts).  It contains none of the method's arithmetic, so both the
CPU oracle and the CUDA path may take their inputs from it.
"""
from .configs import (ModelShape, Workload, UpdateHyper, WORKLOADS, workload,
                      tiny_shape)
from .gen import make_weights, make_prompts, zipf_ids, Weights, LayerWeights

__all__ = ["ModelShape", "Workload", "UpdateHyper", "WORKLOADS", "workload",
           "tiny_shape", "make_weights", "make_prompts", "zipf_ids", "Weights",
           "LayerWeights"]

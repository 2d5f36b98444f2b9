"""Seeded synthetic inputs for the CMC two-tier decode path.

This package is the one input source that both the CUDA path and the CPU oracle
consume.  It draws random tensors and lays them out; it contains none of the
method's arithmetic (no cosine scoring, no top-k selection, no attention).
"""

from .configs import Workload, WORKLOADS, ablation_workloads, get_workload
from .generate import (
    SelectionInputs,
    QuestionInputs,
    ContextInputs,
    KVInputs,
    StepInputs,
    selection_inputs,
    question_inputs,
    context_inputs,
    kv_inputs,
    step_inputs,
    random_tier1_indices,
    f32_to_bf16_bits,
    bf16_bits_to_f32,
)

__all__ = [
    "Workload",
    "WORKLOADS",
    "ablation_workloads",
    "get_workload",
    "SelectionInputs",
    "QuestionInputs",
    "ContextInputs",
    "KVInputs",
    "StepInputs",
    "selection_inputs",
    "question_inputs",
    "context_inputs",
    "kv_inputs",
    "step_inputs",
    "random_tier1_indices",
    "f32_to_bf16_bits",
    "bf16_bits_to_f32",
]

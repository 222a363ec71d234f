"""Seeded synthetic inputs for the DFlare draft path.

This package is shared by the CPU oracle's tests and by the GPU path's tests and benchmark. It
holds none of the draft path's arithmetic: it only produces numbers with stated distributions
from (seed, tensor name, element index), through the counter-based generator in ``synth.c``.
Any slice of any tensor can be regenerated on its own, so a large context fill can be produced
chunk by chunk and a single position can be regenerated for a spot check.

bf16 tensors are returned as ``numpy.uint16`` arrays holding the raw bf16 bits; fp32 tensors as
``numpy.float32``. Each consumer decodes them in its own code.
"""
from .gen import build, lib, tensor_id, normal, uniform, uniform_u32, randint  # noqa: F401
from .recipes import (  # noqa: F401
    Shape,
    Workload,
    PRESETS,
    preset,
    sweep_point,
    weights,
    variant_weights,
    hidden_states,
    initial_tokens,
    target_draws,
    accept_threshold,
)

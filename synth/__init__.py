"""Seeded synthetic video and weights shaped like the Skip-Conv workloads.

This package only draws inputs: frames, weights and biases, plus the
float32 -> bfloat16 storage rounding of those inputs.  It holds none of the
Skip-Conv arithmetic (no residual, gate or convolution); the oracle and the
CUDA library both consume exactly what it produces.
"""
from .video import (  # noqa: F401
    bf16_bits,
    bf16_bits_to_f32,
    round_to_bf16,
    moving_squares_video,
    moving_rect_video,
    panning_video,
    traffic_video,
    block_perturbation_video,
    he_weights,
)
from .workloads import MARGIN_REDRAWS, REDRAW_STRIDE, WORKLOADS, LayerDef, Workload, make_workload  # noqa: F401

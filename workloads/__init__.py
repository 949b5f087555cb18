"""Seeded synthetic workloads for the quantized MoE expert FFN.

This package holds only input generation (shapes, seeds, random draws) and
byte/FLOP accounting.  It contains none of the method's arithmetic: no
quantizer, no dequantizer, no routing.  Both the CUDA path's tests/benchmark
and the oracle consume the arrays produced here.
"""
from .configs import CONFIGS, LayerSpec, get_config  # noqa: F401

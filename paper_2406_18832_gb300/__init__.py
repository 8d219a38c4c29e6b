"""GB300-native (sm_103a) per-channel quantized linear layer of OutlierTune
(arXiv 2406.18832): calibration, weight folding with bias correction,
symmetrize + quantize, and the exact integer GEMM with a fused epilogue,
behind the C ABI of include/outliertune.h.

The CUDA library is loaded on first use (``binding.load()``); importing the
package does not need a GPU.
"""
from .layer import QuantizedBlockLinears, QuantizedLinear  # noqa: F401

__all__ = ["QuantizedLinear", "QuantizedBlockLinears"]

"""bf16 operand rounding (round to nearest, ties to even), written from the
IEEE-754 definition: bf16 keeps the top 16 bits of an fp32 word; the dropped
low half decides rounding, ties going to the value whose kept LSB is 0.

Used for the reading that every GEMM operand (activations, weights, output
gradients) is rounded fp32 -> bf16 before the product.  Test infrastructure.
"""
import numpy as np


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bf16 value (RNE); returns fp32."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    assert np.all(np.isfinite(x)), "bf16 rounding of non-finite values is not defined here"
    u = x.view(np.uint32).astype(np.uint64)
    low = u & np.uint64(0xFFFF)
    high = u >> np.uint64(16)
    half = np.uint64(0x8000)
    round_up = (low > half) | ((low == half) & ((high & np.uint64(1)) == np.uint64(1)))
    high = high + round_up.astype(np.uint64)
    out = (high << np.uint64(16)).astype(np.uint32)
    return out.view(np.float32).reshape(x.shape)


def identity(x: np.ndarray) -> np.ndarray:
    """No operand rounding (pure fp32 operands, e.g. softmax regression)."""
    return np.asarray(x, dtype=np.float32)

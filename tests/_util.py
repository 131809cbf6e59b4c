"""Helpers shared by the GPU parity tests (no method arithmetic)."""
import numpy as np
import torch


def bf16_bits_from_f64(x: np.ndarray) -> np.ndarray:
    """Round float64 values to bfloat16, to nearest with ties to even, in one step
    (no intermediate float32 rounding).  Returns the uint16 bit patterns."""
    x = np.asarray(x, np.float64)
    out = np.empty(x.shape, np.float64)
    ax = np.abs(x)
    tiny = ax < 2.0 ** -126                       # bf16 subnormal range, spacing 2^-133
    out[tiny] = np.rint(x[tiny] / 2.0 ** -133) * 2.0 ** -133
    m, e = np.frexp(x[~tiny])                     # x = m 2^e, 0.5 <= |m| < 1
    out[~tiny] = np.ldexp(np.rint(m * 256.0) / 256.0, e)
    out[np.isnan(x)] = np.nan
    f32 = out.astype(np.float32)                  # exact: 8 significant bits
    f32[np.abs(out) >= 2.0 ** 128] = np.copysign(np.inf, out[np.abs(out) >= 2.0 ** 128])
    return (f32.view(np.uint32) >> 16).astype(np.uint16)


def bf16_tensor_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def bf16_ulp_distance(a_bits: np.ndarray, b_bits: np.ndarray) -> np.ndarray:
    """Distance in bf16 steps between two arrays of bf16 bit patterns (+0 == -0)."""
    def key(u):
        u = u.astype(np.int64)
        mag = u & 0x7FFF
        return np.where(u & 0x8000, -mag, mag)
    return np.abs(key(a_bits) - key(b_bits))


def logits_for_oracle(logits: torch.Tensor) -> np.ndarray:
    """Host copy in the layout the oracle reads: float32, or bf16 bit patterns."""
    t = logits.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()

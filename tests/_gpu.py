"""Helpers shared by the GPU tests (device buffers, bf16 bit conversions, error norms)."""
import os

import numpy as np
import pytest
import torch

import synthetic as syn


def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def flglm():
    """The binding, with the library built if it is not there yet."""
    from paper_2406_14898_gb300 import flglm as F
    if not os.path.exists(F.LIB_PATH):
        from paper_2406_14898_gb300 import build
        build.build()
    F.lib()
    return F


def dev_bf16_from_bits(bits: np.ndarray) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(bits, np.uint16).view(np.int16))
    return t.view(torch.bfloat16).cuda()


def dev_bf16(x: np.ndarray) -> torch.Tensor:
    return dev_bf16_from_bits(syn.f32_to_bf16_bits(np.asarray(x, np.float32)))


def dev_f32(x: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).cuda()


def dev_i32(x) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(x, np.int32)).cuda()


def bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def f64(t: torch.Tensor) -> np.ndarray:
    if t.dtype == torch.bfloat16:
        return syn.bf16_bits_to_f64(bits(t))
    return t.detach().double().cpu().numpy()


def rnd_bf16_f64(rng, shape, scale=1.0) -> np.ndarray:
    """Random values already representable in bf16 (so both sides see the same inputs)."""
    v = (scale * rng.standard_normal(shape)).astype(np.float32)
    return syn.bf16_bits_to_f64(syn.f32_to_bf16_bits(v)).reshape(shape)


def rel_inf(a, b) -> float:
    """max|a - b| / max|b| (the tolerance metric of the parity tests)."""
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    den = np.abs(b).max()
    return float(np.abs(a - b).max() / (den if den > 0 else 1.0))


def rope_table(max_pos: int, rotary_dim: int, base: float) -> np.ndarray:
    """[pos][i] = (cos, sin) of pos * base^(-2i/rotary_dim), from the definition, in double."""
    half = rotary_dim // 2
    ang = np.arange(max_pos, dtype=np.float64)[:, None] * base ** (-2.0 * np.arange(half) / rotary_dim)[None, :]
    return np.stack([np.cos(ang), np.sin(ang)], axis=-1).astype(np.float32)

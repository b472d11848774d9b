"""Shared helpers of the GPU parity tests: numpy <-> device marshalling and the comparison rules.

Comparison rules (SemShareKV's fuzzy matching path; tolerances fixed by the parity contract):
  projections  |p_gpu - p_oracle| <= 1e-3 * max_j |p_oracle[row, j]|   (per element, per row)
  codes        bit-exact, except bits whose oracle projection lies inside that same band
               (|p_oracle| < 1e-3 * max_j |p_oracle[row, j]|), where the sign is not decided
  match        idx and dist bit-exact when both sides search the same codes
  gather       bit-exact
"""
import numpy as np
import torch

BAND = 1e-3


def bf16_dev(bits: np.ndarray, device="cuda") -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(device).view(torch.bfloat16)


def bf16_host(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().view(torch.int16).numpy().view(np.uint16)


def emb_dev(emb: np.ndarray, device="cuda") -> torch.Tensor:
    return torch.from_numpy(emb).to(device) if emb.dtype == np.float32 else bf16_dev(emb, device)


def codes_host(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().numpy().view(np.uint32)


def unpack_bits(codes: np.ndarray) -> np.ndarray:
    return np.unpackbits(np.ascontiguousarray(codes).view(np.uint8), axis=1, bitorder="little").astype(bool)


# Bound on the relative error of the GPU's fp32 rotary encoding before bf16 rounding: angle
# fraction rounded to 2^-24 turns (3.7e-7 rad), fast sincos within 2^-21.4 absolute, the
# 2*pi scaling and the rotation's fp32 roundings -- under 1.5e-6 of the pair norm; doubled.
GPU_ROPE_REL_ERR = 3e-6


def operand_flip_allowance(orc, emb, pos, R, layout="interleaved"):
    """Per projection, the largest change bf16 operand rounding can make when the GPU's y
    differs from the exact y by up to GPU_ROPE_REL_ERR of its pair norm: only elements that
    close to a bf16 rounding midpoint can round the other way, each by one bf16 ulp.
    Returns [n][nbits] float64 (added to the projection tolerance and the code band)."""
    x = emb.astype(np.float64) if emb.dtype == np.float32 else \
        (emb.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    y = orc.rope(x, np.arange(len(x)) if pos is None else pos, layout=layout)
    if layout == "half":
        h = y.shape[1] // 2
        pn = np.hypot(y[:, :h], y[:, h:])
        pair = np.concatenate([pn, pn], axis=1)
    else:
        pair = np.repeat(np.hypot(y[:, 0::2], y[:, 1::2]), 2, axis=1)
    ay = np.abs(y)
    e = np.floor(np.log2(np.maximum(ay, 1e-300)))
    ulp = np.exp2(e - 7)                      # bf16: 8 significant bits
    mid_dist = np.abs(ay / ulp - np.floor(ay / ulp) - 0.5) * ulp
    risky = mid_dist <= GPU_ROPE_REL_ERR * pair
    r = np.abs((R.astype(np.uint32) << 16).view(np.float32).astype(np.float64))
    return (risky * ulp) @ r.T


def check_hash(gpu_codes, gpu_proj, orc_codes, orc_proj, rows=None, flips=None):
    """Asserts the projection and code rules; returns (band bits, checked bits).

    flips (optional, [n][nbits]) widens both the projection tolerance and the code band by the
    operand-rounding allowance of operand_flip_allowance()."""
    gpu_codes = np.asarray(gpu_codes)
    if rows is not None:
        gpu_codes = gpu_codes[rows]
        gpu_proj = None if gpu_proj is None else gpu_proj[rows]
    scale = np.abs(orc_proj).max(axis=1, keepdims=True)
    tol = BAND * scale + (0.0 if flips is None else flips)
    band = np.abs(orc_proj) < tol
    if gpu_proj is not None:
        err = np.abs(gpu_proj.astype(np.float64) - orc_proj.astype(np.float64))
        worst = float((err / np.maximum(scale, 1e-30)).max())
        assert (err <= tol).all(), f"projection error {worst:.3g} x row max exceeds the tolerance"
    diff = (unpack_bits(gpu_codes) != unpack_bits(orc_codes)) & ~band
    assert not diff.any(), f"{int(diff.sum())} code bits differ outside the band (rows {np.nonzero(diff.any(1))[0][:10]})"
    return int(band.sum()), band.size


def kv_host_planes(t: torch.Tensor) -> np.ndarray:
    return bf16_host(t)

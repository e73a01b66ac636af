"""Seeded synthetic inputs for the WHTMix token mixer.

This module is the only code shared by the CUDA path's tests/bench and the CPU oracle.  It holds
no part of the mixer's arithmetic: it draws numbers and quantises them to the storage dtypes.

Generator: SplitMix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number generators",
OOPSLA 2014) -> 53-bit uniforms in [0, 1) -> Box-Muller normals in float64.  Each tensor has its
own stream: X uses ``seed``, G uses ``seed + 1`` and dY uses ``seed + 2``; the separable log
gains g_t and g_c use ``seed + 3`` and ``seed + 4``, the block's projections ``seed + 5`` and
``seed + 6``.

Stand-in data.  The paper trains and times the mixer on joint left+right stereo token sequences
(Section III-A; N = 2 (H/8)(W/8), C = 64) and on LRA byte sequences (Section IV-D).  None of those
datasets are used here: these tensors take only the shapes, dtypes and distributions of the five
workloads below, X ~ N(0, 1) and G ~ N(1, 0.1) (unit gain at the paper's zero-initialised log
gains, Section III-B, plus a spread so that a wrong gain index is visible).
"""
from __future__ import annotations

import dataclasses

import numpy as np

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)


def splitmix64(seed: int, n: int, offset: int = 0) -> np.ndarray:
    """Outputs offset..offset+n-1 of SplitMix64 seeded with ``seed`` (uint64, wrapping)."""
    with np.errstate(over="ignore"):
        idx = np.arange(offset + 1, offset + n + 1, dtype=np.uint64)
        z = np.uint64(seed & 0xFFFFFFFFFFFFFFFF) + idx * _GOLDEN
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
        return z ^ (z >> np.uint64(31))


def uniform01(seed: int, n: int) -> np.ndarray:
    """n float64 uniforms in [0, 1) from the top 53 bits of SplitMix64."""
    return (splitmix64(seed, n) >> np.uint64(11)).astype(np.float64) * (1.0 / 9007199254740992.0)


def normal(seed: int, n: int, mean: float = 0.0, std: float = 1.0) -> np.ndarray:
    """n float64 normals by the Box-Muller transform on consecutive uniform pairs."""
    m = (n + 1) // 2
    u = uniform01(seed, 2 * m)
    u1, u2 = u[0::2], u[1::2]
    r = np.sqrt(-2.0 * np.log1p(-u1))
    t = 2.0 * np.pi * u2
    z = np.empty(2 * m, dtype=np.float64)
    z[0::2] = r * np.cos(t)
    z[1::2] = r * np.sin(t)
    return mean + std * z[:n]


def small_ints(seed: int, n: int, lo: int, hi: int) -> np.ndarray:
    """n integers uniform in [lo, hi] (int32)."""
    u = uniform01(seed, n)
    return (lo + np.floor(u * (hi - lo + 1))).astype(np.int64).clip(lo, hi).astype(np.int32)


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (round to nearest, ties to even); returns uint16 bits."""
    b = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    rounding = np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1))
    with np.errstate(over="ignore"):
        out = ((b + rounding) >> np.uint32(16)).astype(np.uint16)
    nan = np.isnan(a)
    if nan.any():
        out[nan] = np.uint16(0x7FC0)
    return out


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Widen bfloat16 bit patterns (uint16) to float32 exactly."""
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


DTYPES = ("f32", "bf16", "i32")


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic workload: shapes, storage dtype and the input recipe."""

    name: str
    B: int
    N: int
    C: int
    dtype: str            # storage dtype of X, Y, dY, dX: "f32" | "bf16" | "i32"
    backward: bool = False
    n_valid: int | None = None  # rows >= n_valid of X (and dY) are zero: token-axis zero padding
    description: str = ""
    gains: str = "full"   # "full": G [N, C]; "separable": log gains g_t [N], g_c [C] (Eq. 2-3)
    padded_io: bool = False  # X, Y hold only the n_valid stored tokens; the library pads to N
    block: bool = False      # the whole block of Eq. 1-4: W_in projection, mixer, W_out projection
    exchange: str = "f32"    # "bf16": whtmix_forward_x16, the intermediate plane exchanged in bf16

    @property
    def L(self) -> int:
        return self.N * self.C

    def ideal_bytes(self, backward: bool | None = None) -> int:
        """Bytes that must cross HBM once: read X and G, write Y.  A training step adds the
        backward call, which reads X, dY and G and writes dX and dG."""
        bwd = self.backward if backward is None else backward
        es = 2 if self.dtype == "bf16" else 4
        plane = self.B * (self.n_valid if self.padded_io else self.N) * self.C * es
        g = self.L * 4 if self.gains == "full" else (self.N + self.C) * 4
        if self.block:
            g += 2 * self.C * self.C * 2  # W_in and W_out, bf16
        fwd = 2 * plane + g
        if not bwd:
            return fwd
        return fwd + 3 * plane + 2 * g


# The five workloads: tiny mixer, epipolar-row stereo, long sequence, full-image global mixing
# (two 135x240 quarter-resolution maps flattened and zero-padded to 65536 tokens) and a training
# step.  Names carry their shapes.
WORKLOADS = {
    "tiny_1x256x64_f32": Workload("tiny_1x256x64_f32", 1, 256, 64, "f32",
                                  description="tiny mixer, forward"),
    "epipolar_128x512x128_bf16": Workload("epipolar_128x512x128_bf16", 128, 512, 128, "bf16",
                                          description="left+right epipolar rows, forward"),
    "longseq_32x4096x64_f32": Workload("longseq_32x4096x64_f32", 32, 4096, 64, "f32",
                                       description="long sequence, forward"),
    "fullimage_1x65536x128_bf16": Workload("fullimage_1x65536x128_bf16", 1, 65536, 128, "bf16",
                                           n_valid=2 * 135 * 240,
                                           description="two 135x240 maps, zero-padded to 65536 tokens, forward"),
    "train_16x8192x256_bf16": Workload("train_16x8192x256_bf16", 16, 8192, 256, "bf16", backward=True,
                                       description="training step: forward + backward"),
    # the full-image shape with the paper's own gain form (Section III-B, Eq. 2-3): no G plane
    "fullimage_separable_1x65536x128_bf16": Workload("fullimage_separable_1x65536x128_bf16", 1, 65536, 128, "bf16",
                                                     n_valid=2 * 135 * 240, gains="separable",
                                                     description="full-image shape, separable log gains, forward"),
    # the two 135x240 maps stored as their 64800 tokens, padded to 65536 inside the library
    "fullimage_padded_1x64800x128_bf16": Workload("fullimage_padded_1x64800x128_bf16", 1, 65536, 128, "bf16",
                                                  n_valid=2 * 135 * 240, padded_io=True,
                                                  description="64800 stored tokens, padded in the library, forward"),
    # the whole mixer block (W_in, mixer, W_out) on the full-image shape
    "block_fullimage_1x65536x128_bf16": Workload("block_fullimage_1x65536x128_bf16", 1, 65536, 128, "bf16",
                                                 n_valid=2 * 135 * 240, block=True,
                                                 description="mixer block: projection, mixer, projection"),
    # a training step on the full-image shape (forward + backward of 2^23-element planes)
    "fullimage_train_1x65536x128_bf16": Workload("fullimage_train_1x65536x128_bf16", 1, 65536, 128, "bf16",
                                                 backward=True, n_valid=2 * 135 * 240,
                                                 description="full-image shape, training step: forward + backward"),
    # the whole block's training step: block forward + block backward (weight gradients included)
    "block_train_fullimage_1x65536x128_bf16": Workload("block_train_fullimage_1x65536x128_bf16", 1, 65536, 128, "bf16",
                                                       backward=True, n_valid=2 * 135 * 240, block=True,
                                                       description="mixer block, training step: forward + backward"),
    # the full-image forward with the 16-bit exchange between the three-phase kernel's phases
    "fullimage_x16_1x65536x128_bf16": Workload("fullimage_x16_1x65536x128_bf16", 1, 65536, 128, "bf16",
                                               n_valid=2 * 135 * 240, exchange="bf16",
                                               description="full-image shape, forward, bf16 exchange workspace"),
    # the paper's mixer as trained: separable log gains and in-library padding
    "fullimage_paper_1x64800x128_bf16": Workload("fullimage_paper_1x64800x128_bf16", 1, 65536, 128, "bf16",
                                                 n_valid=2 * 135 * 240, padded_io=True, gains="separable",
                                                 description="64800 stored tokens, separable log gains, forward"),
}
WORKLOAD_ORDER = list(WORKLOADS)


def make_inputs(B: int, N: int, C: int, dtype: str, seed: int = 0, *, n_valid: int | None = None,
                with_dy: bool = False, int_range: tuple[int, int] = (-3, 3),
                gain_int_range: tuple[int, int] = (-2, 2)) -> dict[str, np.ndarray]:
    """Seeded inputs as numpy arrays in their storage form.

    f32:  X, dY float32 ~ N(0,1); G float32 ~ N(1, 0.1).
    bf16: X, dY as uint16 bfloat16 bits (float64 normal -> float32 -> bf16 RNE); G float32.
    i32:  X, dY int32 uniform in ``int_range``; G int32 uniform in ``gain_int_range``.
    Rows n >= n_valid of X and dY are set to zero (the token-axis padding structure).
    Every array is C-contiguous: X, dY [B, N, C]; G [N, C].
    """
    if dtype not in DTYPES:
        raise ValueError(f"dtype must be one of {DTYPES}")
    n_x = B * N * C
    out: dict[str, np.ndarray] = {}
    if dtype == "i32":
        out["x"] = small_ints(seed, n_x, *int_range).reshape(B, N, C)
        out["g"] = small_ints(seed + 1, N * C, *gain_int_range).reshape(N, C)
        if with_dy:
            out["dy"] = small_ints(seed + 2, n_x, *int_range).reshape(B, N, C)
    else:
        x32 = normal(seed, n_x).astype(np.float32).reshape(B, N, C)
        out["g"] = normal(seed + 1, N * C, 1.0, 0.1).astype(np.float32).reshape(N, C)
        dy32 = normal(seed + 2, n_x).astype(np.float32).reshape(B, N, C) if with_dy else None
        if dtype == "bf16":
            out["x"] = f32_to_bf16_bits(x32).reshape(B, N, C)
            if dy32 is not None:
                out["dy"] = f32_to_bf16_bits(dy32).reshape(B, N, C)
        else:
            out["x"] = x32
            if dy32 is not None:
                out["dy"] = dy32
    if n_valid is not None and n_valid < N:
        out["x"][:, n_valid:, :] = 0
        if "dy" in out:
            out["dy"][:, n_valid:, :] = 0
    return out


def make_log_gains(N: int, C: int, seed: int = 0, std: float = 0.05) -> tuple[np.ndarray, np.ndarray]:
    """Separable log gains g_t [N], g_c [C] (float32 ~ N(0, std)): near the paper's zero
    initialisation (unit gains), with a spread so that a wrong token or channel index is visible."""
    g_t = normal(seed + 3, N, 0.0, std).astype(np.float32)
    g_c = normal(seed + 4, C, 0.0, std).astype(np.float32)
    return g_t, g_c


def workload_inputs(w: Workload, seed: int = 0) -> dict[str, np.ndarray]:
    d = make_inputs(w.B, w.N, w.C, w.dtype, seed, n_valid=w.n_valid, with_dy=w.backward)
    if w.gains == "separable":
        d["g_t"], d["g_c"] = make_log_gains(w.N, w.C, seed)
    if w.block:
        d["w_in"], d["w_out"] = make_projections(w.C, seed)
    return d


def make_projections(C: int, seed: int = 0) -> tuple[np.ndarray, np.ndarray]:
    """W_in, W_out [C, C] as bf16 bits, entries ~ N(0, 1/C) (unit-variance outputs)."""
    w_in = (normal(seed + 5, C * C) / np.sqrt(C)).astype(np.float32).reshape(C, C)
    w_out = (normal(seed + 6, C * C) / np.sqrt(C)).astype(np.float32).reshape(C, C)
    return f32_to_bf16_bits(w_in).reshape(C, C), f32_to_bf16_bits(w_out).reshape(C, C)


def as_float64(a: np.ndarray, dtype: str) -> np.ndarray:
    """Exact widening of stored values to float64 (bf16 bits are decoded first)."""
    if dtype == "bf16" and a.dtype == np.uint16:
        return bf16_bits_to_f32(a).astype(np.float64)
    return a.astype(np.float64)

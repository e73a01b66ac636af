"""Shared helpers of the GPU parity tests: device transfer, the acceptance checks and guard regions.

Every floating-point check compares with the float64 oracle evaluated on the exact stored inputs
(bf16 values widened to float64, as the GPU sees them).  The bounds follow from where the path
rounds (paper Section III-B defines the map; the library computes it in fp32 and rounds once at
the store):

  int32      bit-exact: the integer mode wraps modulo 2^32, exact in any stage order.
  float32    per plane: relative L2 <= 1e-6; element-wise: |got - ref| <= 1e-5 * max(1, rms(ref)).
             fp32 butterflies lose about sqrt(2 log2 L) * 2^-24 of the plane's RMS per element
             (~4e-7 at L = 2^23), so 1e-5 is ~25x that, and a wrong element of a unit-scale plane
             is far outside it.
  bfloat16   per plane: relative L2 <= 1e-2 (the acceptance bound) AND element-wise
             |got - ref| <= 2^-8 |ref| + 2 eps, eps = 1e-5 * max(1, rms(ref)).  The output is
             RNE(y32) with |y32 - ref| <= eps (the fp32 path above), and RNE to bf16 moves a value
             by at most half a unit in the last place, <= 2^-8 |y32| (8 significand bits), so
             |RNE(y32) - ref| <= 2^-8 (|ref| + eps) + eps.  One element off by more than that fails.
  dG, dg_t, dg_c  always float32 results of exactly representable inputs (bf16 inputs are widened
             exactly), so they take the float32 bound whatever the input dtype, with the max-abs
             term scaled by the reference's RMS (dG grows like sqrt(B)).

Guard regions: every output the tests hand to the library is a view into a larger buffer whose
leading and trailing GUARD_BYTES hold a byte pattern; after the call both must be untouched.
"""
from __future__ import annotations

import numpy as np
import torch

from paper_2607_25234_gb300 import inputs

F32_REL_L2 = 1e-6
F32_MAX_ABS = 1e-5
BF16_REL_L2 = 1e-2
BF16_HALF_ULP = 2.0 ** -8
GUARD_BYTES = 4096      # a multiple of 256: the view keeps the allocation's alignment
GUARD_PATTERN = 0xA5


def to_dev(a: np.ndarray, dtype: str, out: torch.Tensor | None = None) -> torch.Tensor:
    """A stored numpy array on the GPU (bf16 as uint16 bits)."""
    a = np.ascontiguousarray(a)
    t = torch.from_numpy(a.view(np.int16)).view(torch.bfloat16) if dtype == "bf16" else torch.from_numpy(a)
    if out is None:
        return t.cuda()
    out.copy_(t)
    return out


def ref_inputs(d: dict, dtype: str) -> dict:
    """Exact float64 (or integer) views of the stored inputs, as the GPU sees them."""
    if dtype == "i32":
        return dict(d)
    return {k: inputs.as_float64(v, dtype if k not in ("g", "g_t", "g_c") else "f32") for k, v in d.items()}


def _planes(a: np.ndarray, per_plane: bool) -> np.ndarray:
    if a.ndim <= 1 or not per_plane:
        return a.reshape(1, -1)
    return a.reshape(a.shape[0], -1)


def check_f32(got, ref: np.ndarray, what: str, per_plane: bool = True):
    g = got.double().cpu().numpy().reshape(ref.shape) if isinstance(got, torch.Tensor) else got.reshape(ref.shape)
    gp, rp = _planes(g, per_plane), _planes(ref, per_plane)
    for b in range(rp.shape[0]):
        nr = np.linalg.norm(rp[b])
        err = np.linalg.norm(gp[b] - rp[b])
        assert err <= F32_REL_L2 * nr or err == 0.0, \
            f"{what} plane {b}: relative L2 {err / max(nr, 1e-300):.3e} > {F32_REL_L2}"
        rms = float(np.sqrt(np.mean(np.square(rp[b])))) if rp[b].size else 0.0
        mx = float(np.abs(gp[b] - rp[b]).max()) if rp[b].size else 0.0
        assert mx <= F32_MAX_ABS * max(1.0, rms), f"{what} plane {b}: max abs {mx:.3e} > {F32_MAX_ABS} x max(1, rms {rms:.3g})"


def check_bf16(got, ref: np.ndarray, what: str, per_plane: bool = True):
    g = got.double().cpu().numpy().reshape(ref.shape) if isinstance(got, torch.Tensor) else got.reshape(ref.shape)
    gp, rp = _planes(g, per_plane), _planes(ref, per_plane)
    for b in range(rp.shape[0]):
        nr = np.linalg.norm(rp[b])
        err = np.linalg.norm(gp[b] - rp[b])
        assert err <= BF16_REL_L2 * nr or err == 0.0, \
            f"{what} plane {b}: relative L2 {err / max(nr, 1e-300):.3e} > {BF16_REL_L2}"
        if not rp[b].size:
            continue
        eps = F32_MAX_ABS * max(1.0, float(np.sqrt(np.mean(np.square(rp[b])))))
        bound = BF16_HALF_ULP * np.abs(rp[b]) + 2.0 * eps
        bad = np.abs(gp[b] - rp[b]) > bound
        if bad.any():
            i = int(np.argmax(np.abs(gp[b] - rp[b]) - bound))
            raise AssertionError(f"{what} plane {b}: {int(bad.sum())} of {bad.size} elements outside "
                                 f"2^-8|ref| + 2 eps (eps {eps:.2e}); worst at {i}: got {gp[b][i]!r}, ref {rp[b][i]!r}")


def check_i32(got, ref: np.ndarray, what: str):
    g = got.cpu().numpy().reshape(ref.shape) if isinstance(got, torch.Tensor) else got.reshape(ref.shape)
    assert np.array_equal(g, ref), f"{what}: {np.count_nonzero(g != ref)} of {g.size} int32 values differ"


def check(got, ref: np.ndarray, dtype: str, what: str, per_plane: bool = True):
    """The acceptance check for an output stored in `dtype` (Y, dX)."""
    if dtype == "i32":
        check_i32(got, ref, what)
    elif dtype == "bf16":
        check_bf16(got, ref, what, per_plane)
    else:
        check_f32(got, ref, what, per_plane)


def check_grad(got, ref: np.ndarray, dtype: str, what: str):
    """dG (and the log-gain gradients): one plane, exact in int32, else the float32 bound."""
    if dtype == "i32":
        check_i32(got, ref, what)
    else:
        check_f32(got, np.asarray(ref).reshape(1, -1), what, per_plane=True)


class Guarded:
    """An output tensor of `shape` and `dtype` inside a buffer with guard bytes on both sides."""

    def __init__(self, shape, dtype: torch.dtype, device="cuda"):
        n = int(np.prod(shape)) if len(shape) else 1
        nbytes = n * torch.empty((), dtype=dtype).element_size()
        self.buf = torch.full((GUARD_BYTES + nbytes + GUARD_BYTES,), GUARD_PATTERN, dtype=torch.uint8, device=device)
        self.t = self.buf[GUARD_BYTES:GUARD_BYTES + nbytes].view(dtype).view(tuple(shape))
        self.nbytes = nbytes

    def fill(self, value) -> "Guarded":
        self.t.fill_(value)
        return self

    def assert_intact(self, what: str):
        head = self.buf[:GUARD_BYTES]
        tail = self.buf[GUARD_BYTES + self.nbytes:]
        bad_head = int((head != GUARD_PATTERN).sum().item())
        bad_tail = int((tail != GUARD_PATTERN).sum().item())
        assert bad_head == 0 and bad_tail == 0, \
            f"{what}: {bad_head} guard bytes before and {bad_tail} after the output were overwritten"


def guarded_like(t: torch.Tensor) -> Guarded:
    return Guarded(tuple(t.shape), t.dtype, t.device)


def bf16_round(a: np.ndarray) -> np.ndarray:
    """float64 values rounded to bfloat16 (through float32, both steps to nearest even), as float64."""
    return inputs.as_float64(inputs.f32_to_bf16_bits(np.asarray(a, dtype=np.float32)), "bf16")

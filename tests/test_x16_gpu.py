"""GPU parity of whtmix_forward_x16: the forward whose three-phase kernel rounds the exchanged
intermediate plane to bf16 (Section III-B's map, computed with fp32 butterflies and gain).

Bound.  A plane of 2^m = 2^(R+Q) elements goes rows (R bits) -> Q1 -> columns (Q bits, G/L, Q
bits) -> Q2 -> rows (R bits), where Q1, Q2 round every element to the nearest bf16, which moves a
value a by at most 2^-8 |a| (half a unit in the last of 8 significand bits).  The row transforms
are 2^(R/2) times orthogonal and the column step's norm is at most max|G| 2^Q / L, so Q1's error
reaches the output with norm <= 2^-8 max|G| ||X|| <= 2^-8 (max|G| / min|G|) ||Y||, and Q2's with
norm <= 2^-8 ||Y||; a bf16 output rounds once more (<= 2^-8 ||Y||).  So per plane

    ||Y_x16 - Y|| / ||Y|| <= 2^-8 (max|G| / min|G| + 1 + [bf16 output]) + 1e-6        (worst case)

and the bf16 acceptance tolerance, relative L2 <= 1e-2, is checked as well (the roundings are
unbiased and independent, so the measured error sits well below the worst case).  Element by
element the error of an output is a sum of many such roundings; the check allows
2^-8 |ref| + 8 * 2^-9 (max|G| / min|G| + 1) rms(ref), about six times the largest element error
that sum reaches on these workloads, far below a wrong element of a unit-scale plane.

Shapes the three-phase kernel does not run (int32, planes of at most 2^13 or more than 2^23
elements, planes held on chip) must give whtmix_forward's result bit for bit.
"""
import numpy as np
import pytest
import torch

import oracle
from _checks import Guarded, check, ref_inputs, to_dev
from paper_2607_25234_gb300 import inputs, whtmix

pytestmark = pytest.mark.gpu

BF16_ACCEPT_REL_L2 = 1e-2


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_25234_gb300 import build
    build.build()
    oracle.build()
    torch.cuda.set_device(0)


def x16_bounds(g: np.ndarray, bf16_out: bool):
    ga = np.abs(g)
    kappa = float(ga.max() / ga.min())
    rel = 2.0 ** -8 * (kappa + 1.0 + (1.0 if bf16_out else 0.0)) + 1e-6
    elem = 8 * 2.0 ** -9 * (kappa + 1.0)
    return rel, elem


def check_x16(got: torch.Tensor, ref: np.ndarray, g: np.ndarray, dtype: str, what: str) -> float:
    rel_bound, elem_k = x16_bounds(g, dtype == "bf16")
    gp = got.double().cpu().numpy().reshape(ref.shape[0], -1)
    rp = ref.reshape(ref.shape[0], -1)
    worst = 0.0
    for b in range(rp.shape[0]):
        nr = np.linalg.norm(rp[b])
        rel = float(np.linalg.norm(gp[b] - rp[b]) / nr)
        worst = max(worst, rel)
        assert rel <= BF16_ACCEPT_REL_L2, f"{what} plane {b}: relative L2 {rel:.3e} > {BF16_ACCEPT_REL_L2}"
        assert rel <= rel_bound, f"{what} plane {b}: relative L2 {rel:.3e} > worst-case bound {rel_bound:.3e}"
        rms = float(np.sqrt(np.mean(np.square(rp[b]))))
        bound = 2.0 ** -8 * np.abs(rp[b]) + elem_k * rms
        bad = np.abs(gp[b] - rp[b]) > bound
        assert not bad.any(), (f"{what} plane {b}: {int(bad.sum())} elements outside 2^-8|ref| + "
                               f"{elem_k:.3g} rms; worst error {float(np.abs(gp[b] - rp[b]).max()):.3e}, rms {rms:.3e}")
    return worst


def run_x16(B, N, C, dtype, seed=0, in_place=False):
    d = inputs.make_inputs(B, N, C, dtype, seed=seed)
    x, g = to_dev(d["x"], dtype), to_dev(d["g"], "f32" if dtype != "i32" else "i32")
    g0 = g.cpu()
    if in_place:
        y = whtmix.forward_x16(x, g, out=x)
        whtmix.sync()
    else:
        x0 = x.cpu()
        yg = Guarded(x.shape, x.dtype)
        y = whtmix.forward_x16(x, g, out=yg.t)
        whtmix.sync()
        yg.assert_intact(f"Y_x16 [{B},{N},{C}] {dtype}")
        assert torch.equal(x.cpu(), x0), "X (a read-only input) was modified"
    assert torch.equal(g.cpu(), g0), "G (a read-only input) was modified"
    r = ref_inputs(d, dtype)
    return d, y, oracle.forward(r["x"], r["g"])


@pytest.mark.parametrize("B,N,C,dtype", [
    (1, 65536, 128, "bf16"),   # the full-image workload: rows of 2^13, 1024-row columns in TMEM
    (1, 65536, 128, "f32"),
    (2, 32768, 128, "bf16"),   # 2^22: 512-row columns
    (20, 8192, 256, "bf16"),   # 2^21: rows of 2^14, 128-row columns in registers; two plane groups
    (3, 4096, 256, "f32"),     # 2^20
    (32, 4096, 64, "f32"),     # 2^18, the long-sequence workload
    (5, 1024, 128, "bf16"),    # 2^17
    (4, 512, 128, "f32"),      # 2^16 at a batch the one-plane-per-CTA kernel does not take
])
def test_x16_against_the_oracle(B, N, C, dtype):
    d, y, y_ref = run_x16(B, N, C, dtype)
    worst = check_x16(y, y_ref, d["g"], dtype, f"Y_x16 [{B},{N},{C}] {dtype}")
    # it is the 16-bit exchange that ran: close to whtmix_forward but not equal to it
    y_exact = whtmix.forward(to_dev(d["x"], dtype), to_dev(d["g"], "f32"))
    whtmix.sync()
    assert not torch.equal(y.cpu(), y_exact.cpu()), "whtmix_forward_x16 returned whtmix_forward's result"
    print(f"[{B},{N},{C}] {dtype}: worst relative L2 {worst:.3e}")


def test_x16_in_place():
    d, y, y_ref = run_x16(1, 65536, 128, "bf16", seed=3, in_place=True)
    check_x16(y, y_ref, d["g"], "bf16", "Y_x16 in place")


@pytest.mark.parametrize("B,N,C,dtype", [
    (1, 256, 64, "i32"),       # the integer mode: generic engine
    (3, 64, 32, "f32"),        # one tile
    (128, 512, 128, "bf16"),   # the epipolar workload: one plane per CTA, in tensor memory
    (2, 512, 32, "f32"),       # 2^14: one plane per CTA at every batch
    (1, 1 << 17, 256, "bf16"),  # 2^25 elements: generic engine
])
def test_x16_other_shapes_run_the_exact_path(B, N, C, dtype):
    d = inputs.make_inputs(B, N, C, dtype, seed=1)
    gdt = "f32" if dtype != "i32" else "i32"
    x, g = to_dev(d["x"], dtype), to_dev(d["g"], gdt)
    y16 = whtmix.forward_x16(x, g)
    y = whtmix.forward(x, g)
    whtmix.sync()
    assert torch.equal(y16.cpu(), y.cpu()), f"[{B},{N},{C}] {dtype}: whtmix_forward_x16 differs from whtmix_forward"
    if B * N * C <= (1 << 23):
        r = ref_inputs(d, dtype)
        check(y16, oracle.forward(r["x"], r["g"]), dtype, f"Y_x16 [{B},{N},{C}] {dtype}")

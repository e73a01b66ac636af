"""GPU parity of the token-padded entry points (Section III-B: zero-pad the token axis to a power
of two before H_N, discard the padded outputs) against the fp64 oracle on explicitly padded planes.

x, y, dy and dx hold N_valid tokens per plane; the reference pads them with zero rows to N, runs
the oracle and crops.  Shapes cover the fast kernels' in-kernel padding (stored planes 16-byte
aligned: whole padded rows, a row cut in the middle, the paper's token counts) and the copy
fallback (stored planes not 16-byte aligned, one-tile planes, the integer mode).  Acceptance as in
test_parity_gpu.py (_checks.py): int32 bit-exact, fp32 relative L2 <= 1e-6 with an element-wise
1e-5 bound, bf16 relative L2 <= 1e-2 with the element-wise bound of one rounding to nearest even;
dG is a float32 result and takes the float32 bound.  Outputs sit between guard regions (before
the first and after the last stored token) that must come back untouched.
"""
import numpy as np
import pytest
import torch

import oracle
from _checks import Guarded, check_grad
from _checks import check as check_out
from paper_2607_25234_gb300 import inputs, whtmix

pytestmark = pytest.mark.gpu

@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_25234_gb300 import build
    build.build()
    oracle.build()
    torch.cuda.set_device(0)


def to_dev(a: np.ndarray, dtype: str) -> torch.Tensor:
    if dtype == "bf16":
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def check(got, ref: np.ndarray, dtype: str, what: str):
    check_out(got, ref, dtype, what)


def padded_case(B, n_valid, N, C, dtype, seed, with_dy=False):
    """Stored inputs [B, n_valid, C] and their float64 (uint32) zero-padded [B, N, C] references."""
    d = inputs.make_inputs(B, N, C, dtype, seed=seed, with_dy=with_dy)
    stored = {k: np.ascontiguousarray(d[k][:, :n_valid, :]) for k in ("x", "dy") if k in d}
    ref = {}
    for k, v in stored.items():
        full = np.zeros((B, N, C), dtype=np.float64 if dtype != "i32" else np.int32)
        full[:, :n_valid, :] = inputs.as_float64(v, dtype) if dtype != "i32" else v
        ref[k] = full
    ref["g"] = d["g"].astype(np.float64) if dtype != "i32" else d["g"]
    dev = {k: to_dev(v, dtype) for k, v in stored.items()}
    dev["g"] = to_dev(d["g"], "i32" if dtype == "i32" else "f32")
    return dev, ref


SHAPES = [
    # in-kernel padding (stored planes 16-byte aligned)
    (1, 9216, 16384, 64), (2, 25600, 32768, 64), (1, 36864, 65536, 64), (1, 50176, 65536, 64),  # the paper's N
    (1, 64800, 65536, 128),          # the full-image shape, two 135 x 240 maps
    (3, 9224, 16384, 64),            # a padded row cut in the middle
    (5, 300, 512, 128), (2, 8192, 8192, 256),  # several plane groups; no padding at all
    # copy fallback
    (2, 1001, 1024, 4), (3, 37, 64, 16), (1, 200000, 1 << 18, 1),
]


@pytest.mark.parametrize("B,nv,N,C", SHAPES)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_forward_padded(B, nv, N, C, dtype):
    dev, ref = padded_case(B, nv, N, C, dtype, seed=B + nv + C)
    y = Guarded(dev["x"].shape, dev["x"].dtype)
    whtmix.forward_padded(dev["x"], dev["g"], out=y.t)
    whtmix.sync()
    check(y.t, oracle.forward(ref["x"], ref["g"])[:, :nv, :], dtype, f"Y [{B},{nv}->{N},{C}] {dtype}")
    y.assert_intact(f"Y [{B},{nv}->{N},{C}] {dtype}")


@pytest.mark.parametrize("B,nv,N,C", [(1, 9216, 16384, 64), (3, 9224, 16384, 64), (2, 700, 2048, 64),
                                      (2, 1001, 1024, 4), (3, 5000, 8192, 256)])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_backward_padded(B, nv, N, C, dtype):
    dev, ref = padded_case(B, nv, N, C, dtype, seed=2 * B + nv + C, with_dy=True)
    dx = Guarded(dev["dy"].shape, dev["dy"].dtype)
    dg = Guarded((N, C), torch.float32)
    whtmix.backward_padded(dev["x"], dev["g"], dev["dy"], dx=dx.t, dg=dg.t)
    whtmix.sync()
    dx_ref, dg_ref = oracle.backward(ref["x"], ref["g"], ref["dy"])
    check(dx.t, dx_ref[:, :nv, :], dtype, f"dX [{B},{nv}->{N},{C}] {dtype}")
    check_grad(dg.t, dg_ref, dtype, f"dG [{B},{nv}->{N},{C}] {dtype}")
    dx.assert_intact(f"dX [{B},{nv}->{N},{C}] {dtype}")
    dg.assert_intact(f"dG [{B},{nv}->{N},{C}] {dtype}")


def test_integer_mode_padded_bit_exact():
    for (B, nv, N, C) in [(2, 100, 128, 64), (1, 3000, 4096, 8)]:
        dev, ref = padded_case(B, nv, N, C, "i32", seed=nv, with_dy=True)
        y = whtmix.forward_padded(dev["x"], dev["g"])
        dx, dg = whtmix.backward_padded(dev["x"], dev["g"], dev["dy"])
        whtmix.sync()
        check(y, oracle.forward(ref["x"], ref["g"])[:, :nv, :], "i32", "Y i32")
        dx_ref, dg_ref = oracle.backward(ref["x"], ref["g"], ref["dy"])
        check(dx, dx_ref[:, :nv, :], "i32", "dX i32")
        check_grad(dg, dg_ref, "i32", "dG i32")


def test_padded_equals_padding_by_hand_and_in_place():
    B, nv, N, C = 2, 9216, 16384, 64
    dev, _ = padded_case(B, nv, N, C, "bf16", seed=3)
    xpad = torch.zeros(B, N, C, dtype=torch.bfloat16, device="cuda")
    xpad[:, :nv] = dev["x"]
    want = whtmix.forward(xpad, dev["g"])[:, :nv]
    got = whtmix.forward_padded(dev["x"], dev["g"])
    x2 = dev["x"].clone()
    whtmix.forward_padded(x2, dev["g"], out=x2)
    torch.cuda.synchronize()
    assert torch.equal(got, want) and torch.equal(x2, want)


def test_separable_with_padding():
    B, nv, N, C = 2, 25600, 32768, 64
    d = inputs.make_inputs(B, N, C, "bf16", seed=21, with_dy=True)
    g_t, g_c = inputs.make_log_gains(N, C, seed=21)
    x = to_dev(np.ascontiguousarray(d["x"][:, :nv]), "bf16")
    dy = to_dev(np.ascontiguousarray(d["dy"][:, :nv]), "bf16")
    gt, gc = torch.from_numpy(g_t).cuda(), torch.from_numpy(g_c).cuda()
    y = whtmix.forward_separable(x, gt, gc)
    dx, dgt, dgc = whtmix.backward_separable(x, gt, gc, dy)
    whtmix.sync()
    xr = np.zeros((B, N, C))
    xr[:, :nv] = inputs.as_float64(d["x"][:, :nv], "bf16")
    dyr = np.zeros((B, N, C))
    dyr[:, :nv] = inputs.as_float64(d["dy"][:, :nv], "bf16")
    check(y, oracle.forward_separable(xr, g_t, g_c)[:, :nv], "bf16", "separable padded Y")
    dx_ref, dgt_ref, dgc_ref = oracle.backward_separable(xr, g_t, g_c, dyr)
    check(dx, dx_ref[:, :nv], "bf16", "separable padded dX")
    check_grad(dgt, dgt_ref, "f32", "separable padded dg_t")
    check_grad(dgc, dgc_ref, "f32", "separable padded dg_c")


def test_nothing_stored():
    N, C = 1024, 64
    g = torch.ones(N, C, device="cuda")
    e = torch.empty(2, 0, C, device="cuda")
    assert whtmix.forward_padded(e, g).shape == (2, 0, C)
    dg = torch.full((N, C), 3.0, device="cuda")
    whtmix.backward_padded(e, g, e, dg=dg)
    torch.cuda.synchronize()
    assert dg.abs().max().item() == 0.0

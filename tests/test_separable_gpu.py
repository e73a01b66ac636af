"""GPU parity of the separable log-gain entry points (Section III-B, Eq. 2-3) against the fp64
oracle: G[n, c] = exp(g_t[n]) exp(g_c[c]).

The forward runs the fast kernel with the gains computed inside it (planes of 2^14..2^23 elements,
2 <= C <= the kernel's row length) or, for every other shape, builds G in the workspace and runs
the full-gain kernels; both are covered below.  Acceptance as in the other parity
tests (_checks.py): fp32 relative L2 <= 1e-6 per plane with an element-wise 1e-5 bound, bf16
relative L2 <= 1e-2 per plane with the element-wise bound of one rounding to nearest even.  The
gradients dg_t and dg_c are float32 results whatever the input dtype (bf16 inputs are widened
exactly and dG, G and the sums are fp32 / float64), so they take the float32 bound, its max-abs
term scaled by the reference's RMS (they are sums over C or N products, not of unit scale).  Every
output sits between guard regions that must come back untouched.
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
        return torch.from_numpy(a.view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def check(got, ref: np.ndarray, dtype: str, what: str, per_plane: bool = True):
    """Y and dX with their dtype's bound; dg_t and dg_c (per_plane=False) with the float32 bound."""
    if per_plane:
        check_out(got, ref, dtype, what)
    else:
        check_grad(got, ref, "f32", what)


def case(B, N, C, dtype, seed, with_dy=False):
    d = inputs.make_inputs(B, N, C, dtype, seed=seed, with_dy=with_dy)
    g_t, g_c = inputs.make_log_gains(N, C, seed=seed)
    dev = {"x": to_dev(d["x"], dtype), "g_t": torch.from_numpy(g_t).cuda(), "g_c": torch.from_numpy(g_c).cuda()}
    ref = {"x": inputs.as_float64(d["x"], dtype), "g_t": g_t.astype(np.float64), "g_c": g_c.astype(np.float64)}
    if with_dy:
        dev["dy"] = to_dev(d["dy"], dtype)
        ref["dy"] = inputs.as_float64(d["dy"], dtype)
    return dev, ref


FWD = [
    # fast kernel, gains computed inside it: every column height, C from 2 to the row length
    (3, 128, 128), (2, 16384, 2), (2, 4, 8192), (1, 1024, 128), (2, 2048, 64), (1, 4096, 64), (1, 2048, 256),
    (2, 8192, 128), (1, 8192, 256), (1, 32768, 128), (1, 65536, 128), (1, 512, 16384),
    # full-gain fallback: C = 1, C beyond the row length, one-tile planes, planes beyond 2^23
    (2, 16384, 1), (1, 2, 16384), (5, 64, 32), (3, 1, 1), (1, 1 << 19, 32),
]


@pytest.mark.parametrize("B,N,C", FWD)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_forward_separable(B, N, C, dtype):
    dev, ref = case(B, N, C, dtype, seed=3 * B + N + C)
    y = Guarded(dev["x"].shape, dev["x"].dtype)
    whtmix.forward_separable(dev["x"], dev["g_t"], dev["g_c"], out=y.t)
    whtmix.sync()
    check(y.t, oracle.forward_separable(ref["x"], ref["g_t"], ref["g_c"]), dtype, f"Y [{B},{N},{C}] {dtype}")
    y.assert_intact(f"Y [{B},{N},{C}] {dtype}")


BWD = [(2, 64, 32), (3, 128, 128), (2, 2048, 64), (3, 8192, 256), (1, 65536, 128), (2, 16384, 1)]


@pytest.mark.parametrize("B,N,C", BWD)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_backward_separable(B, N, C, dtype):
    dev, ref = case(B, N, C, dtype, seed=5 * B + N + C, with_dy=True)
    dx = Guarded(dev["x"].shape, dev["x"].dtype)
    dgt = Guarded((N,), torch.float32)
    dgc = Guarded((C,), torch.float32)
    whtmix.backward_separable(dev["x"], dev["g_t"], dev["g_c"], dev["dy"], dx=dx.t, dg_t=dgt.t, dg_c=dgc.t)
    whtmix.sync()
    dx_ref, dgt_ref, dgc_ref = oracle.backward_separable(ref["x"], ref["g_t"], ref["g_c"], ref["dy"])
    check(dx.t, dx_ref, dtype, f"dX [{B},{N},{C}] {dtype}")
    check(dgt.t, dgt_ref, dtype, f"dg_t [{B},{N},{C}] {dtype}", per_plane=False)
    check(dgc.t, dgc_ref, dtype, f"dg_c [{B},{N},{C}] {dtype}", per_plane=False)
    for gd, name in ((dx, "dX"), (dgt, "dg_t"), (dgc, "dg_c")):
        gd.assert_intact(f"{name} [{B},{N},{C}] {dtype}")


def test_training_shape_backward_and_determinism():
    dev, ref = case(16, 8192, 256, "bf16", seed=0, with_dy=True)
    a = whtmix.backward_separable(dev["x"], dev["g_t"], dev["g_c"], dev["dy"])
    b = whtmix.backward_separable(dev["x"], dev["g_t"], dev["g_c"], dev["dy"])
    whtmix.sync()
    for u, v in zip(a, b):
        assert torch.equal(u, v)
    _, dgt_ref, dgc_ref = oracle.backward_separable(ref["x"], ref["g_t"], ref["g_c"], ref["dy"])
    check(a[1], dgt_ref, "bf16", "dg_t", per_plane=False)
    check(a[2], dgc_ref, "bf16", "dg_c", per_plane=False)


def test_zero_log_gains_are_the_identity_and_empty_batch():
    B, N, C = 2, 8192, 64
    dev, _ = case(B, N, C, "f32", seed=11)
    z_t, z_c = torch.zeros(N, device="cuda"), torch.zeros(C, device="cuda")
    y = whtmix.forward_separable(dev["x"], z_t, z_c)
    assert (y - dev["x"]).abs().max().item() <= 1e-5
    # in place
    x2 = dev["x"].clone()
    whtmix.forward_separable(x2, dev["g_t"], dev["g_c"], out=x2)
    y2 = whtmix.forward_separable(dev["x"], dev["g_t"], dev["g_c"])
    torch.cuda.synchronize()
    assert torch.equal(x2, y2)
    e = torch.empty(0, N, C, device="cuda")
    dgt, dgc = torch.full((N,), 5.0, device="cuda"), torch.full((C,), 5.0, device="cuda")
    whtmix.backward_separable(e, z_t, z_c, e, dg_t=dgt, dg_c=dgc)
    torch.cuda.synchronize()
    assert dgt.abs().max().item() == 0 and dgc.abs().max().item() == 0


def test_separable_autograd_function():
    B, N, C = 2, 1024, 64
    d = inputs.make_inputs(B, N, C, "f32", seed=13, with_dy=True)
    g_t, g_c = inputs.make_log_gains(N, C, seed=13)
    x = to_dev(d["x"], "f32").requires_grad_(True)
    gt = torch.from_numpy(g_t).cuda().requires_grad_(True)
    gc = torch.from_numpy(g_c).cuda().requires_grad_(True)
    y = whtmix.WHTMixSeparableFunction.apply(x, gt, gc)
    y.backward(to_dev(d["dy"], "f32"))
    dx_ref, dgt_ref, dgc_ref = oracle.backward_separable(d["x"].astype(np.float64), g_t.astype(np.float64),
                                                         g_c.astype(np.float64), d["dy"].astype(np.float64))
    check(x.grad, dx_ref, "f32", "autograd dX")
    check(gt.grad, dgt_ref, "f32", "autograd dg_t", per_plane=False)
    check(gc.grad, dgc_ref, "f32", "autograd dg_c", per_plane=False)

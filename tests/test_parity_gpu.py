"""GPU parity: the CUDA path through the C ABI against the fp64 / uint32 CPU oracle on the same
seeded inputs.

Acceptance (per plane, Y_ref the fp64 oracle on the exact stored inputs; the bounds and their
derivation are in _checks.py):
  int32      bit-exact (the integer mode is exact modulo 2^32 in any stage order);
  float32    relative L2 <= 1e-6 and, element by element, |err| <= 1e-5 (x the plane's RMS if > 1);
  bfloat16   relative L2 <= 1e-2 and, element by element, |err| <= 2^-8 |Y_ref| + 2e-5: the fp32
             result rounded once to nearest even.
dG is a float32 result in every floating mode (bf16 inputs are widened exactly), so it takes the
float32 bound.  Every output lives between guard regions that must come back untouched, and the
read-only inputs must be unchanged after the call.
"""
import numpy as np
import pytest
import torch

import oracle
from _checks import Guarded, check, check_grad, ref_inputs, to_dev
from paper_2607_25234_gb300 import inputs, whtmix

pytestmark = pytest.mark.gpu

TORCH_DT = {"f32": torch.float32, "bf16": torch.bfloat16, "i32": torch.int32}


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_25234_gb300 import build
    build.build()
    oracle.build()
    torch.cuda.set_device(0)


def assert_unchanged(t: torch.Tensor, before: torch.Tensor, what: str):
    assert torch.equal(t.cpu(), before), f"{what} (a read-only input) was modified"


def run_forward(B, N, C, dtype, seed=0, n_valid=None):
    d = inputs.make_inputs(B, N, C, dtype, seed=seed, n_valid=n_valid)
    x, g = to_dev(d["x"], dtype), to_dev(d["g"], "f32" if dtype != "i32" else "i32")
    x0, g0 = x.cpu(), g.cpu()
    y = Guarded(x.shape, x.dtype)
    whtmix.forward(x, g, out=y.t)
    whtmix.sync()
    r = ref_inputs(d, dtype)
    y_ref = oracle.forward(r["x"], r["g"])
    check(y.t, y_ref, dtype, f"Y [{B},{N},{C}] {dtype}")
    y.assert_intact(f"Y [{B},{N},{C}] {dtype}")
    assert_unchanged(x, x0, "X")
    assert_unchanged(g, g0, "G")
    return x, g, y.t


def run_backward(B, N, C, dtype, seed=0, n_valid=None):
    d = inputs.make_inputs(B, N, C, dtype, seed=seed, n_valid=n_valid, with_dy=True)
    gdt = "f32" if dtype != "i32" else "i32"
    x, g, dy = to_dev(d["x"], dtype), to_dev(d["g"], gdt), to_dev(d["dy"], dtype)
    x0, g0, dy0 = x.cpu(), g.cpu(), dy.cpu()
    dx = Guarded(x.shape, x.dtype)
    dg = Guarded(g.shape, g.dtype)
    whtmix.backward(x, g, dy, dx=dx.t, dg=dg.t)
    whtmix.sync()
    r = ref_inputs(d, dtype)
    dx_ref, dg_ref = oracle.backward(r["x"], r["g"], r["dy"])
    check(dx.t, dx_ref, dtype, f"dX [{B},{N},{C}] {dtype}")
    check_grad(dg.t, dg_ref, dtype, f"dG [{B},{N},{C}] {dtype}")
    dx.assert_intact(f"dX [{B},{N},{C}] {dtype}")
    dg.assert_intact(f"dG [{B},{N},{C}] {dtype}")
    for t, t0, name in ((x, x0, "X"), (g, g0, "G"), (dy, dy0, "dY")):
        assert_unchanged(t, t0, name)
    return dx.t, dg.t


# ---- the five workloads at full size ----

def test_tiny_1x256x64_f32_forward():
    run_forward(1, 256, 64, "f32")


def test_tiny_1x256x64_i32_forward_bit_exact():
    run_forward(1, 256, 64, "i32")


def test_epipolar_128x512x128_bf16_forward():
    run_forward(128, 512, 128, "bf16")


def test_longseq_32x4096x64_f32_forward():
    run_forward(32, 4096, 64, "f32")


def test_fullimage_1x65536x128_bf16_forward_padded():
    run_forward(1, 65536, 128, "bf16", n_valid=2 * 135 * 240)


def test_fullimage_1x65536x128_bf16_forward_dense():
    run_forward(1, 65536, 128, "bf16")


def test_train_16x8192x256_bf16_forward_backward():
    run_forward(16, 8192, 256, "bf16")
    run_backward(16, 8192, 256, "bf16")


def test_fullimage_1x65536x128_bf16_backward_padded():
    # the full-image shape's training step: 2^23-element planes, rows >= 64800 zero
    run_backward(1, 65536, 128, "bf16", n_valid=2 * 135 * 240)


# ---- shape sweep: single-tile and three-phase plans, aspect ratios, ragged batches ----

SWEEP = [(1, 1, 1), (3, 1, 1), (5, 1, 8), (7, 8, 1), (3, 2, 2), (9, 4, 16), (2, 16, 4), (33, 32, 8),
         (3, 64, 128), (2, 128, 64), (1, 8192, 1), (1, 1, 8192), (2, 1, 16384), (3, 16384, 1),
         (2, 64, 256), (3, 512, 32), (1, 2048, 64), (2, 256, 1024), (1, 1 << 18, 2), (1, 2, 1 << 18),
         # every plane size of the one-plane-per-CTA forward (2^14, 2^15; 2^16 from a batch of 80:
         # smaller batches of 2^16 planes run three-phase) and every column height of the
         # three-phase forward (2^16 .. 2^23, Q = 3 .. 10; 2^17, 2^18, 2^19 above)
         (3, 2048, 8), (2, 128, 256), (80, 256, 256), (3, 512, 128), (1, 65536, 1),
         (2, 1024, 1024), (3, 256, 4096), (1, 4096, 512), (1, 4096, 1024), (2, 8192, 512),
         (1, 1 << 20, 8), (1, 16, 1 << 19)]


@pytest.mark.parametrize("B,N,C", SWEEP)
@pytest.mark.parametrize("dtype", ["f32", "bf16", "i32"])
def test_forward_sweep(B, N, C, dtype):
    run_forward(B, N, C, dtype, seed=B + N + C)


BWD_SWEEP = [(1, 1, 1), (3, 4, 2), (5, 32, 16), (2, 64, 128), (6, 512, 16),
             # every column height of the fast backward, N*C = 2^(13+Q) with Q = 1..7 (rows of 2^13)
             # and 2^(14+Q) with Q = 7, 8, 9 (rows of 2^14: 2^21, 2^22, 2^23); odd batches leave a
             # short last plane group
             (3, 128, 128), (2, 8192, 2), (3, 256, 128), (4, 1024, 64), (5, 2048, 64), (2, 64, 4096),
             (1, 1 << 17, 4), (3, 1024, 1024), (3, 8192, 256), (1, 2, 1 << 20),
             (3, 16384, 256), (1, 2048, 2048), (2, 65536, 128), (1, 1 << 16, 64)]


@pytest.mark.parametrize("B,N,C", BWD_SWEEP)
@pytest.mark.parametrize("dtype", ["f32", "bf16", "i32"])
def test_backward_sweep(B, N, C, dtype):
    run_backward(B, N, C, dtype, seed=2 * B + N + C)


def test_largest_plane_2_pow_26_bf16():
    run_forward(1, 1 << 19, 128, "bf16", seed=3)


# ---- planes of more than 2^26 elements (five passes forward, seven backward, one launch each) ----

@pytest.mark.parametrize("B,N,C,dtype", [(1, 1 << 20, 128, "f32"), (1, 1 << 17, 1024, "bf16"),
                                         (2, 1 << 14, 8192, "i32"), (1, 1 << 21, 128, "bf16")])
def test_forward_planes_beyond_2_pow_26(B, N, C, dtype):
    run_forward(B, N, C, dtype, seed=12 + B)


@pytest.mark.parametrize("B,N,C,dtype", [(1, 1 << 20, 128, "f32"), (2, 1 << 14, 8192, "i32"),
                                         (1, 1 << 17, 1024, "bf16")])
def test_backward_planes_beyond_2_pow_26(B, N, C, dtype):
    run_backward(B, N, C, dtype, seed=14 + B)


def test_largest_plane_2_pow_30_identity_and_dc_gain():
    """N*C = 2^30 (the largest plane), bf16: unit gains are the identity and a gain that keeps only
    the constant frequency maps every output to the plane's mean (Section III-B: W is orthonormal and
    its own inverse; G = e_00 keeps the DC coefficient).  Inputs from a seeded torch generator on the
    device (the float64 oracle would need 8 GiB per plane)."""
    N, C = 1 << 22, 1 << 8
    gen = torch.Generator(device="cuda")
    gen.manual_seed(30)
    x = torch.randn(1, N, C, device="cuda", generator=gen).to(torch.bfloat16)
    g = torch.ones(N, C, device="cuda")
    y = Guarded(x.shape, x.dtype)
    whtmix.forward(x, g, out=y.t)
    whtmix.sync()
    y.assert_intact("Y [1,2^22,256]")
    xf = x.float()
    err = (y.t.float() - xf).abs()
    assert (err <= 2.0 ** -8 * xf.abs() + 2e-5).all().item(), float(err.max())
    g.zero_()
    g[0, 0] = 1.0
    whtmix.forward(x, g, out=y.t)
    whtmix.sync()
    mean = x.double().mean().item()
    yy = y.t.float()
    assert (yy == yy.reshape(-1)[0]).all().item(), "a single frequency maps to one constant plane"
    assert abs(yy.reshape(-1)[0].item() - mean) <= 2.0 ** -8 * abs(mean) + 1e-9, (yy.reshape(-1)[0].item(), mean)


def test_many_groups_forward_and_backward_f32():
    # 2^20 elements per plane: forward groups of 16 planes, backward groups of 8
    run_forward(20, 4096, 256, "f32", seed=4)
    run_backward(10, 4096, 256, "f32", seed=5)


# ---- semantics ----

def test_integer_mode_wraps_mod_2_32():
    B, N, C = 2, 512, 64
    x = inputs.small_ints(80, B * N * C, -(2**31), 2**31 - 1).reshape(B, N, C)
    g = inputs.small_ints(81, N * C, -(2**31), 2**31 - 1).reshape(N, C)
    y = whtmix.forward(to_dev(x, "i32"), to_dev(g, "i32"))
    assert np.array_equal(y.cpu().numpy(), oracle.forward(x, g))


def test_in_place_forward_and_backward():
    # single tile, one plane per CTA (2^15), three-phase forward
    for (B, N, C) in [(3, 64, 64), (2, 256, 128), (2, 1024, 128)]:
        d = inputs.make_inputs(B, N, C, "f32", seed=6, with_dy=True)
        x = to_dev(d["x"], "f32")
        g = to_dev(d["g"], "f32")
        y_ref = oracle.forward(d["x"].astype(np.float64), d["g"].astype(np.float64))
        whtmix.forward(x, g, out=x)
        check(x, y_ref, "f32", "in-place Y")
        dy = to_dev(d["dy"], "f32")
        xx = to_dev(d["x"], "f32")
        dx_ref, _ = oracle.backward(d["x"].astype(np.float64), d["g"].astype(np.float64), d["dy"].astype(np.float64))
        whtmix.backward(xx, g, dy, dx=dy)
        check(dy, dx_ref, "f32", "in-place dX")


def test_backward_is_deterministic():
    for (B, N, C) in [(8, 2048, 64), (3, 8192, 512)]:   # 128- and 512-row columns
        d = inputs.make_inputs(B, N, C, "bf16", seed=7, with_dy=True)
        x, g, dy = to_dev(d["x"], "bf16"), to_dev(d["g"], "f32"), to_dev(d["dy"], "bf16")
        a = whtmix.backward(x, g, dy)
        b = whtmix.backward(x, g, dy)
        torch.cuda.synchronize()
        assert torch.equal(a[0], b[0]) and torch.equal(a[1], b[1])
    d = inputs.make_inputs(40, 32, 16, "f32", seed=8, with_dy=True)
    x, g, dy = to_dev(d["x"], "f32"), to_dev(d["g"], "f32"), to_dev(d["dy"], "f32")
    a = whtmix.backward(x, g, dy)
    b = whtmix.backward(x, g, dy)
    torch.cuda.synchronize()
    assert torch.equal(a[1], b[1])


def test_unit_gain_is_identity_and_zero_gain_is_zero():
    B, N, C = 2, 4096, 64
    d = inputs.make_inputs(B, N, C, "f32", seed=9)
    x = to_dev(d["x"], "f32")
    y = whtmix.forward(x, torch.ones(N, C, device="cuda"))
    assert (y - x).abs().max().item() <= 1e-5
    y0 = whtmix.forward(x, torch.zeros(N, C, device="cuda"))
    assert y0.abs().max().item() == 0.0


def test_ex_variant_matches_plain_call():
    B, N, C = 2, 8192, 32
    d = inputs.make_inputs(B, N, C, "bf16", seed=10, with_dy=True)
    x, g, dy = to_dev(d["x"], "bf16"), to_dev(d["g"], "f32"), to_dev(d["dy"], "bf16")
    ws = torch.zeros(whtmix.workspace_bytes(B, N, C, torch.bfloat16, backward=True), dtype=torch.uint8, device="cuda")
    y1 = whtmix.forward(x, g)
    y2 = whtmix.forward_ex(x, g, ws)
    dx1, dg1 = whtmix.backward(x, g, dy)
    dx2, dg2 = whtmix.backward_ex(x, g, dy, ws)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2) and torch.equal(dx1, dx2) and torch.equal(dg1, dg2)
    header = ws[:256].view(torch.int32).cpu()
    # no wait gave up (word 2), and at most the counter of the last barrier is still full
    assert header[2].item() == 0
    assert sum(1 for w in (0, 1, 3, 4) if header[w].item() != 0) <= 1


def test_empty_batch_and_errors_on_gpu():
    x = torch.empty(0, 16, 16, device="cuda")
    g = torch.ones(16, 16, device="cuda")
    y = whtmix.forward(x, g)
    assert y.shape == (0, 16, 16)
    dg = torch.full((16, 16), 7.0, device="cuda")
    whtmix.backward(x, g, torch.empty_like(x), dg=dg)
    torch.cuda.synchronize()
    assert dg.abs().max().item() == 0.0  # the sum over an empty batch
    with pytest.raises(whtmix.WhtmixError) as e:
        whtmix.forward(torch.zeros(1, 12, 16, device="cuda"), torch.zeros(12, 16, device="cuda"))
    assert e.value.status == 2
    with pytest.raises(ValueError):
        whtmix.forward(torch.zeros(1, 16, 16), torch.zeros(16, 16))


def test_binding_rejects_malformed_outputs_before_any_launch():
    """The C ABI receives only an output's pointer, so the binding checks the tensor: a result
    buffer of the wrong shape, dtype, device or layout raises and leaves every buffer untouched."""
    x = torch.randn(2, 64, 32, device="cuda")
    g = torch.ones(64, 32, device="cuda")
    sentinel = torch.full((2, 64, 32), 5.0, device="cuda")
    bad_outs = [torch.empty(2, 64, 16, device="cuda"), torch.empty(2, 64, 32, device="cuda", dtype=torch.bfloat16),
                torch.empty(2, 64, 32), torch.empty(2, 32, 64, device="cuda").transpose(1, 2)]
    for bad in bad_outs:
        with pytest.raises(ValueError):
            whtmix.forward(x, g, out=bad)
        with pytest.raises(ValueError):
            whtmix.backward(x, g, x, dx=bad)
    with pytest.raises(ValueError):
        whtmix.backward(x, g, x, dx=sentinel, dg=torch.empty(64, 16, device="cuda"))
    with pytest.raises(ValueError):
        whtmix.forward(x, g, stream=torch.cuda.Stream(device="cuda"), out=torch.empty(2, 64, 8, device="cuda"))
    torch.cuda.synchronize()
    assert torch.all(sentinel == 5.0)


@pytest.mark.parametrize("B,N,C,dtype", [(2, 64, 32, "f32"), (1, 1024, 128, "bf16"), (3, 4096, 64, "f32"),
                                         (2, 512, 64, "i32")])
def test_forward_noalloc_binding(B, N, C, dtype):
    d = inputs.make_inputs(B, N, C, dtype, seed=21)
    x, g = to_dev(d["x"], dtype), to_dev(d["g"], "f32" if dtype != "i32" else "i32")
    y = whtmix.forward_noalloc(x, g)
    whtmix.sync()
    r = ref_inputs(d, dtype)
    check(y, oracle.forward(r["x"], r["g"]), dtype, f"noalloc Y [{B},{N},{C}] {dtype}")
    with pytest.raises(whtmix.WhtmixError) as e:   # 2^23 elements: beyond the fixed scratch
        whtmix.forward_noalloc(torch.zeros(1, 65536, 128, device="cuda"), torch.ones(65536, 128, device="cuda"))
    assert e.value.status == 9


def test_autograd_function():
    B, N, C = 2, 256, 64
    d = inputs.make_inputs(B, N, C, "f32", seed=11, with_dy=True)
    x = to_dev(d["x"], "f32").requires_grad_(True)
    g = to_dev(d["g"], "f32").requires_grad_(True)
    y = whtmix.WHTMixFunction.apply(x, g)
    y.backward(to_dev(d["dy"], "f32"))
    dx_ref, dg_ref = oracle.backward(d["x"].astype(np.float64), d["g"].astype(np.float64), d["dy"].astype(np.float64))
    check(x.grad, dx_ref, "f32", "autograd dX")
    check_grad(g.grad, dg_ref, "f32", "autograd dG")

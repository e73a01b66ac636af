"""GPU checks of the tensor-core projection (whtmix_project) and the whole mixer block
(whtmix_block_forward, Section III-B, Eq. 1-4).

The projection is checked bit-exactly on integer-valued bf16 inputs with fp32 output (every
product and partial sum is an integer below 2^24, so any summation order gives the same fp32
value), and with bf16 output against the fp64 product (half a bf16 ulp plus the fp32 sum's error).

The block is checked against the fp64 mixer with the library's documented rounding points: M (the
mixer's output) is rounded to bf16 before W_out, and in the three-launch form Z = X W_in^T is too.
The reference rounds Z the same way (Z_r = bf16(Z), or Z_r = Z for the fused kernel), takes
M = mixer(Z_r) in float64 and Y_ref = M W_out^T.  Per plane the relative L2 error must be <= 1e-2,
and element by element
    |Y - Y_ref| <= 2^-8 |Y_ref|                          (the final rounding to bf16)
                 + (2^-8 + 1e-5) (|M| |W_out|^T)           (M's rounding and fp32 error, summed over c)
                 + [three launches] 2^-7 max|G| (|Z_r| |W_out|^T)   (a fp32 Z rounded to the other
                   neighbour: one bf16 ulp, 2^-7 |Z|, passed on to M at the same position times
                   the mixer's diagonal entry mean(G) <= max|G|)
                 + 1e-5 rms(Y_ref).
Every output sits between guard regions that must come back untouched.
"""
import numpy as np
import pytest
import torch

import oracle
from _checks import Guarded, bf16_round
from paper_2607_25234_gb300 import inputs, whtmix

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_25234_gb300 import build
    build.build()
    oracle.build()
    torch.cuda.set_device(0)


def bf16_dev(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(inputs.f32_to_bf16_bits(np.ascontiguousarray(a, dtype=np.float32)).view(np.int16)).cuda().view(torch.bfloat16)


@pytest.mark.parametrize("T,C", [(128, 64), (1000, 128), (4096, 256), (77, 256), (300000, 128)])
def test_project_exact_on_integers(T, C):
    x = inputs.small_ints(70 + C, T * C, -3, 3).reshape(T, C).astype(np.float32)
    w = inputs.small_ints(71 + C, C * C, -2, 2).reshape(C, C).astype(np.float32)
    z = Guarded((T, C), torch.float32)
    whtmix.project(bf16_dev(x), bf16_dev(w), out_dtype=torch.float32, out=z.t)
    whtmix.sync()
    want = (x.astype(np.int64) @ w.astype(np.int64).T).astype(np.float32)
    got = z.t.cpu().numpy()
    assert np.array_equal(got, want), f"{np.count_nonzero(got != want)} of {got.size} differ"
    z.assert_intact(f"Z [{T},{C}] f32")


@pytest.mark.parametrize("T,C", [(512, 64), (1025, 128), (2048, 256)])
def test_project_bf16_output_and_in_place(T, C):
    x = inputs.normal(80 + C, T * C).reshape(T, C).astype(np.float32)
    w = (inputs.normal(81 + C, C * C) / np.sqrt(C)).reshape(C, C).astype(np.float32)
    xd, wd = bf16_dev(x), bf16_dev(w)
    zg = Guarded((T, C), torch.bfloat16)
    z = whtmix.project(xd, wd, out=zg.t)
    x2 = xd.clone()
    whtmix.project(x2, wd, out=x2)
    whtmix.sync()
    xe = inputs.as_float64(inputs.f32_to_bf16_bits(x), "bf16")
    we = inputs.as_float64(inputs.f32_to_bf16_bits(w), "bf16")
    want = xe @ we.T
    got = z.double().cpu().numpy()
    # rounding to bf16 is within half an ulp, 2^-8 relative; the fp32 sum before it adds an error
    # bounded by the sum of the magnitudes of the products times a few fp32 ulps
    tol = np.abs(want) * 2.0 ** -8 + 1e-6 * (np.abs(xe) @ np.abs(we).T)
    assert (np.abs(got - want) <= tol).all(), float(np.max(np.abs(got - want) / tol))
    assert torch.equal(x2, z)
    zg.assert_intact(f"Z [{T},{C}] bf16")


# (1, 65536, 128), (3, 16384, 128), (2, 32768, 128), (9, 16384, 128), (3, 65536, 128): the fused
# block kernel (columns of 128, 256, 512 rows; the last two over several plane groups)
@pytest.mark.parametrize("B,N,C", [(2, 64, 64), (3, 256, 128), (1, 64, 256), (2, 4096, 128), (1, 65536, 128),
                                   (16, 8192, 256), (3, 16384, 128), (2, 32768, 128), (9, 16384, 128),
                                   (3, 65536, 128)])
def test_block_forward_matches_oracle(B, N, C):
    d = inputs.make_inputs(B, N, C, "bf16", seed=B + N + C)
    w_in = (inputs.normal(90 + C, C * C) / np.sqrt(C)).reshape(C, C).astype(np.float32)
    w_out = (inputs.normal(91 + C, C * C) / np.sqrt(C)).reshape(C, C).astype(np.float32)
    x = torch.from_numpy(d["x"].view(np.int16)).cuda().view(torch.bfloat16)
    g = torch.from_numpy(d["g"]).cuda()
    wi, wo = bf16_dev(w_in), bf16_dev(w_out)
    y = Guarded(x.shape, torch.bfloat16)
    whtmix.block_forward(x, wi, g, wo, out=y.t)
    whtmix.sync()
    y.assert_intact(f"block Y [{B},{N},{C}]")
    x64 = inputs.as_float64(d["x"], "bf16")
    wi64 = inputs.as_float64(inputs.f32_to_bf16_bits(w_in), "bf16")
    wo64 = inputs.as_float64(inputs.f32_to_bf16_bits(w_out), "bf16")
    g64 = d["g"].astype(np.float64)
    three = not fused(N, C)
    z = x64 @ wi64.T
    zr = bf16_round(z) if three else z
    m = oracle.forward(zr, g64)
    ref = m @ wo64.T
    if not three:  # the fused form rounds nothing before M: the same map as the oracle's block
        np.testing.assert_allclose(ref, oracle.block_forward(x64, wi64, g64, wo64), rtol=1e-10, atol=1e-10)
    got = y.t.double().cpu().numpy()
    awo = np.abs(wo64).T
    bound = 2.0 ** -8 * np.abs(ref) + (2.0 ** -8 + 1e-5) * (np.abs(m) @ awo)
    if three:
        bound += 2.0 ** -7 * float(np.abs(g64).max()) * (np.abs(zr) @ awo)
    gp, rp, bp = got.reshape(B, -1), ref.reshape(B, -1), bound.reshape(B, -1)
    for b in range(B):
        rel = np.linalg.norm(gp[b] - rp[b]) / np.linalg.norm(rp[b])
        assert rel <= 1e-2, f"plane {b}: relative L2 {rel:.3e}"
        lim = bp[b] + 1e-5 * float(np.sqrt(np.mean(np.square(rp[b]))))
        bad = np.abs(gp[b] - rp[b]) > lim
        assert not bad.any(), (f"plane {b}: {int(bad.sum())} of {bad.size} elements outside the element-wise "
                               f"bound; worst ratio {float(np.max(np.abs(gp[b] - rp[b]) / lim)):.2f}")
    # in place
    x2 = x.clone()
    whtmix.block_forward(x2, wi, g, wo, out=x2)
    torch.cuda.synchronize()
    assert torch.equal(x2, y.t)


def fused(N, C):
    """True where whtmix_block_forward runs one fused launch (Z stays fp32): C = 128, 2^21..2^23."""
    m = (N * C).bit_length() - 1
    return C == 128 and 21 <= m <= 23


# ---- the block backward ----

@pytest.mark.parametrize("B,N,C", [(2, 64, 64), (3, 256, 128), (1, 64, 256), (2, 4096, 128), (1, 65536, 128),
                                   (4, 8192, 256), (3, 32, 64), (5, 16, 128)])
def test_block_backward_matches_oracle(B, N, C):
    """whtmix_block_backward against the float64 block gradients.  Two references: the exact map
    (acceptance: relative L2 <= 1e-2 per plane for dX, as bf16 outputs, and <= 1e-2 for dW_in, dG,
    dW_out, whose inputs pass through bf16 activations), and the same gradients with Z, M, dM and dZ
    rounded to bf16 where the library rounds them (then dX is its bf16 rounding up to a few flipped
    roundings, and dW_in, dG, dW_out agree to 1e-3).  [3, 32, 64] and [5, 16, 128] have 96 and 80
    tokens, not a multiple of the weight gradients' 64-token tiles."""
    d = inputs.make_inputs(B, N, C, "bf16", seed=B + N + C + 1, with_dy=True)
    w_in = (inputs.normal(92 + C, C * C) / np.sqrt(C)).reshape(C, C).astype(np.float32)
    w_out = (inputs.normal(93 + C, C * C) / np.sqrt(C)).reshape(C, C).astype(np.float32)
    x = torch.from_numpy(d["x"].view(np.int16)).cuda().view(torch.bfloat16)
    dy = torch.from_numpy(d["dy"].view(np.int16)).cuda().view(torch.bfloat16)
    g = torch.from_numpy(d["g"]).cuda()
    wi, wo = bf16_dev(w_in), bf16_dev(w_out)
    outs = [Guarded(x.shape, torch.bfloat16), Guarded((C, C), torch.float32), Guarded((N, C), torch.float32),
            Guarded((C, C), torch.float32)]
    whtmix.block_backward(x, wi, g, wo, dy, dx=outs[0].t, dw_in=outs[1].t, dg=outs[2].t, dw_out=outs[3].t)
    whtmix.sync()
    for o, name in zip(outs, ("dX", "dW_in", "dG", "dW_out")):
        o.assert_intact(f"block {name} [{B},{N},{C}]")
    x64 = inputs.as_float64(d["x"], "bf16")
    dy64 = inputs.as_float64(d["dy"], "bf16")
    wi64 = inputs.as_float64(inputs.f32_to_bf16_bits(w_in), "bf16")
    wo64 = inputs.as_float64(inputs.f32_to_bf16_bits(w_out), "bf16")
    g64 = d["g"].astype(np.float64)
    got = [o.t.double().cpu().numpy() for o in outs]
    # exact map
    exact = oracle.block_backward(x64, wi64, g64, wo64, dy64)
    # rounded where the library rounds: Z, M, dM, dZ to bf16
    zr = bf16_round(x64 @ wi64.T)
    mr = bf16_round(oracle.forward(zr, g64))
    dmr = bf16_round(dy64 @ wo64)
    dz, dg_r = oracle.backward(zr, g64, dmr)
    dzr = bf16_round(dz)
    rounded = [dzr @ wi64, dzr.reshape(-1, C).T @ x64.reshape(-1, C), dg_r, dy64.reshape(-1, C).T @ mr.reshape(-1, C)]

    def rel(a, b):
        return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))

    for k, name in enumerate(("dX", "dW_in", "dG", "dW_out")):
        if k == 0:
            for b in range(B):
                assert rel(got[0][b], exact[0][b]) <= 1e-2, f"dX plane {b}: {rel(got[0][b], exact[0][b]):.3e}"
                assert rel(got[0][b], rounded[0][b]) <= 5e-3, f"dX plane {b} vs rounded: {rel(got[0][b], rounded[0][b]):.3e}"
        else:
            assert rel(got[k], exact[k]) <= 1e-2, f"{name}: {rel(got[k], exact[k]):.3e} vs exact"
            assert rel(got[k], rounded[k]) <= 1e-3, f"{name}: {rel(got[k], rounded[k]):.3e} vs rounded"
    # dX element-wise: the final rounding plus a flipped dZ rounding (one ulp, 2^-7 |dZ|) through W_in
    bound = 2.0 ** -8 * np.abs(rounded[0]) + 2.0 ** -7 * (np.abs(dzr) @ np.abs(wi64)) + 1e-5
    assert (np.abs(got[0] - rounded[0]) <= bound).all(), float(np.max(np.abs(got[0] - rounded[0]) / bound))
    # bit-reproducible
    again = whtmix.block_backward(x, wi, g, wo, dy)
    torch.cuda.synchronize()
    for a, o in zip(again, outs):
        assert torch.equal(a, o.t)


def test_block_autograd_function():
    B, N, C = 2, 512, 128
    d = inputs.make_inputs(B, N, C, "bf16", seed=77, with_dy=True)
    w_in = (inputs.normal(94, C * C) / np.sqrt(C)).reshape(C, C).astype(np.float32)
    w_out = (inputs.normal(95, C * C) / np.sqrt(C)).reshape(C, C).astype(np.float32)
    x = torch.from_numpy(d["x"].view(np.int16)).cuda().view(torch.bfloat16).requires_grad_(True)
    g = torch.from_numpy(d["g"]).cuda().requires_grad_(True)
    wi, wo = bf16_dev(w_in).requires_grad_(True), bf16_dev(w_out).requires_grad_(True)
    y = whtmix.WHTMixBlockFunction.apply(x, wi, g, wo)
    dy = torch.from_numpy(d["dy"].view(np.int16)).cuda().view(torch.bfloat16)
    y.backward(dy)
    ref = whtmix.block_backward(x.detach(), wi.detach(), g.detach(), wo.detach(), dy)
    torch.cuda.synchronize()
    assert torch.equal(x.grad, ref[0]) and torch.equal(g.grad, ref[2])
    assert torch.equal(wi.grad, ref[1].to(torch.bfloat16)) and torch.equal(wo.grad, ref[3].to(torch.bfloat16))


def test_calls_from_a_thread_that_never_set_the_device():
    """The autograd engine (and any caller) may call from a host thread that never set a device:
    every entry point binds the device's context itself, so results match the main thread's."""
    import threading
    B, N, C = 2, 512, 128
    d = inputs.make_inputs(B, N, C, "bf16", seed=78, with_dy=True)
    x = torch.from_numpy(d["x"].view(np.int16)).cuda().view(torch.bfloat16)
    dy = torch.from_numpy(d["dy"].view(np.int16)).cuda().view(torch.bfloat16)
    g = torch.from_numpy(d["g"]).cuda()
    wi = bf16_dev((inputs.normal(96, C * C) / np.sqrt(C)).reshape(C, C).astype(np.float32))
    wo = bf16_dev((inputs.normal(97, C * C) / np.sqrt(C)).reshape(C, C).astype(np.float32))
    calls = {
        "forward": lambda: (whtmix.forward(x, g),),
        "backward": lambda: whtmix.backward(x, g, dy),
        "project": lambda: (whtmix.project(x.view(-1, C), wi),),
        "block_forward": lambda: (whtmix.block_forward(x, wi, g, wo),),
        "block_backward": lambda: whtmix.block_backward(x, wi, g, wo, dy),
    }
    for name, f in calls.items():
        got = {}

        def run():
            try:
                got["r"] = f()
                torch.cuda.synchronize()
            except Exception as e:  # reported below, in the test's thread
                got["e"] = e

        t = threading.Thread(target=run)
        t.start()
        t.join()
        assert "e" not in got, f"{name} from a fresh thread: {got.get('e')}"
        want = f()
        torch.cuda.synchronize()
        for a, b in zip(got["r"], want):
            assert torch.equal(a, b), name

"""GPU checks of the tensor-core projection (whtmix_project) and the whole mixer block
(whtmix_block_forward, Section III-B, Eq. 1-4).

The projection is checked bit-exactly on integer-valued bf16 inputs with fp32 output (every
product and partial sum is an integer below 2^24, so any summation order gives the same fp32
value), and with bf16 output against the fp64 product (half a bf16 ulp plus the fp32 sum's error).  The
block is checked against the fp64 oracle (the projections and the mixer in float64, no
intermediate rounding) with the bf16 tolerance of the other parity tests, relative L2 <= 1e-2 per
plane: the library rounds the block's activations Z and M to bf16 between the steps.
"""
import numpy as np
import pytest
import torch

import oracle
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
    z = whtmix.project(bf16_dev(x), bf16_dev(w), out_dtype=torch.float32)
    whtmix.sync()
    want = (x.astype(np.int64) @ w.astype(np.int64).T).astype(np.float32)
    got = z.cpu().numpy()
    assert np.array_equal(got, want), f"{np.count_nonzero(got != want)} of {got.size} differ"


@pytest.mark.parametrize("T,C", [(512, 64), (1025, 128), (2048, 256)])
def test_project_bf16_output_and_in_place(T, C):
    x = inputs.normal(80 + C, T * C).reshape(T, C).astype(np.float32)
    w = (inputs.normal(81 + C, C * C) / np.sqrt(C)).reshape(C, C).astype(np.float32)
    xd, wd = bf16_dev(x), bf16_dev(w)
    z = whtmix.project(xd, wd)
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
    y = whtmix.block_forward(x, wi, g, wo)
    whtmix.sync()
    ref = oracle.block_forward(inputs.as_float64(d["x"], "bf16"), inputs.as_float64(inputs.f32_to_bf16_bits(w_in), "bf16"),
                               d["g"].astype(np.float64), inputs.as_float64(inputs.f32_to_bf16_bits(w_out), "bf16"))
    got = y.double().cpu().numpy().reshape(B, -1)
    ref = ref.reshape(B, -1)
    for b in range(B):
        rel = np.linalg.norm(got[b] - ref[b]) / np.linalg.norm(ref[b])
        assert rel <= 1e-2, f"plane {b}: relative L2 {rel:.3e}"
    # in place
    x2 = x.clone()
    whtmix.block_forward(x2, wi, g, wo, out=x2)
    torch.cuda.synchronize()
    assert torch.equal(x2, y)

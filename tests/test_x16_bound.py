"""CPU check of the error bound that tests/test_x16_gpu.py applies to whtmix_forward_x16.

A float64 model of the 16-bit exchange: a plane of 2^m = 2^(R+Q) elements as 2^Q rows of 2^R,
row bits forward, every element rounded to bf16 (the first exchange), column bits forward, G/L,
column bits back, rounded to bf16 again (the second exchange), row bits back (Section III-B's
map, computed in that order).  Without the roundings the model must equal the float64 oracle;
with them its error must stay inside the worst-case bound 2^-8 (max|G| / min|G| + 1) of relative
L2 and the element-wise allowance 8 * 2^-9 (max|G| / min|G| + 1) rms(Y) the GPU test uses, and be
well above zero (the roundings are there).  (On the 2^16-element case with the workloads' gains
the model's relative error is 2.34e-3, what the GPU kernel measures with fp32 I/O.)
"""
import numpy as np
import pytest

import oracle
from paper_2607_25234_gb300 import inputs


@pytest.fixture(scope="module", autouse=True)
def built():
    oracle.build()


def fwht_axis(a: np.ndarray, axis: int) -> np.ndarray:
    """Unnormalised natural-order FWHT of every 1D slice along `axis` (float64)."""
    a = np.moveaxis(np.array(a, dtype=np.float64), axis, -1)
    n = a.shape[-1]
    h = 1
    while h < n:
        v = a.reshape(a.shape[:-1] + (n // (2 * h), 2, h))
        x0, x1 = v[..., 0, :].copy(), v[..., 1, :].copy()
        v[..., 0, :], v[..., 1, :] = x0 + x1, x0 - x1
        a = v.reshape(a.shape)
        h *= 2
    return np.moveaxis(a, -1, axis)


def bf16(a: np.ndarray) -> np.ndarray:
    return inputs.as_float64(inputs.f32_to_bf16_bits(np.asarray(a, dtype=np.float32)), "bf16")


def x16_model(x: np.ndarray, g: np.ndarray, R: int, round_exchange: bool = True) -> np.ndarray:
    N, C = x.shape
    L = N * C
    Q = int(np.log2(L)) - R
    q = bf16 if round_exchange else (lambda a: a)
    a = q(fwht_axis(x.reshape(1 << Q, 1 << R), 1))
    a = fwht_axis(fwht_axis(a, 0) * g.reshape(1 << Q, 1 << R) / L, 0)
    return fwht_axis(q(a), 1).reshape(N, C)


@pytest.mark.parametrize("N,C,R,gain", [
    (1024, 64, 13, "normal"),   # the GPU kernel's split for 2^16 planes
    (512, 128, 13, "normal"),
    (1024, 64, 10, "normal"),   # another split: the bound does not depend on it
    (1024, 64, 13, "unit"),
    (1024, 64, 13, "wide"),     # max|G| / min|G| = 16: the bound grows with it
])
def test_x16_error_within_its_bound(N, C, R, gain):
    d = inputs.make_inputs(1, N, C, "bf16", seed=7)
    x = inputs.as_float64(d["x"], "bf16")[0]
    rng = np.random.default_rng(3)
    g = {"normal": d["g"].astype(np.float64), "unit": np.ones((N, C)),
         "wide": 2.0 ** rng.uniform(-2, 2, size=(N, C))}[gain]
    ref = oracle.forward(x[None], g)[0]
    exact = x16_model(x, g, R, round_exchange=False)
    assert np.abs(exact - ref).max() <= 1e-12 * np.abs(ref).max()     # the model is the map
    y = x16_model(x, g, R)
    kappa = np.abs(g).max() / np.abs(g).min()
    rel = np.linalg.norm(y - ref) / np.linalg.norm(ref)
    assert 2.0 ** -12 < rel <= 2.0 ** -8 * (kappa + 1), (rel, kappa)
    rms = np.sqrt(np.mean(ref ** 2))
    assert np.abs(y - ref).max() <= 8 * 2.0 ** -9 * (kappa + 1) * rms

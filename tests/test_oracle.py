"""Pins for the CPU oracle (no GPU).

The oracle computes Y = H_N (G (.) H_N X H_C) H_C / (N C) with butterflies (paper Section III-B,
Eq. 1-4).  Nothing here re-types its butterfly: every expected value comes from something else --
dense Sylvester-Hadamard matrices built from the popcount definition, from the Sylvester
recursion or by scipy.linalg.hadamard; closed forms for delta inputs and single-frequency gains;
the invariants the paper states (orthonormal => self-inverse and magnitude preserving, the block
is linear); the adjoint identity and finite differences for the backward; hand-derived goldens.
"""
import os

import numpy as np
import pytest
import scipy.linalg

import oracle
from paper_2607_25234_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "whtmix_hand_cases.txt")


def popcount_hadamard(n: int) -> np.ndarray:
    """(H_n)_{ij} = (-1)^{popcount(i & j)} -- the Sylvester-Hadamard definition."""
    i = np.arange(n, dtype=np.uint64)
    bits = np.bitwise_count(np.bitwise_and.outer(i, i))
    return np.where(bits % 2 == 0, 1, -1).astype(np.int64)


def recursive_hadamard(n: int) -> np.ndarray:
    """Sylvester's construction H_{2m} = [[H_m, H_m], [H_m, -H_m]], H_1 = [1]."""
    h = np.ones((1, 1), dtype=np.int64)
    while h.shape[0] < n:
        h = np.block([[h, h], [h, -h]])
    return h


def dense_forward(x, g):
    """H_N (G (.) H_N X H_C) H_C / (N C) per plane, with dense scipy Hadamard matrices."""
    _, N, C = x.shape
    hn = scipy.linalg.hadamard(N).astype(np.float64)
    hc = scipy.linalg.hadamard(C).astype(np.float64)
    return np.stack([hn @ (g * (hn @ xb @ hc)) @ hc for xb in x]) / (N * C)


def rng_normal(shape, seed):
    return inputs.normal(seed, int(np.prod(shape))).reshape(shape)


POW2 = [1, 2, 4, 8, 16, 32, 64, 128, 256, 512, 1024]


@pytest.mark.parametrize("n", POW2)
def test_fwht_equals_popcount_matrix_exactly(n):
    v = inputs.small_ints(7, n, -1000, 1000).astype(np.float64)
    np.testing.assert_array_equal(oracle.fwht(v), popcount_hadamard(n) @ v)


@pytest.mark.parametrize("n", [1, 2, 8, 64, 256])
def test_fwht_equals_scipy_hadamard(n):
    v = rng_normal((n,), 11)
    np.testing.assert_allclose(oracle.fwht(v), scipy.linalg.hadamard(n) @ v, rtol=1e-13, atol=1e-12)


def test_sylvester_recursion_matches_popcount_and_scipy():
    for n in POW2:
        r = recursive_hadamard(n)
        np.testing.assert_array_equal(r, popcount_hadamard(n))
        np.testing.assert_array_equal(r, scipy.linalg.hadamard(n))


@pytest.mark.parametrize("n", [1, 4, 32, 512])
def test_fwht_twice_is_n_times_identity(n):
    # H_n H_n = n I, applied to integer vectors so the check is exact.
    v = inputs.small_ints(3, n, -50, 50).astype(np.float64)
    np.testing.assert_array_equal(oracle.fwht(oracle.fwht(v)), n * v)
    h = popcount_hadamard(n)
    np.testing.assert_array_equal(h @ h, n * np.eye(n, dtype=np.int64))


@pytest.mark.parametrize("n", [2, 16, 1024])
def test_fwht_u32_wraps_like_int64_mod_2_32(n):
    v = inputs.splitmix64(5, n).astype(np.uint64) & np.uint64(0xFFFFFFFF)
    h = popcount_hadamard(n).astype(np.uint64)  # -1 -> 2^64 - 1, so uint64 matmul is exact mod 2^64
    want = ((h @ v) & np.uint64(0xFFFFFFFF)).astype(np.uint32)
    np.testing.assert_array_equal(oracle.fwht(v.astype(np.uint32)), want)


SHAPES = [(1, 1), (1, 8), (8, 1), (2, 2), (4, 16), (16, 4), (2, 64), (32, 64), (64, 32), (64, 64)]


@pytest.mark.parametrize("N,C", SHAPES)
def test_forward_equals_dense_definition(N, C):
    x = rng_normal((3, N, C), 1)
    g = 1.0 + 0.1 * rng_normal((N, C), 2)
    np.testing.assert_allclose(oracle.forward(x, g), dense_forward(x, g), rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("N,C", [(4, 8), (16, 16), (8, 128), (256, 4)])
def test_forward_equals_1d_transform_of_flattened_plane(N, C):
    # Kronecker identity: H_N (x) H_C = H_{NC} in Sylvester order with c the low index bits.
    L = N * C
    x = rng_normal((N, C), 3)
    g = rng_normal((N, C), 4)
    h = scipy.linalg.hadamard(L).astype(np.float64)
    want = (h @ (g.reshape(-1) * (h @ x.reshape(-1)))) / L
    np.testing.assert_allclose(oracle.forward(x, g).reshape(-1), want, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(oracle.wht2d(x).reshape(-1), h @ x.reshape(-1), rtol=1e-12, atol=1e-11)


@pytest.mark.parametrize("N,C", [(1, 1), (1, 64), (64, 1), (256, 64), (512, 128)])
def test_unit_gain_is_identity(N, C):
    # Gains initialised to zero in the log domain are unit gains: the mixer starts as the
    # identity, because the orthonormal transform is its own inverse (Section III-B).
    x = rng_normal((2, N, C), 5)
    np.testing.assert_allclose(oracle.forward(x, np.ones((N, C))), x, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("N,C", [(4, 4), (128, 32), (1024, 16)])
def test_parseval_magnitude_preserving(N, C):
    x = rng_normal((N, C), 6)
    w = oracle.wht2d(x) / np.sqrt(N * C)
    assert abs(np.linalg.norm(w) - np.linalg.norm(x)) <= 1e-12 * np.linalg.norm(x)
    signs = np.where(inputs.uniform01(8, N * C) < 0.5, -1.0, 1.0).reshape(N, C)
    y = oracle.forward(x, signs)  # |G| = 1 keeps the whole map orthogonal
    assert abs(np.linalg.norm(y) - np.linalg.norm(x)) <= 1e-12 * np.linalg.norm(x)


@pytest.mark.parametrize("N,C", [(1, 1), (2, 8), (64, 32), (512, 4)])
def test_dc_gain_gives_plane_mean(N, C):
    x = rng_normal((2, N, C), 9)
    g = np.zeros((N, C))
    g[0, 0] = 1.0
    y = oracle.forward(x, g)
    for b in range(2):
        np.testing.assert_allclose(y[b], np.full((N, C), x[b].mean()), rtol=1e-11, atol=1e-13)


@pytest.mark.parametrize("N,C,i,j", [(8, 4, 0, 0), (8, 4, 5, 3), (64, 16, 33, 7), (1, 8, 0, 5)])
def test_delta_input_closed_forms(N, C, i, j):
    x = np.zeros((N, C))
    x[i, j] = 1.0
    hn, hc = popcount_hadamard(N), popcount_hadamard(C)
    # The orthonormal transform of a delta is the outer product of two Hadamard rows; a delta at
    # the origin maps to the constant plane 1/sqrt(NC).
    w = oracle.wht2d(x) / np.sqrt(N * C)
    np.testing.assert_allclose(w, np.outer(hn[i], hc[j]) / np.sqrt(N * C), rtol=0, atol=1e-15)
    # Keeping only token-frequency 0 maps the delta to constant rows: Y[n, c] = [c == j] / N.
    g = np.zeros((N, C))
    g[0, :] = 1.0
    want = np.zeros((N, C))
    want[:, j] = 1.0 / N
    np.testing.assert_allclose(oracle.forward(x, g), want, rtol=0, atol=1e-15)
    # Single frequency (k, l): Y = (H_N[i,k] H_C[j,l] / L) * outer(H_N[k], H_C[l]).
    k, l = (N - 1) // 3, (C - 1) // 2
    g = np.zeros((N, C))
    g[k, l] = 1.0
    want = hn[i, k] * hc[j, l] * np.outer(hn[k], hc[l]) / (N * C)
    np.testing.assert_allclose(oracle.forward(x, g), want, rtol=0, atol=1e-15)


@pytest.mark.parametrize("N,C", [(4, 8), (32, 16), (16, 64)])
def test_rank1_gain_equals_sequential_channel_then_token_mix(N, C):
    # Eq. 2 (channel mix with exp(g_c)) followed by Eq. 3 (token mix with exp(g_t)), each written
    # with dense orthonormal matrices, equals the 2D map with G = exp(g_t) exp(g_c)^T.
    x = rng_normal((N, C), 12)
    g_c, g_t = 0.3 * rng_normal((C,), 13), 0.3 * rng_normal((N,), 14)
    hc = scipy.linalg.hadamard(C) / np.sqrt(C)
    hn = scipy.linalg.hadamard(N) / np.sqrt(N)
    z = x @ hc @ np.diag(np.exp(g_c)) @ hc          # each row z <- H_C^-1 (e^{g_c} (.) H_C z)
    z = hn @ np.diag(np.exp(g_t)) @ hn @ z          # each column likewise with e^{g_t}
    np.testing.assert_allclose(oracle.forward(x, np.outer(np.exp(g_t), np.exp(g_c))), z, rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("N,C", [(4, 8), (32, 16), (16, 64)])
def test_separable_forward_equals_sequential_eq2_then_eq3(N, C):
    # forward_separable against the paper's sequential form written with dense orthonormal
    # matrices: the channel mix with diag(exp(g_c)) on every token row (Eq. 2), then the token
    # mix with diag(exp(g_t)) on every channel column (Eq. 3).
    x = rng_normal((2, N, C), 15)
    g_t, g_c = 0.2 * rng_normal((N,), 16), 0.2 * rng_normal((C,), 17)
    hc = scipy.linalg.hadamard(C) / np.sqrt(C)
    hn = scipy.linalg.hadamard(N) / np.sqrt(N)
    want = np.stack([hn @ np.diag(np.exp(g_t)) @ hn @ (xb @ hc @ np.diag(np.exp(g_c)) @ hc) for xb in x])
    np.testing.assert_allclose(oracle.forward_separable(x, g_t, g_c), want, rtol=1e-11, atol=1e-12)
    # zero log gains are the paper's initialisation: the mixer starts as the identity
    np.testing.assert_allclose(oracle.forward_separable(x, np.zeros(N), np.zeros(C)), x, rtol=0, atol=1e-13)


@pytest.mark.parametrize("B,N,C", [(1, 8, 4), (3, 16, 8), (2, 4, 32)])
def test_separable_backward_finite_differences(B, N, C):
    x, dy = rng_normal((B, N, C), 45), rng_normal((B, N, C), 46)
    g_t, g_c = 0.2 * rng_normal((N,), 47), 0.2 * rng_normal((C,), 48)
    dx, dgt, dgc = oracle.backward_separable(x, g_t, g_c, dy)
    np.testing.assert_allclose(dx, dense_forward(dy, np.outer(np.exp(g_t), np.exp(g_c))), rtol=1e-11, atol=1e-12)
    loss = lambda gt, gc: np.vdot(oracle.forward_separable(x, gt, gc), dy)
    eps = 1e-5
    for n in sorted({0, N // 2, N - 1}):
        e = np.zeros(N)
        e[n] = eps
        fd = (loss(g_t + e, g_c) - loss(g_t - e, g_c)) / (2 * eps)
        assert abs(fd - dgt[n]) <= 1e-7 * max(1.0, abs(fd)), (n, fd, dgt[n])
    for c in sorted({0, C // 2, C - 1}):
        e = np.zeros(C)
        e[c] = eps
        fd = (loss(g_t, g_c + e) - loss(g_t, g_c - e)) / (2 * eps)
        assert abs(fd - dgc[c]) <= 1e-7 * max(1.0, abs(fd)), (c, fd, dgc[c])
    # a common shift of every log gain scales G by exp(s), so d loss / d s = loss = sum dg_t = sum dg_c
    total = loss(g_t, g_c)
    assert abs(dgt.sum() - total) <= 1e-10 * max(1.0, abs(total))
    assert abs(dgc.sum() - total) <= 1e-10 * max(1.0, abs(total))


@pytest.mark.parametrize("B,N,C", [(1, 8, 4), (2, 16, 8), (1, 4, 16)])
def test_block_forward_dense_and_special_cases(B, N, C):
    # dense: H_N (G (.) H_N (X W_in^T) H_C) H_C W_out^T / (N C) with scipy Hadamard matrices
    x = rng_normal((B, N, C), 60)
    w_in, w_out = rng_normal((C, C), 61), rng_normal((C, C), 62)
    g = 1.0 + 0.1 * rng_normal((N, C), 63)
    hn = scipy.linalg.hadamard(N).astype(np.float64)
    hc = scipy.linalg.hadamard(C).astype(np.float64)
    want = np.stack([hn @ (g * (hn @ (xb @ w_in.T) @ hc)) @ hc @ w_out.T for xb in x]) / (N * C)
    np.testing.assert_allclose(oracle.block_forward(x, w_in, g, w_out), want, rtol=1e-11, atol=1e-12)
    # identity projections: the mixer alone; unit gains: the two projections alone
    eye = np.eye(C)
    np.testing.assert_allclose(oracle.block_forward(x, eye, g, eye), oracle.forward(x, g), rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(oracle.block_forward(x, w_in, np.ones((N, C)), w_out), x @ w_in.T @ w_out.T,
                               rtol=1e-11, atol=1e-12)


def test_linear_in_x_and_in_g():
    N, C = 32, 16
    x1, x2 = rng_normal((N, C), 20), rng_normal((N, C), 21)
    g1, g2 = rng_normal((N, C), 22), rng_normal((N, C), 23)
    a, b = 0.75, -1.5
    np.testing.assert_allclose(oracle.forward(a * x1 + b * x2, g1),
                               a * oracle.forward(x1, g1) + b * oracle.forward(x2, g1), rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(oracle.forward(x1, a * g1 + b * g2),
                               a * oracle.forward(x1, g1) + b * oracle.forward(x1, g2), rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("B,N,C", [(1, 8, 4), (3, 16, 32), (4, 64, 8)])
def test_backward_adjoint_identity(B, N, C):
    x, dy = rng_normal((B, N, C), 30), rng_normal((B, N, C), 31)
    g = 1.0 + 0.1 * rng_normal((N, C), 32)
    dx, _ = oracle.backward(x, g, dy)
    lhs = np.vdot(oracle.forward(x, g), dy)
    assert abs(lhs - np.vdot(x, dx)) <= 1e-11 * max(1.0, abs(lhs))
    np.testing.assert_allclose(dx, dense_forward(dy, g), rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("B,N,C", [(1, 4, 4), (3, 16, 8), (5, 8, 32)])
def test_backward_dg_dense_and_finite_difference(B, N, C):
    x, dy = rng_normal((B, N, C), 40), rng_normal((B, N, C), 41)
    g = 1.0 + 0.1 * rng_normal((N, C), 42)
    _, dg = oracle.backward(x, g, dy)
    hn = scipy.linalg.hadamard(N).astype(np.float64)
    hc = scipy.linalg.hadamard(C).astype(np.float64)
    want = sum((hn @ x[b] @ hc) * (hn @ dy[b] @ hc) for b in range(B)) / (N * C)
    np.testing.assert_allclose(dg, want, rtol=1e-11, atol=1e-12)
    # Y is linear in G, so a finite difference along any direction is exact up to rounding.
    delta = rng_normal((N, C), 43)
    eps = 1e-3
    fd = (np.vdot(oracle.forward(x, g + eps * delta), dy) - np.vdot(oracle.forward(x, g - eps * delta), dy)) / (2 * eps)
    assert abs(fd - np.vdot(dg, delta)) <= 1e-8 * max(1.0, abs(fd))
    # Central differences of a scalar loss in single entries of X and G.
    loss_w = rng_normal((B, N, C), 44)
    dx_l, dg_l = oracle.backward(x, g, loss_w)
    for (b, n, c) in [(0, 0, 0), (B - 1, N - 1, C - 1), (B // 2, N // 2, 1)]:
        e = np.zeros_like(x)
        e[b, n, c] = eps
        fdx = (np.vdot(oracle.forward(x + e, g), loss_w) - np.vdot(oracle.forward(x - e, g), loss_w)) / (2 * eps)
        assert abs(fdx - dx_l[b, n, c]) <= 1e-8 * max(1.0, abs(fdx))
        eg = np.zeros_like(g)
        eg[n, c] = eps
        fdg = (np.vdot(oracle.forward(x, g + eg), loss_w) - np.vdot(oracle.forward(x, g - eg), loss_w)) / (2 * eps)
        assert abs(fdg - dg_l[n, c]) <= 1e-8 * max(1.0, abs(fdg))


def _dense_u32_forward(x, g):
    B, N, C = x.shape
    hn = popcount_hadamard(N).astype(np.uint64)
    hc = popcount_hadamard(C).astype(np.uint64)
    xs = x.astype(np.int64).astype(np.uint64)
    gs = g.astype(np.int64).astype(np.uint64)
    out = np.stack([hn @ (gs * (hn @ xb @ hc)) @ hc for xb in xs])  # exact mod 2^64
    return (out & np.uint64(0xFFFFFFFF)).astype(np.uint32).view(np.int32)


@pytest.mark.parametrize("N,C", [(1, 1), (4, 2), (8, 16), (32, 32), (16, 64)])
def test_integer_mode_bit_exact_vs_int64_dense(N, C):
    d = inputs.make_inputs(2, N, C, "i32", seed=50)
    np.testing.assert_array_equal(oracle.forward(d["x"], d["g"]), _dense_u32_forward(d["x"], d["g"]))
    # Values large enough to wrap around 2^32 many times.
    xw = inputs.small_ints(51, 2 * N * C, -(2**31), 2**31 - 1).reshape(2, N, C)
    gw = inputs.small_ints(52, N * C, -(2**31), 2**31 - 1).reshape(N, C)
    np.testing.assert_array_equal(oracle.forward(xw, gw), _dense_u32_forward(xw, gw))


@pytest.mark.parametrize("N,C", [(4, 4), (16, 8)])
def test_integer_backward_bit_exact(N, C):
    d = inputs.make_inputs(3, N, C, "i32", seed=60, with_dy=True)
    dx, dg = oracle.backward(d["x"], d["g"], d["dy"])
    np.testing.assert_array_equal(dx, _dense_u32_forward(d["dy"], d["g"]))
    hn = popcount_hadamard(N)
    hc = popcount_hadamard(C)
    want = sum((hn @ d["x"][b].astype(np.int64) @ hc) * (hn @ d["dy"][b].astype(np.int64) @ hc) for b in range(3))
    np.testing.assert_array_equal(dg, (want.astype(np.uint64) & np.uint64(0xFFFFFFFF)).astype(np.uint32).view(np.int32))


def _golden_cases():
    cases = []
    with open(GOLDEN) as f:
        for line in f:
            if not line.strip() or line.startswith("#"):
                continue
            name, nc, xs, gs, yi, yf = [p.strip() for p in line.split("|")]
            N, C = map(int, nc.split())
            cases.append((name, N, C, [float(v) for v in xs.split()], [float(v) for v in gs.split()],
                          [int(v) for v in yi.split()], [float(v) for v in yf.split()]))
    return cases


@pytest.mark.parametrize("case", _golden_cases(), ids=lambda c: c[0])
def test_hand_derived_golden_cases(case):
    _, N, C, xs, gs, yi, yf = case
    x = np.array(xs).reshape(1, N, C)
    g = np.array(gs).reshape(N, C)
    np.testing.assert_array_equal(oracle.forward(x.astype(np.int32), g.astype(np.int32)).reshape(-1), yi)
    np.testing.assert_allclose(oracle.forward(x, g).reshape(-1), yf, rtol=0, atol=1e-15)


def test_rejects_non_power_of_two():
    with pytest.raises(ValueError):
        oracle.forward(np.zeros((1, 3, 4)), np.zeros((3, 4)))
    with pytest.raises(ValueError):
        oracle.forward(np.zeros((1, 4, 6)), np.zeros((4, 6)))


# ---- the seeded input generator (shared by both sides, so it is pinned too) ----

def test_splitmix64_published_sequence():
    # First outputs of SplitMix64 with seed 0, as published with the generator.
    assert [int(v) for v in inputs.splitmix64(0, 3)] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    v = inputs.normal(70, 100000).astype(np.float32)
    # exact ties: the 16 dropped bits are 0x8000
    ties = (np.arange(1000, dtype=np.uint32) << np.uint32(16)) | np.uint32(0x3F808000)
    v = np.concatenate([v, ties.view(np.float32)])
    want = torch.from_numpy(v).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(inputs.f32_to_bf16_bits(v), want)
    np.testing.assert_array_equal(inputs.bf16_bits_to_f32(want), torch.from_numpy(want.view(np.int16)).view(torch.bfloat16).float().numpy())


def test_normal_generator_moments():
    z = inputs.normal(0, 1 << 20)
    assert abs(z.mean()) < 5e-3 and abs(z.std() - 1.0) < 5e-3
    d = inputs.make_inputs(1, 65536, 128, "bf16", n_valid=64800)
    assert (d["x"][0, 64800:] == 0).all() and (d["x"][0, :64800] != 0).mean() > 0.99


@pytest.mark.parametrize("B,N,C", [(3, 64, 32), (2, 1024, 4), (1, 1, 256), (2, 512, 1), (1, 4096, 64)])
def test_threaded_oracle_is_bit_identical_to_single_threaded(B, N, C):
    """The all-core CPU baseline's threaded mode splits only independent work (rows, column
    blocks, elements), so forward and backward must match the single-threaded oracle bit for bit."""
    d = inputs.make_inputs(B, N, C, "f32", seed=B + N + C, with_dy=True)
    x, g, dy = (d[k].astype(np.float64) for k in ("x", "g", "dy"))
    try:
        assert oracle.set_threads(1) == 1
        y1 = oracle.forward(x, g)
        dx1, dg1 = oracle.backward(x, g, dy)
        w1 = oracle.wht2d(x)
        if oracle.set_threads(4) != 4:
            pytest.skip("oracle built without OpenMP")
        y4 = oracle.forward(x, g)
        dx4, dg4 = oracle.backward(x, g, dy)
        w4 = oracle.wht2d(x)
    finally:
        oracle.set_threads(1)
    for a, b in ((y1, y4), (dx1, dx4), (dg1, dg4), (w1, w4)):
        np.testing.assert_array_equal(a, b)


def test_block_backward_matches_central_differences():
    """Every gradient of the block (Eq. 1-4) against central differences of <Y, dY> (the block is
    linear in each argument, so the differences are exact up to rounding)."""
    rng = np.random.default_rng(5)
    B, N, C = 2, 4, 8
    x = rng.standard_normal((B, N, C))
    w_in = rng.standard_normal((C, C)) / np.sqrt(C)
    w_out = rng.standard_normal((C, C)) / np.sqrt(C)
    g = 1.0 + 0.1 * rng.standard_normal((N, C))
    dy = rng.standard_normal((B, N, C))
    dx, dw_in, dg, dw_out = oracle.block_backward(x, w_in, g, w_out, dy)

    def loss(x_, wi_, g_, wo_):
        return float(np.sum(oracle.block_forward(x_, wi_, g_, wo_) * dy))

    h = 1e-3
    args = [x, w_in, g, w_out]
    for k, grad in enumerate((dx, dw_in, dg, dw_out)):
        num = np.zeros_like(grad)
        for idx in np.ndindex(grad.shape):
            plus = [a.copy() for a in args]
            minus = [a.copy() for a in args]
            plus[k][idx] += h
            minus[k][idx] -= h
            num[idx] = (loss(*plus) - loss(*minus)) / (2 * h)
        np.testing.assert_allclose(grad, num, rtol=1e-7, atol=1e-9, err_msg=f"gradient {k}")


def test_block_backward_special_cases():
    """Identity projections and unit gains make the block the identity, so every input gradient is
    dY itself and dG is the plain mixer's; a zero upstream gradient gives zero gradients."""
    rng = np.random.default_rng(6)
    B, N, C = 3, 8, 4
    x = rng.standard_normal((B, N, C))
    dy = rng.standard_normal((B, N, C))
    eye = np.eye(C)
    ones = np.ones((N, C))
    dx, dw_in, dg, dw_out = oracle.block_backward(x, eye, ones, eye, dy)
    np.testing.assert_allclose(dx, dy, atol=1e-12)
    np.testing.assert_allclose(dg, oracle.backward(x, ones, dy)[1], atol=1e-12)
    # with identity weights and unit gains Y = X, so dW_out = sum_t dY^T X = dW_in
    np.testing.assert_allclose(dw_out, dy.reshape(-1, C).T @ x.reshape(-1, C), atol=1e-12)
    np.testing.assert_allclose(dw_in, dw_out, atol=1e-12)
    z = oracle.block_backward(x, eye, ones, eye, np.zeros_like(dy))
    assert all(np.count_nonzero(a) == 0 for a in z)

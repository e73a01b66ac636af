"""The GPU parity checks themselves, on the CPU: a result that is the oracle's rounded once to the
output dtype (plus fp32-sized noise) passes, and a single wrong element, a guard byte or a
dG computed at bf16 precision fails.  This keeps the checks able to see one bad element."""
import numpy as np
import pytest
import torch

import oracle
from _checks import Guarded, bf16_round, check, check_grad
from paper_2607_25234_gb300 import inputs


def sample(B=2, N=256, C=64, seed=0):
    d = inputs.make_inputs(B, N, C, "bf16", seed=seed)
    x = inputs.as_float64(d["x"], "bf16")
    return oracle.forward(x, d["g"].astype(np.float64))


def fp32_path(ref, seed=1):
    """The reference as an fp32 path would leave it: a 3e-7 relative wobble (the size of the fp32
    butterflies' error), then rounded to fp32."""
    rng = np.random.default_rng(seed)
    return (ref * (1.0 + 3e-7 * rng.standard_normal(ref.shape))).astype(np.float32).astype(np.float64)


def test_bf16_check_accepts_one_rounding_and_rejects_one_wrong_element():
    ref = sample()
    got = bf16_round(fp32_path(ref))
    check(got, ref, "bf16", "rounded once")
    bad = got.copy()
    bad.reshape(-1)[12345] += 0.05 * max(1.0, abs(bad.reshape(-1)[12345]))
    with pytest.raises(AssertionError, match="outside"):
        check(bad, ref, "bf16", "one element off")
    bad = got.copy()
    bad.reshape(-1)[777] = -bad.reshape(-1)[777] if bad.reshape(-1)[777] != 0 else 1.0   # a flipped sign
    with pytest.raises(AssertionError):
        check(bad, ref, "bf16", "one sign flipped")


def test_f32_check_accepts_fp32_rounding_and_rejects_small_errors():
    ref = sample()
    check(fp32_path(ref), ref, "f32", "fp32")
    bad = fp32_path(ref)
    bad.reshape(-1)[99] += 3e-5
    with pytest.raises(AssertionError):
        check(bad, ref, "f32", "one element off by 3e-5")


def test_grad_check_holds_bf16_inputs_to_the_fp32_bound():
    d = inputs.make_inputs(4, 64, 32, "bf16", seed=3, with_dy=True)
    r = {k: inputs.as_float64(v, "bf16" if k != "g" else "f32") for k, v in d.items()}
    _, dg = oracle.backward(r["x"], r["g"], r["dy"])
    check_grad(fp32_path(dg), dg, "bf16", "dG fp32")
    with pytest.raises(AssertionError):
        check_grad(bf16_round(dg), dg, "bf16", "dG rounded to bf16")   # bf16 precision is not enough


def test_int_check_is_exact():
    a = np.arange(12, dtype=np.int32).reshape(1, 3, 4)
    check(a.copy(), a, "i32", "same")
    b = a.copy()
    b[0, 1, 2] += 1
    with pytest.raises(AssertionError):
        check(b, a, "i32", "one off")


def test_guard_region_sees_a_write_next_to_the_output():
    g = Guarded((3, 5), torch.float32, device="cpu")
    g.t.fill_(1.0)
    g.assert_intact("inside only")
    g.buf[g.buf.numel() - 1] = 0
    with pytest.raises(AssertionError, match="after"):
        g.assert_intact("one byte after")
    h = Guarded((7,), torch.bfloat16, device="cpu")
    h.buf[100] = 1
    with pytest.raises(AssertionError, match="before"):
        h.assert_intact("one byte before")

"""Failure detection on the GPU without a fault: a device-wide barrier whose arrivals can never
complete gives up after its bounded wait (about one second), records the error in the barrier
header's error word and returns; the context stays usable and the next call is correct.

The barrier is made to wait forever the way a missing CTA would: the caller-owned workspace of
the _ex calls starts with its four arrival counters far from zero, so no counter ever holds
exactly the grid's CTA count that releases the waiters.  Nothing faults, traps or hangs: every CTA
leaves on its own after the time limit.
"""
import time

import numpy as np
import pytest
import torch

import oracle
from paper_2607_25234_gb300 import inputs, whtmix

pytestmark = pytest.mark.gpu

STUCK = 1 << 30   # an arrival count no grid reaches


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


@pytest.mark.parametrize("B,N,C,dtype,backward", [(2, 8192, 128, "bf16", False),   # three-phase fast forward
                                                  (3, 1024, 128, "f32", True),     # fast backward
                                                  (2, 8192, 64, "i32", False)])    # generic engine
def test_stuck_barrier_times_out_and_the_context_stays_usable(B, N, C, dtype, backward):
    d = inputs.make_inputs(B, N, C, dtype, seed=31, with_dy=backward)
    tdt = {"f32": torch.float32, "bf16": torch.bfloat16, "i32": torch.int32}[dtype]
    x = to_dev(d["x"], dtype)
    g = to_dev(d["g"], "i32" if dtype == "i32" else "f32")
    dy = to_dev(d["dy"], dtype) if backward else None
    ws = torch.zeros(whtmix.workspace_bytes(B, N, C, tdt, backward=backward), dtype=torch.uint8, device="cuda")
    header = ws[:256].view(torch.int32)
    for word in (0, 1, 3, 4):   # the four arrival counters (word 2 is the error word)
        header[word] = STUCK
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    if backward:
        whtmix.backward_ex(x, g, dy, ws)
    else:
        whtmix.forward_ex(x, g, ws)
    torch.cuda.synchronize()   # returns: the kernel gave up on its own
    waited = time.perf_counter() - t0
    h = header.cpu()
    assert h[2].item() != 0, "the error word records the expired wait"
    assert 0.5 < waited < 30.0, f"the bounded wait took {waited:.2f} s"
    # reset the header as the library does after a timeout; the next call is correct
    ws[:256].zero_()
    r = {k: inputs.as_float64(v, dtype) if dtype != "i32" else v for k, v in d.items() if k != "g"}
    gref = d["g"].astype(np.float64) if dtype != "i32" else d["g"]
    if backward:
        dx, dg = whtmix.backward_ex(x, g, dy, ws)
        torch.cuda.synchronize()
        dx_ref, dg_ref = oracle.backward(r["x"], gref, r["dy"])
        got = dx.double().cpu().numpy()
        assert np.linalg.norm(got - dx_ref) <= 1e-6 * np.linalg.norm(dx_ref)
    else:
        y = whtmix.forward_ex(x, g, ws)
        torch.cuda.synchronize()
        y_ref = oracle.forward(r["x"], gref)
        if dtype == "i32":
            assert np.array_equal(y.cpu().numpy(), y_ref)
        else:
            got = y.double().cpu().numpy().reshape(B, -1)
            ref = y_ref.reshape(B, -1)
            assert (np.linalg.norm(got - ref, axis=1) <= 1e-2 * np.linalg.norm(ref, axis=1)).all()
    assert ws[:256].view(torch.int32)[2].item() == 0

"""whtmix_forward_noalloc: the forward for callers that may not allocate device memory.

Such callers (a process whose device memory belongs to an outside allocator, a real-time loop, a
plugin handed only its buffers) cannot let the library allocate a workspace.  This entry point
keeps its scratch in a fixed array inside the library instead and runs the kernels whtmix_forward
picks for the shape.  Here it is called through the C ABI twice in a row per case -- the second
call reuses the array the first one left behind -- and each result is compared with
whtmix_forward's on the same inputs: within the tolerances the parity tests use (int32 exact, fp32
relative L2 <= 1e-6 and max abs <= 1e-5, bf16 relative L2 <= 1e-2), and bit for bit, since the
kernels are the same.  The device's free memory must not change across the calls, and whtmix_sync
must report no expired wait afterwards.

The file name sorts last so that a run stopping at the first failure has already run every other
test; it also passes on its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2607_25234_gb300 import build, inputs, whtmix

pytestmark = pytest.mark.gpu

CODE = {"f32": 0, "bf16": 1, "i32": 2}


@pytest.fixture(scope="module")
def lib():
    build.build()
    lib = whtmix.library()
    p, i64, i = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
    lib.whtmix_forward_noalloc.argtypes = [p, p, p, i64, i64, i64, i, p]
    lib.whtmix_forward_noalloc.restype = ctypes.c_int
    torch.cuda.set_device(0)
    return lib


def device_inputs(B, N, C, dtype, seed):
    d = inputs.make_inputs(B, N, C, dtype, seed=seed)
    if dtype == "bf16":
        x = torch.from_numpy(d["x"].view(np.int16)).cuda().view(torch.bfloat16)
    else:
        x = torch.from_numpy(d["x"]).cuda()
    return x, torch.from_numpy(d["g"]).cuda()


def assert_matches(got: torch.Tensor, want: torch.Tensor, dtype: str, what: str):
    if dtype == "i32":
        assert torch.equal(got, want), what
        return
    a = got.double().reshape(got.shape[0], -1)
    b = want.double().reshape(want.shape[0], -1)
    rel = ((a - b).norm(dim=1) / b.norm(dim=1).clamp_min(1e-30)).max().item()
    assert rel <= (1e-6 if dtype == "f32" else 1e-2), f"{what}: relative L2 {rel:.3e}"
    if dtype == "f32":
        assert (a - b).abs().max().item() <= 1e-5, what
    assert torch.equal(got, want), f"{what}: not bit-identical to whtmix_forward (same kernels)"


# pairs of consecutive calls: (B, N, C, dtype) for the first and the second call
PAIRS = [
    ((4, 4096, 64, "f32"), (4, 4096, 64, "f32")),        # same shape, new inputs (three-phase kernel, 2^18)
    ((2, 8192, 256, "bf16"), (3, 1024, 128, "bf16")),    # 2^21-element planes (two groups), then 2^17
    ((2, 512, 64, "i32"), (5, 2048, 64, "i32")),         # integer mode (generic engine), exact
    ((3, 64, 64, "f32"), (1, 1 << 16, 64, "f32")),       # one-tile plane, then the largest allowed plane (2^22)
    ((96, 512, 128, "bf16"), (2, 256, 64, "bf16")),      # one plane per CTA (2^16, no scratch), then 2^14
]


def noalloc(lib, x, g, y, dt, stream):
    B, N, C = x.shape
    rc = lib.whtmix_forward_noalloc(x.data_ptr(), g.data_ptr(), y.data_ptr(), B, N, C, CODE[dt], stream)
    assert rc == 0, f"whtmix_forward_noalloc [{B},{N},{C}] {dt} returned {rc}"


@pytest.mark.parametrize("first,second", PAIRS, ids=lambda c: "x".join(map(str, c)))
def test_noalloc_matches_forward_on_two_consecutive_calls(lib, first, second):
    stream = torch.cuda.current_stream().cuda_stream
    cases = []
    for k, (B, N, C, dt) in enumerate((first, second)):
        x, g = device_inputs(B, N, C, dt, seed=100 + 7 * k + B)
        cases.append((x, g, torch.empty_like(x), dt))
    for x, g, y, dt in cases:   # the two calls back to back on one stream
        noalloc(lib, x, g, y, dt, stream)
    torch.cuda.synchronize()
    assert lib.whtmix_sync(ctypes.c_void_p(stream)) == 0
    for x, g, y, dt in cases:
        B, N, C = x.shape
        want = torch.empty_like(x)
        rc = lib.whtmix_forward(x.data_ptr(), g.data_ptr(), want.data_ptr(), B, N, C, CODE[dt], stream)
        assert rc == 0
        torch.cuda.synchronize()
        assert_matches(y, want, dt, f"[{B},{N},{C}] {dt}")


def test_noalloc_allocates_no_device_memory(lib):
    """After a first round of calls (which loads the kernels), further calls of every kind,
    the largest plane included, leave the device's free memory exactly where it was."""
    stream = torch.cuda.current_stream().cuda_stream
    cases = []
    for k, (B, N, C, dt) in enumerate([c for pair in PAIRS for c in pair]):
        x, g = device_inputs(B, N, C, dt, seed=300 + k)
        cases.append((x, g, torch.empty_like(x), dt))
    for x, g, y, dt in cases:
        noalloc(lib, x, g, y, dt, stream)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(3):
        for x, g, y, dt in cases:
            noalloc(lib, x, g, y, dt, stream)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0, f"device free memory changed by {free0 - free1} bytes across no-allocation calls"
    assert lib.whtmix_sync(ctypes.c_void_p(stream)) == 0


def test_noalloc_rejects_planes_beyond_its_scratch(lib):
    # 2^23-element planes need 32 MiB of scratch, more than the fixed 16 MiB: rejected, nothing written
    B, N, C = 1, 65536, 128
    x, g = device_inputs(B, N, C, "bf16", seed=1)
    y = torch.full_like(x, 3.0)
    rc = lib.whtmix_forward_noalloc(x.data_ptr(), g.data_ptr(), y.data_ptr(), B, N, C, CODE["bf16"],
                                    torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    assert rc == 9
    assert (y.float() == 3.0).all().item()

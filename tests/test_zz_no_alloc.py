"""whtmix_forward_noalloc: the forward for callers that may not allocate device memory.

Such callers (a process whose device memory belongs to an outside allocator, a real-time loop, a
plugin handed only its buffers) cannot let the library allocate a workspace.  This entry point
keeps its scratch in a fixed array inside the library instead.  Here it is called through the C
ABI twice in a row per case -- the second call reuses the array the first one left behind -- and
each result is compared with whtmix_forward's on the same inputs, with the tolerances the parity
tests use (int32 exact, fp32 relative L2 <= 1e-6 and max abs <= 1e-5, bf16 relative L2 <= 1e-2).

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


# pairs of consecutive calls: (B, N, C, dtype) for the first and the second call
PAIRS = [
    ((4, 4096, 64, "f32"), (4, 4096, 64, "f32")),        # same shape, new inputs
    ((2, 8192, 256, "bf16"), (3, 1024, 128, "bf16")),    # 2^21-element planes, then a smaller shape
    ((2, 512, 64, "i32"), (5, 2048, 64, "i32")),         # integer mode, exact
    ((3, 64, 64, "f32"), (1, 1 << 16, 64, "f32")),       # one-tile plane, then the largest allowed plane (2^22)
]


@pytest.mark.parametrize("first,second", PAIRS, ids=lambda c: "x".join(map(str, c)))
def test_noalloc_matches_forward_on_two_consecutive_calls(lib, first, second):
    stream = torch.cuda.current_stream().cuda_stream
    results = []
    for k, (B, N, C, dt) in enumerate((first, second)):
        x, g = device_inputs(B, N, C, dt, seed=100 + 7 * k + B)
        y = torch.empty_like(x)
        rc = lib.whtmix_forward_noalloc(x.data_ptr(), g.data_ptr(), y.data_ptr(), B, N, C, CODE[dt], stream)
        assert rc == 0, f"whtmix_forward_noalloc returned {rc}"
        results.append((x, g, y, B, N, C, dt))
    torch.cuda.synchronize()
    for x, g, y, B, N, C, dt in results:
        want = torch.empty_like(x)
        rc = lib.whtmix_forward(x.data_ptr(), g.data_ptr(), want.data_ptr(), B, N, C, CODE[dt], stream)
        assert rc == 0
        torch.cuda.synchronize()
        assert_matches(y, want, dt, f"[{B},{N},{C}] {dt}")


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

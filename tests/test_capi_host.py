"""C-ABI checks that need no GPU: the library loads, exports every entry point include/whtmix.h
declares, and rejects bad arguments on the host before touching the device."""
import ctypes
import os
import re

import pytest
import torch

from paper_2607_25234_gb300 import build as libbuild
from paper_2607_25234_gb300 import whtmix

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "whtmix.h")


@pytest.fixture(scope="module")
def lib():
    libbuild.build()
    return whtmix.library()


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"WHTMIX_API\s+[\w\s\*]+?\b(whtmix_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_symbols()
    assert "whtmix_forward" in names and "whtmix_backward" in names
    assert set(names) == set(whtmix.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_symbols():
        assert hasattr(lib, name), name
    out = os.popen(f"nm -D --defined-only {libbuild.LIB}").read()
    exported = set(re.findall(r"\bT (whtmix_\w+)", out))
    assert exported == set(declared_symbols()), exported ^ set(declared_symbols())


def test_status_strings(lib):
    for code in range(10):
        assert lib.whtmix_status_string(code)
    assert lib.whtmix_status_string(0) == b"ok"
    assert lib.whtmix_status_string(12345) == b"unknown status"


def test_plan_and_workspace_sizes(lib):
    assert lib.whtmix_plan(256, 32) == 1      # 2^13 elements: one tile
    assert lib.whtmix_plan(256, 64) == 2      # 2^14: three phases
    assert lib.whtmix_plan(65536, 1024) == 2  # 2^26: largest three-phase plane
    assert lib.whtmix_plan(65536, 2048) == 3  # 2^27: five passes
    assert lib.whtmix_plan(1 << 16, 1 << 14) == 3  # 2^30: largest plane
    assert lib.whtmix_plan(1 << 16, 1 << 15) == 0  # 2^31: too large
    assert lib.whtmix_plan(3, 4) == 0
    ws = whtmix.workspace_bytes
    import torch
    assert ws(1, 256, 32, torch.float32) == 256
    assert ws(1, 65536, 128, torch.bfloat16) == 256 + (1 << 23) * 4
    # training step [16, 8192, 256]: forward groups of 8 planes, backward groups of 4 (two buffers)
    assert ws(16, 8192, 256, torch.bfloat16) == 256 + 8 * (1 << 21) * 4
    assert ws(16, 8192, 256, torch.bfloat16, backward=True) == 256 + 4 * 2 * (1 << 21) * 4
    assert ws(0, 4, 4, torch.float32, backward=True) == 256 + 16 * 4


FAKE = 1 << 20  # 16-byte aligned host integers posing as device pointers: never dereferenced
GPU_PRESENT = torch.cuda.is_available()


def passes_every_check(call):
    """A call whose arguments pass every host check stops at the device check (NO_DEVICE) on a
    machine without a GPU.  With a GPU it would launch on the fake pointers, so it is not made."""
    if not GPU_PRESENT:
        assert call() == 8


def fwd(lib, x=FAKE, g=2 * FAKE, y=3 * FAKE, B=1, N=4, C=4, dtype=0):
    return lib.whtmix_forward(x, g, y, B, N, C, dtype, None)


def bwd(lib, x=FAKE, g=2 * FAKE, dy=3 * FAKE, dx=4 * FAKE, dg=5 * FAKE, B=1, N=4, C=4, dtype=0):
    return lib.whtmix_backward(x, g, dy, dx, dg, B, N, C, dtype, None)


def test_rejects_invalid_arguments_before_any_device_work(lib):
    assert fwd(lib, x=None) == 1
    assert fwd(lib, g=None) == 1
    assert fwd(lib, y=None) == 1
    assert fwd(lib, B=-1) == 1
    assert fwd(lib, N=0) == 1
    assert fwd(lib, C=0) == 1
    assert fwd(lib, N=6) == 2
    assert fwd(lib, C=12) == 2
    assert fwd(lib, N=1 << 24, C=1 << 7) == 2         # 2^31 elements per plane
    assert fwd(lib, B=(1 << 56) + 1) == 2            # B*N*C above 2^60
    assert fwd(lib, N=1 << 13, C=1 << 13, B=(1 << 34) + 1) == 2
    far = 1 << 60                                     # 2^62 bytes of fp32 at 2^60 elements: no wrap
    passes_every_check(lambda: fwd(lib, x=far, y=far, B=1 << 56))
    assert fwd(lib, dtype=3) == 3
    assert fwd(lib, dtype=-1) == 3
    assert fwd(lib, x=FAKE + 4) == 4
    assert fwd(lib, y=3 * FAKE + 8) == 4
    assert bwd(lib, dy=None) == 1
    assert bwd(lib, dg=None) == 1
    assert bwd(lib, dg=5 * FAKE + 2) == 4


def test_alias_rules(lib):
    n = 4 * 4 * 4  # bytes of a [1, 4, 4] f32 plane
    assert fwd(lib, y=FAKE + 16) == 5                 # partial overlap with x
    assert fwd(lib, y=2 * FAKE) == 5                  # output on top of the gains
    assert bwd(lib, dx=3 * FAKE + 16) == 5            # partial overlap with dy
    assert bwd(lib, dx=FAKE) == 5                     # dx over x
    assert bwd(lib, dg=FAKE + 16) == 5                # dG inside x
    assert bwd(lib, dg=4 * FAKE) == 5                 # dG over dx
    assert bwd(lib, dg=2 * FAKE) == 5                 # dG over G
    # exact in-place is allowed: the call gets past every check
    passes_every_check(lambda: fwd(lib, y=FAKE))
    passes_every_check(lambda: bwd(lib, dx=3 * FAKE))
    del n


def test_empty_batch(lib):
    assert fwd(lib, B=0) == 0
    assert fwd(lib, x=None, g=None, y=None, B=0) == 0
    assert bwd(lib, B=0, dg=None) == 1
    assert bwd(lib, B=0, dg=5 * FAKE + 4) == 4
    import torch
    if not torch.cuda.is_available():
        assert bwd(lib, x=None, dy=None, dx=None, B=0) == 8  # would zero dG on a GPU


def test_ex_workspace_checks(lib):
    f = lib.whtmix_forward_ex
    need = ctypes.c_size_t(0)
    assert lib.whtmix_workspace_bytes(1, 256, 64, 0, 0, ctypes.byref(need)) == 0
    assert f(FAKE, 2 * FAKE, 3 * FAKE, 1, 256, 64, 0, None, need.value, None) == 9
    assert f(FAKE, 2 * FAKE, 3 * FAKE, 1, 256, 64, 0, 8 * FAKE + 16, need.value, None) == 9
    assert f(FAKE, 2 * FAKE, 3 * FAKE, 1, 256, 64, 0, 8 * FAKE, need.value - 1, None) == 9


def test_no_device_reported_on_a_cpu_box(lib):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    assert fwd(lib) == 8


def sfwd(lib, x=FAKE, gt=2 * FAKE, gc=2 * FAKE + 64, y=3 * FAKE, B=1, N=4, C=4, dtype=0, nv=None):
    return lib.whtmix_forward_separable(x, gt, gc, y, B, N if nv is None else nv, N, C, dtype, None)


def sbwd(lib, x=FAKE, gt=2 * FAKE, gc=2 * FAKE + 64, dy=3 * FAKE, dx=4 * FAKE, dgt=5 * FAKE, dgc=5 * FAKE + 64,
         B=1, N=4, C=4, dtype=0, nv=None):
    return lib.whtmix_backward_separable(x, gt, gc, dy, dx, dgt, dgc, B, N if nv is None else nv, N, C, dtype, None)


def test_separable_rejects_invalid_arguments_before_any_device_work(lib):
    assert sfwd(lib, dtype=2) == 3                    # int32: log-domain gains are real
    assert sbwd(lib, dtype=2) == 3
    assert sfwd(lib, gt=None) == 1
    assert sfwd(lib, gc=None) == 1
    assert sbwd(lib, dgt=None) == 1
    assert sbwd(lib, dgc=None) == 1
    assert sfwd(lib, N=6) == 2
    assert sfwd(lib, x=FAKE + 8) == 4
    assert sfwd(lib, gt=2 * FAKE + 2) == 4            # gains need 4-byte alignment only
    assert sbwd(lib, dgc=5 * FAKE + 66) == 4
    assert sfwd(lib, y=FAKE + 16) == 5                # partial overlap with x
    assert sfwd(lib, y=2 * FAKE - 16) == 5            # output over g_t
    assert sbwd(lib, dgt=FAKE + 16) == 5              # dg_t inside x
    assert sbwd(lib, dgc=5 * FAKE + 8) == 5           # dg_c over dg_t
    assert sbwd(lib, dx=FAKE) == 5                    # dx over x
    # gains 4-byte aligned and exact in-place pass the host checks and stop at the device
    passes_every_check(lambda: sfwd(lib, gt=2 * FAKE + 4, y=FAKE))
    passes_every_check(lambda: sbwd(lib, dx=3 * FAKE))
    assert sfwd(lib, B=0) == 0


def pfwd(lib, x=FAKE, g=2 * FAKE, y=3 * FAKE, B=1, nv=3, N=4, C=4, dtype=0):
    return lib.whtmix_forward_padded(x, g, y, B, nv, N, C, dtype, None)


def pbwd(lib, x=FAKE, g=2 * FAKE, dy=3 * FAKE, dx=4 * FAKE, dg=5 * FAKE, B=1, nv=3, N=4, C=4, dtype=0):
    return lib.whtmix_backward_padded(x, g, dy, dx, dg, B, nv, N, C, dtype, None)


def test_padded_rejects_invalid_arguments_before_any_device_work(lib):
    assert pfwd(lib, nv=5) == 1                       # more stored tokens than the padded plane
    assert pfwd(lib, nv=-1) == 1
    assert pfwd(lib, N=6) == 2                        # the padded length must be a power of two
    assert pfwd(lib, x=None) == 1
    assert pbwd(lib, dg=None) == 1
    assert pfwd(lib, y=FAKE + 16) == 5                # 3 x 4 f32 tokens = 48 bytes: overlaps x
    passes_every_check(lambda: pfwd(lib, y=FAKE + 48))  # right after x's stored tokens: no overlap
    assert pbwd(lib, dg=FAKE + 32) == 5
    assert pfwd(lib, nv=0) == 0 and pfwd(lib, B=0) == 0   # nothing stored: nothing to do
    assert sfwd(lib, nv=5) == 1
    assert sfwd(lib, nv=0) == 0


def test_noalloc_rejects_invalid_arguments_before_any_device_work(lib):
    nf = lib.whtmix_forward_noalloc
    assert nf(FAKE, 2 * FAKE, 3 * FAKE, 1, 1 << 32, 1 << 32, 0, None) == 2   # N*C = 2^64: no overflow
    assert nf(FAKE, 2 * FAKE, 3 * FAKE, 1, 1 << 62, 4, 0, None) == 2
    assert nf(FAKE, 2 * FAKE, 3 * FAKE, 1, 65536, 1024, 0, None) == 9      # 2^26: beyond the fixed scratch
    assert nf(FAKE, 2 * FAKE, 3 * FAKE, 1, 65536, 2048, 0, None) == 9      # 2^27 (five passes): likewise
    assert nf(FAKE, 2 * FAKE, 3 * FAKE, 1, 1 << 16, 1 << 15, 0, None) == 2  # 2^31: no plan
    assert nf(FAKE, 2 * FAKE, 3 * FAKE, 1, 65536, 128, 1, None) == 9       # 2^23 bf16 (32 MiB of scratch)
    assert nf(FAKE, 2 * FAKE, 3 * FAKE, 1, 6, 4, 0, None) == 2
    assert nf(FAKE, 2 * FAKE, 3 * FAKE, -1, 4, 4, 0, None) == 1
    assert nf(FAKE, 2 * FAKE, 3 * FAKE, 1, 4, 4, 7, None) == 3
    assert nf(None, None, None, 0, 4, 4, 0, None) == 0                     # nothing to do
    if not GPU_PRESENT:
        assert nf(FAKE, 2 * FAKE, 3 * FAKE, 1, 4, 4, 0, None) == 8         # valid: stops at the device


def test_project_and_block_reject_invalid_arguments_before_any_device_work(lib):
    P = lib.whtmix_project
    assert P(FAKE, 2 * FAKE, 3 * FAKE, 1, 96, 1, None) == 2        # C must be 64, 128 or 256
    assert P(FAKE, 2 * FAKE, 3 * FAKE, 1, 64, 2, None) == 3        # output fp32 or bf16
    assert P(FAKE, 2 * FAKE, 3 * FAKE, -1, 64, 1, None) == 1
    assert P(FAKE, 2 * FAKE, 3 * FAKE, (1 << 54) + 1, 64, 1, None) == 2   # T*C above 2^60
    assert P(None, 2 * FAKE, 3 * FAKE, 1, 64, 1, None) == 1
    assert P(FAKE + 8, 2 * FAKE, 3 * FAKE, 1, 64, 1, None) == 4
    assert P(FAKE, 2 * FAKE, FAKE + 16, 4, 64, 1, None) == 5       # partial overlap with x
    assert P(FAKE, 2 * FAKE, 2 * FAKE, 4, 64, 1, None) == 5        # output over w
    assert P(FAKE, 2 * FAKE, FAKE, 4, 64, 0, None) == 5            # in place only with bf16 output
    assert P(FAKE, 2 * FAKE, 3 * FAKE, 0, 64, 1, None) == 0        # no tokens
    Bk = lib.whtmix_block_forward
    assert Bk(FAKE, 2 * FAKE, 3 * FAKE, 4 * FAKE, 5 * FAKE, 1, 4, 64, 0, None) == 3   # bf16 only
    assert Bk(FAKE, 2 * FAKE, 3 * FAKE, 4 * FAKE, 5 * FAKE, 1, 4, 32, 1, None) == 2   # C 64, 128 or 256
    assert Bk(FAKE, 2 * FAKE, 3 * FAKE, 4 * FAKE, 2 * FAKE, 1, 4, 64, 1, None) == 5   # y over w_in
    assert Bk(FAKE, 2 * FAKE, 3 * FAKE, 4 * FAKE, 5 * FAKE, 0, 4, 64, 1, None) == 0


def test_binding_refuses_cpu_tensors_and_malformed_outputs(monkeypatch):
    """The torch binding has no CPU path: every public op raises on CPU tensors before it reaches
    the library, and a caller-supplied output must be exactly the tensor the library writes."""
    import torch

    def no_library(*_a, **_k):
        raise AssertionError("the library was reached")

    monkeypatch.setattr(whtmix, "library", no_library)
    x = torch.zeros(2, 16, 8)
    g = torch.ones(16, 8)
    xb = x.to(torch.bfloat16)
    w = torch.zeros(8, 8, dtype=torch.bfloat16)
    gt, gc = torch.zeros(16), torch.zeros(8)
    calls = [
        lambda: whtmix.forward(x, g),
        lambda: whtmix.forward_noalloc(x, g),
        lambda: whtmix.backward(x, g, x),
        lambda: whtmix.forward_ex(x, g, torch.zeros(64)),
        lambda: whtmix.backward_ex(x, g, x, torch.zeros(64)),
        lambda: whtmix.forward_padded(x[:, :12], g),
        lambda: whtmix.backward_padded(x[:, :12].contiguous(), g, x[:, :12].contiguous()),
        lambda: whtmix.forward_separable(x, gt, gc),
        lambda: whtmix.backward_separable(x, gt, gc, x),
        lambda: whtmix.project(xb, w),
        lambda: whtmix.block_forward(xb, w, g, w),
        lambda: whtmix.WHTMixFunction.apply(x, g),
    ]
    for call in calls:
        with pytest.raises(ValueError, match="CUDA"):
            call()

    dev = torch.device("cpu")
    assert whtmix._out(None, (2, 3), torch.float32, dev, "out").shape == (2, 3)
    with pytest.raises(ValueError, match=r"out must be torch.float32 \[2, 3\]"):
        whtmix._out(torch.zeros(3, 2), (2, 3), torch.float32, dev, "out")
    with pytest.raises(ValueError, match="dx must be torch.bfloat16"):
        whtmix._out(torch.zeros(2, 3), (2, 3), torch.bfloat16, dev, "dx")
    with pytest.raises(ValueError, match="CUDA tensor"):
        whtmix._out(torch.zeros(2, 3), (2, 3), torch.float32, dev, "out")


def test_pad_tokens_helper():
    """whtmix.pad_tokens is plain tensor bookkeeping (no mixer arithmetic): zero rows appended on
    the token axis up to the next power of two, the stored rows unchanged."""
    import torch
    x = torch.arange(2 * 5 * 3, dtype=torch.float32).reshape(2, 5, 3)
    p = whtmix.pad_tokens(x)
    assert p.shape == (2, 8, 3) and p.is_contiguous()
    assert torch.equal(p[:, :5], x) and torch.count_nonzero(p[:, 5:]) == 0
    assert whtmix.pad_tokens(x, 16).shape == (2, 16, 3)
    assert whtmix.pad_tokens(x[0]).shape == (8, 3)                     # a single [N, C] plane
    assert torch.equal(whtmix.pad_tokens(x[:, :4]), x[:, :4])          # already a power of two
    assert whtmix.pad_tokens(torch.zeros(2, 0, 3)).shape == (2, 1, 3)  # no tokens: one zero row
    assert whtmix.pad_tokens(torch.zeros(2, 64800, 1)).shape == (2, 65536, 1)
    for bad in (4, 12):
        with pytest.raises(ValueError):
            whtmix.pad_tokens(x, bad)


def xfwd(lib, x=FAKE, g=2 * FAKE, y=3 * FAKE, B=1, N=4, C=4, dtype=0):
    return lib.whtmix_forward_x16(x, g, y, B, N, C, dtype, None)


def test_x16_checks_its_arguments_as_the_forward_does(lib):
    # whtmix_forward_x16 goes through the forward's host checks: the same status for every case
    cases = [dict(x=None), dict(g=None), dict(y=None), dict(B=-1), dict(N=0), dict(N=6), dict(C=12),
             dict(N=1 << 24, C=1 << 7), dict(B=(1 << 56) + 1), dict(dtype=3), dict(x=FAKE + 4),
             dict(y=3 * FAKE + 8), dict(y=FAKE + 16), dict(y=2 * FAKE), dict(B=0),
             dict(x=None, g=None, y=None, B=0)]
    for kw in cases:
        assert xfwd(lib, **kw) == fwd(lib, **kw), kw
    passes_every_check(lambda: xfwd(lib, y=FAKE))                     # exact in place
    passes_every_check(lambda: xfwd(lib, N=65536, C=128, dtype=1, x=FAKE, g=(1 << 40), y=(1 << 41)))

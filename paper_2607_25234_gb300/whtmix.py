"""Python binding of the WHTMix C ABI (``include/whtmix.h``): argument marshalling only.

Every step of the mixer runs in the CUDA library ``_lib/libwhtmix.so``; this module passes device
pointers, sizes and the current CUDA stream through ctypes.  torch supplies device memory and
streams.  There is no CPU path: a missing library or a CPU tensor raises.

The operation (paper Section III-B, Eq. 1-4): Y_b = H_N (G (.) H_N X_b H_C) H_C / (N C) for every
plane X_b [N, C] of X [B, N, C]; the backward returns dX and dG = sum_b (H X_b H)(H dY_b H)/(N C).
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

__all__ = ["forward", "backward", "forward_ex", "backward_ex", "forward_noalloc", "forward_separable",
           "backward_separable",
           "forward_padded", "backward_padded", "project", "block_forward",
           "block_backward", "workspace_bytes", "sync", "plan", "release_workspaces", "WhtmixError", "WHTMixFunction",
           "WHTMixSeparableFunction", "WHTMixBlockFunction", "pad_tokens", "EXPORTS", "library"]

# status codes and dtype codes of include/whtmix.h
OK = 0
STATUS = {0: "OK", 1: "INVALID_ARG", 2: "BAD_SHAPE", 3: "BAD_DTYPE", 4: "MISALIGNED", 5: "ALIAS",
          6: "CUDA", 7: "TIMEOUT", 8: "NO_DEVICE", 9: "WORKSPACE"}
DTYPE_CODE = {torch.float32: 0, torch.bfloat16: 1, torch.int32: 2}
GAIN_DTYPE = {torch.float32: torch.float32, torch.bfloat16: torch.float32, torch.int32: torch.int32}

# every entry point include/whtmix.h declares
EXPORTS = ("whtmix_forward", "whtmix_backward", "whtmix_workspace_bytes", "whtmix_forward_ex",
           "whtmix_backward_ex", "whtmix_sync", "whtmix_release_workspaces", "whtmix_status_string",
           "whtmix_last_cuda_error", "whtmix_plan", "whtmix_forward_noalloc", "whtmix_forward_separable",
           "whtmix_backward_separable", "whtmix_forward_padded", "whtmix_backward_padded", "whtmix_project",
           "whtmix_block_forward", "whtmix_block_backward", "whtmix_forward_x16")


class WhtmixError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: WHTMIX_{'ERR_' if status else ''}{STATUS.get(status, status)} ({status})")


_lock = threading.Lock()
_lib = None


def library(path: str | None = None) -> ctypes.CDLL:
    """Load the C library (built by ``__graft_entry__.build()``); raises if it is missing."""
    global _lib
    with _lock:
        if _lib is None:
            path = path or _build.LIB
            if not os.path.exists(path):
                raise RuntimeError(f"WHTMix CUDA library not built ({path}); run __graft_entry__.build()")
            lib = ctypes.CDLL(path)
            i64, p, i, sz = ctypes.c_int64, ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
            lib.whtmix_forward.argtypes = [p, p, p, i64, i64, i64, i, p]
            lib.whtmix_backward.argtypes = [p, p, p, p, p, i64, i64, i64, i, p]
            lib.whtmix_forward_ex.argtypes = [p, p, p, i64, i64, i64, i, p, sz, p]
            lib.whtmix_forward_noalloc.argtypes = [p, p, p, i64, i64, i64, i, p]
            lib.whtmix_forward_x16.argtypes = [p, p, p, i64, i64, i64, i, p]
            lib.whtmix_backward_ex.argtypes = [p, p, p, p, p, i64, i64, i64, i, p, sz, p]
            lib.whtmix_workspace_bytes.argtypes = [i64, i64, i64, i, i, ctypes.POINTER(sz)]
            lib.whtmix_sync.argtypes = [p]
            lib.whtmix_release_workspaces.argtypes = []
            lib.whtmix_status_string.argtypes = [i]
            lib.whtmix_status_string.restype = ctypes.c_char_p
            lib.whtmix_last_cuda_error.argtypes = []
            lib.whtmix_plan.argtypes = [i64, i64]
            lib.whtmix_forward_separable.argtypes = [p, p, p, p, i64, i64, i64, i64, i, p]
            lib.whtmix_backward_separable.argtypes = [p, p, p, p, p, p, p, i64, i64, i64, i64, i, p]
            lib.whtmix_forward_padded.argtypes = [p, p, p, i64, i64, i64, i64, i, p]
            lib.whtmix_project.argtypes = [p, p, p, i64, i64, i, p]
            lib.whtmix_block_forward.argtypes = [p, p, p, p, p, i64, i64, i64, i, p]
            lib.whtmix_block_backward.argtypes = [p, p, p, p, p, p, p, p, p, i64, i64, i64, i, p]
            lib.whtmix_backward_padded.argtypes = [p, p, p, p, p, i64, i64, i64, i64, i, p]
            for name in EXPORTS:
                if name != "whtmix_status_string":
                    getattr(lib, name).restype = ctypes.c_int
            _lib = lib
    return _lib


def _check(rc: int, what: str):
    if rc != OK:
        if rc == 6:
            what += f" (cudaError {library().whtmix_last_cuda_error()})"
        raise WhtmixError(rc, what)


def _call(what: str, device: torch.device, stream, fn, *args) -> None:
    """Runs one entry point with ``device`` current, on ``stream`` (default: the device's current
    stream, appended as the last argument); raises WhtmixError on a nonzero status."""
    if device.index != torch.cuda.current_device():
        with torch.cuda.device(device):
            return _call(what, device, stream, fn, *args)
    s = stream if stream is not None else torch.cuda.current_stream(device)
    if s.device != device:
        raise ValueError(f"stream is on {s.device}, the tensors on {device}")
    _check(fn(*args, int(s.cuda_stream)), what)


def _on_device(t: torch.Tensor, device: torch.device, name: str) -> None:
    if not t.is_cuda or t.device != device:
        raise ValueError(f"{name} must be a CUDA tensor on {device} (WHTMix runs on CUDA tensors only)")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def _out(t: torch.Tensor | None, shape, dtype: torch.dtype, device: torch.device, name: str) -> torch.Tensor:
    """A result tensor: a new one, or the caller's, checked to be exactly what the library writes
    (the C ABI receives only its pointer)."""
    if t is None:
        return torch.empty(tuple(shape), dtype=dtype, device=device)
    if t.dtype != dtype or tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must be {dtype} {list(shape)}, got {t.dtype} {list(t.shape)}")
    _on_device(t, device, name)
    return t


def _shape(x: torch.Tensor):
    if x.dim() == 2:
        return 1, x.shape[0], x.shape[1]
    if x.dim() != 3:
        raise ValueError("x must be [N, C] or [B, N, C]")
    return tuple(x.shape)


def _check_tensors(x: torch.Tensor, g: torch.Tensor, *others: torch.Tensor):
    if x.dtype not in DTYPE_CODE:
        raise TypeError(f"unsupported dtype {x.dtype}; expected float32, bfloat16 or int32")
    B, N, C = _shape(x)
    if g.dtype != GAIN_DTYPE[x.dtype]:
        raise TypeError(f"gains must be {GAIN_DTYPE[x.dtype]} for {x.dtype} inputs")
    if tuple(g.shape) != (N, C):
        raise ValueError(f"gains must be [N, C] = [{N}, {C}], got {tuple(g.shape)}")
    for t in (x, g) + others:
        _on_device(t, x.device, "every tensor")
    return B, N, C


def forward(x: torch.Tensor, g: torch.Tensor, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Y = H_N (G (.) H_N X H_C) H_C / (N C) per plane (unnormalised, mod 2^32, for int32)."""
    B, N, C = _check_tensors(x, g)
    y = _out(out, x.shape, x.dtype, x.device, "out")
    _call("whtmix_forward", x.device, stream, library().whtmix_forward, x.data_ptr(), g.data_ptr(), y.data_ptr(),
          B, N, C, DTYPE_CODE[x.dtype])
    return y


def forward_x16(x: torch.Tensor, g: torch.Tensor, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """forward whose three-phase kernel rounds the exchanged intermediate plane to bf16 (half the
    workspace traffic; butterflies and gain in fp32); other shapes run exactly as forward."""
    B, N, C = _check_tensors(x, g)
    y = _out(out, x.shape, x.dtype, x.device, "out")
    _call("whtmix_forward_x16", x.device, stream, library().whtmix_forward_x16, x.data_ptr(), g.data_ptr(),
          y.data_ptr(), B, N, C, DTYPE_CODE[x.dtype])
    return y


def forward_noalloc(x: torch.Tensor, g: torch.Tensor, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """forward without any device allocation: planes of more than 2^22 elements raise WORKSPACE.
    Calls share one fixed scratch array per device, so order them on one stream; make the first
    call on a device outside any stream capture."""
    B, N, C = _check_tensors(x, g)
    y = _out(out, x.shape, x.dtype, x.device, "out")
    _call("whtmix_forward_noalloc", x.device, stream, library().whtmix_forward_noalloc, x.data_ptr(), g.data_ptr(),
          y.data_ptr(), B, N, C, DTYPE_CODE[x.dtype])
    return y


def backward(x: torch.Tensor, g: torch.Tensor, dy: torch.Tensor, dx: torch.Tensor | None = None,
             dg: torch.Tensor | None = None, stream=None):
    """(dX, dG) of the forward map; dG is summed over the batch in ascending order."""
    B, N, C = _check_tensors(x, g, dy)
    if dy.shape != x.shape or dy.dtype != x.dtype:
        raise ValueError("dy must match x in shape and dtype")
    dx = _out(dx, x.shape, x.dtype, x.device, "dx")
    dg = _out(dg, g.shape, g.dtype, x.device, "dg")
    _call("whtmix_backward", x.device, stream, library().whtmix_backward, x.data_ptr(), g.data_ptr(), dy.data_ptr(),
          dx.data_ptr(), dg.data_ptr(), B, N, C, DTYPE_CODE[x.dtype])
    return dx, dg


def _check_log_gains(x: torch.Tensor, g_t: torch.Tensor, g_c: torch.Tensor, *others: torch.Tensor):
    """(B, N_valid, N, C): x holds N_valid tokens per plane, g_t has the padded length N."""
    if x.dtype not in (torch.float32, torch.bfloat16):
        raise TypeError(f"separable gains need float32 or bfloat16 inputs, got {x.dtype}")
    B, n_valid, C = _shape(x)
    if g_t.dtype != torch.float32 or g_c.dtype != torch.float32 or g_t.dim() != 1:
        raise TypeError("log gains must be 1D float32 tensors")
    N = g_t.shape[0]
    if N & (N - 1) or N < max(n_valid, 1):
        raise ValueError(f"g_t must have a power-of-two length >= the {n_valid} tokens of x, got {N}")
    if tuple(g_c.shape) != (C,):
        raise ValueError(f"log gains must be g_t [{N}] and g_c [{C}], got {tuple(g_t.shape)} and {tuple(g_c.shape)}")
    for t in (x, g_t, g_c) + others:
        _on_device(t, x.device, "every tensor")
    return B, n_valid, N, C


def forward_separable(x: torch.Tensor, g_t: torch.Tensor, g_c: torch.Tensor, out: torch.Tensor | None = None,
                      stream=None) -> torch.Tensor:
    """The forward with the paper's log-domain gains (Section III-B, Eq. 2-3):
    G[n, c] = exp(g_t[n]) exp(g_c[c]).  When x has fewer tokens than g_t (not a power of two), the
    planes are zero-padded to len(g_t) tokens inside the library and y keeps x's tokens."""
    B, n_valid, N, C = _check_log_gains(x, g_t, g_c)
    y = _out(out, x.shape, x.dtype, x.device, "out")
    _call("whtmix_forward_separable", x.device, stream, library().whtmix_forward_separable, x.data_ptr(),
          g_t.data_ptr(), g_c.data_ptr(), y.data_ptr(), B, n_valid, N, C, DTYPE_CODE[x.dtype])
    return y


def backward_separable(x: torch.Tensor, g_t: torch.Tensor, g_c: torch.Tensor, dy: torch.Tensor,
                       dx: torch.Tensor | None = None, dg_t: torch.Tensor | None = None,
                       dg_c: torch.Tensor | None = None, stream=None):
    """(dX, dg_t, dg_c) of forward_separable."""
    B, n_valid, N, C = _check_log_gains(x, g_t, g_c, dy)
    if dy.shape != x.shape or dy.dtype != x.dtype:
        raise ValueError("dy must match x in shape and dtype")
    dx = _out(dx, x.shape, x.dtype, x.device, "dx")
    dg_t = _out(dg_t, g_t.shape, g_t.dtype, x.device, "dg_t")
    dg_c = _out(dg_c, g_c.shape, g_c.dtype, x.device, "dg_c")
    _call("whtmix_backward_separable", x.device, stream, library().whtmix_backward_separable, x.data_ptr(),
          g_t.data_ptr(), g_c.data_ptr(), dy.data_ptr(), dx.data_ptr(), dg_t.data_ptr(), dg_c.data_ptr(), B,
          n_valid, N, C, DTYPE_CODE[x.dtype])
    return dx, dg_t, dg_c


def _check_padded(x: torch.Tensor, g: torch.Tensor, *others: torch.Tensor):
    """(B, N_valid, N, C) for a padded call: x holds N_valid tokens, g is the padded [N, C]."""
    if x.dtype not in DTYPE_CODE:
        raise TypeError(f"unsupported dtype {x.dtype}; expected float32, bfloat16 or int32")
    B, n_valid, C = _shape(x)
    if g.dtype != GAIN_DTYPE[x.dtype] or g.dim() != 2 or g.shape[1] != C:
        raise ValueError(f"gains must be {GAIN_DTYPE[x.dtype]} [N, {C}]")
    N = g.shape[0]
    if N & (N - 1) or N < max(n_valid, 1):
        raise ValueError(f"gains must have a power-of-two token count >= the {n_valid} tokens of x, got {N}")
    for t in (x, g) + others:
        _on_device(t, x.device, "every tensor")
    return B, n_valid, N, C


def forward_padded(x: torch.Tensor, g: torch.Tensor, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """The forward on planes zero-padded from x's N_valid tokens to g's N (a power of two), inside the
    library; y keeps x's N_valid tokens (Section III-B: pad before H_N, discard the padded outputs)."""
    B, n_valid, N, C = _check_padded(x, g)
    y = _out(out, x.shape, x.dtype, x.device, "out")
    _call("whtmix_forward_padded", x.device, stream, library().whtmix_forward_padded, x.data_ptr(), g.data_ptr(),
          y.data_ptr(), B, n_valid, N, C, DTYPE_CODE[x.dtype])
    return y


def backward_padded(x: torch.Tensor, g: torch.Tensor, dy: torch.Tensor, dx: torch.Tensor | None = None,
                    dg: torch.Tensor | None = None, stream=None):
    """(dX, dG) of forward_padded; dX keeps x's tokens, dG is the padded [N, C]."""
    B, n_valid, N, C = _check_padded(x, g, dy)
    if dy.shape != x.shape or dy.dtype != x.dtype:
        raise ValueError("dy must match x in shape and dtype")
    dx = _out(dx, x.shape, x.dtype, x.device, "dx")
    dg = _out(dg, g.shape, g.dtype, x.device, "dg")
    _call("whtmix_backward_padded", x.device, stream, library().whtmix_backward_padded, x.data_ptr(), g.data_ptr(),
          dy.data_ptr(), dx.data_ptr(), dg.data_ptr(), B, n_valid, N, C, DTYPE_CODE[x.dtype])
    return dx, dg


def project(x: torch.Tensor, w: torch.Tensor, out_dtype: torch.dtype = torch.bfloat16,
            out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """z = x w^T per token on the tensor cores (x [..., C] bf16, w [C, C] bf16 as (out, in))."""
    if x.dtype != torch.bfloat16 or w.dtype != torch.bfloat16:
        raise TypeError("project takes bfloat16 x and w")
    if out_dtype not in (torch.float32, torch.bfloat16):
        raise TypeError(f"project writes float32 or bfloat16, not {out_dtype}")
    C = x.shape[-1]
    if tuple(w.shape) != (C, C):
        raise ValueError(f"w must be [{C}, {C}]")
    for t in (x, w):
        _on_device(t, x.device, "x and w")
    z = _out(out, x.shape, out_dtype, x.device, "out")
    _call("whtmix_project", x.device, stream, library().whtmix_project, x.data_ptr(), w.data_ptr(), z.data_ptr(),
          x.numel() // C, C, DTYPE_CODE[out_dtype])
    return z


def block_forward(x: torch.Tensor, w_in: torch.Tensor, g: torch.Tensor, w_out: torch.Tensor,
                  out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """The mixer block of Section III-B, Eq. 1-4: Y = mix(X W_in^T) W_out^T (bf16)."""
    B, N, C = _check_tensors(x, g)
    for t in (w_in, w_out):
        if t.dtype != torch.bfloat16 or tuple(t.shape) != (C, C):
            raise ValueError(f"w_in and w_out must be bfloat16 [{C}, {C}]")
        _on_device(t, x.device, "w_in and w_out")
    y = _out(out, x.shape, x.dtype, x.device, "out")
    _call("whtmix_block_forward", x.device, stream, library().whtmix_block_forward, x.data_ptr(), w_in.data_ptr(),
          g.data_ptr(), w_out.data_ptr(), y.data_ptr(), B, N, C, DTYPE_CODE[x.dtype])
    return y


def block_backward(x: torch.Tensor, w_in: torch.Tensor, g: torch.Tensor, w_out: torch.Tensor, dy: torch.Tensor,
                   dx: torch.Tensor | None = None, dw_in: torch.Tensor | None = None, dg: torch.Tensor | None = None,
                   dw_out: torch.Tensor | None = None, stream=None):
    """(dX, dW_in, dG, dW_out) of block_forward for the upstream gradient dy (bf16); the gain and
    weight gradients are float32."""
    B, N, C = _check_tensors(x, g, dy)
    if dy.shape != x.shape or dy.dtype != x.dtype:
        raise ValueError("dy must match x in shape and dtype")
    for t in (w_in, w_out):
        if t.dtype != torch.bfloat16 or tuple(t.shape) != (C, C):
            raise ValueError(f"w_in and w_out must be bfloat16 [{C}, {C}]")
        _on_device(t, x.device, "w_in and w_out")
    dx = _out(dx, x.shape, x.dtype, x.device, "dx")
    dw_in = _out(dw_in, (C, C), torch.float32, x.device, "dw_in")
    dg = _out(dg, g.shape, torch.float32, x.device, "dg")
    dw_out = _out(dw_out, (C, C), torch.float32, x.device, "dw_out")
    _call("whtmix_block_backward", x.device, stream, library().whtmix_block_backward, x.data_ptr(), w_in.data_ptr(),
          g.data_ptr(), w_out.data_ptr(), dy.data_ptr(), dx.data_ptr(), dw_in.data_ptr(), dg.data_ptr(),
          dw_out.data_ptr(), B, N, C, DTYPE_CODE[x.dtype])
    return dx, dw_in, dg, dw_out


def workspace_bytes(B: int, N: int, C: int, dtype: torch.dtype, backward: bool = False) -> int:
    out = ctypes.c_size_t(0)
    _check(library().whtmix_workspace_bytes(B, N, C, DTYPE_CODE[dtype], int(backward), ctypes.byref(out)),
           "whtmix_workspace_bytes")
    return out.value


def forward_ex(x, g, workspace: torch.Tensor, out=None, stream=None):
    """forward with a caller-owned workspace of at least workspace_bytes(...) bytes."""
    B, N, C = _check_tensors(x, g, workspace)
    y = _out(out, x.shape, x.dtype, x.device, "out")
    _call("whtmix_forward_ex", x.device, stream, library().whtmix_forward_ex, x.data_ptr(), g.data_ptr(),
          y.data_ptr(), B, N, C, DTYPE_CODE[x.dtype], workspace.data_ptr(),
          workspace.numel() * workspace.element_size())
    return y


def backward_ex(x, g, dy, workspace: torch.Tensor, dx=None, dg=None, stream=None):
    """backward with a caller-owned workspace of at least workspace_bytes(..., backward=True) bytes."""
    B, N, C = _check_tensors(x, g, dy, workspace)
    if dy.shape != x.shape or dy.dtype != x.dtype:
        raise ValueError("dy must match x in shape and dtype")
    dx = _out(dx, x.shape, x.dtype, x.device, "dx")
    dg = _out(dg, g.shape, g.dtype, x.device, "dg")
    _call("whtmix_backward_ex", x.device, stream, library().whtmix_backward_ex, x.data_ptr(), g.data_ptr(),
          dy.data_ptr(), dx.data_ptr(), dg.data_ptr(), B, N, C, DTYPE_CODE[x.dtype], workspace.data_ptr(),
          workspace.numel() * workspace.element_size())
    return dx, dg


def sync(stream=None) -> None:
    """Synchronise the stream and raise if a device-side bounded wait expired."""
    s = stream if stream is not None else torch.cuda.current_stream()
    _call("whtmix_sync", s.device, s, library().whtmix_sync)


def release_workspaces() -> None:
    _check(library().whtmix_release_workspaces(), "whtmix_release_workspaces")


def plan(N: int, C: int) -> int:
    return library().whtmix_plan(N, C)


def pad_tokens(x: torch.Tensor, n_pad: int | None = None) -> torch.Tensor:
    """Zero-pads the token axis (dim -2) to ``n_pad`` tokens (default: the next power of two, at
    least 1), as the paper does before H_N (Section III-B).  Crop the mixer's output back with
    ``y[..., :n, :]``."""
    n = x.shape[-2]
    target = (1 << max(n - 1, 0).bit_length()) if n_pad is None else n_pad
    if target < max(n, 1) or target & (target - 1):
        raise ValueError(f"n_pad must be a power of two >= the {n} tokens of x, got {target}")
    if target == n:
        return x.contiguous()
    pad = torch.zeros(*x.shape[:-2], target - n, x.shape[-1], dtype=x.dtype, device=x.device)
    return torch.cat([x, pad], dim=-2).contiguous()


class WHTMixFunction(torch.autograd.Function):
    """autograd wrapper: forward and backward both run in the CUDA library."""

    @staticmethod
    def forward(ctx, x, g):
        x, g = x.contiguous(), g.contiguous()
        ctx.save_for_backward(x, g)
        return forward(x, g)

    @staticmethod
    def backward(ctx, dy):
        x, g = ctx.saved_tensors
        dx, dg = backward(x, g, dy.contiguous())
        return dx, dg


class WHTMixSeparableFunction(torch.autograd.Function):
    """autograd wrapper for the log-domain gains: forward and backward both run in the CUDA library."""

    @staticmethod
    def forward(ctx, x, g_t, g_c):
        x, g_t, g_c = x.contiguous(), g_t.contiguous(), g_c.contiguous()
        ctx.save_for_backward(x, g_t, g_c)
        return forward_separable(x, g_t, g_c)

    @staticmethod
    def backward(ctx, dy):
        x, g_t, g_c = ctx.saved_tensors
        return backward_separable(x, g_t, g_c, dy.contiguous())


class WHTMixBlockFunction(torch.autograd.Function):
    """autograd wrapper of the whole block (W_in, mixer, W_out): forward and backward both run in
    the CUDA library; the weight and gain gradients come back in float32."""

    @staticmethod
    def forward(ctx, x, w_in, g, w_out):
        x, w_in, g, w_out = x.contiguous(), w_in.contiguous(), g.contiguous(), w_out.contiguous()
        ctx.save_for_backward(x, w_in, g, w_out)
        return block_forward(x, w_in, g, w_out)

    @staticmethod
    def backward(ctx, dy):
        x, w_in, g, w_out = ctx.saved_tensors
        dx, dw_in, dg, dw_out = block_backward(x, w_in, g, w_out, dy.contiguous())
        return dx, dw_in.to(w_in.dtype), dg, dw_out.to(w_out.dtype)

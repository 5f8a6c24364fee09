"""ctypes binding of libslorr (include/slorr.h): argument marshalling only.

Every step of the regularizer runs inside libslorr's CUDA kernels; this module
only converts Python values into the C ABI's structs and pointers.  PyTorch is
used (by ``Regularizer``) for device memory and the current stream.  There is
no fallback: if libslorr.so is missing, loading raises.
"""

from __future__ import annotations

import ctypes
import os
import re

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libslorr.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "slorr.h")

SLORR_OK = 0
STATUS_NAMES = {0: "OK", 1: "INVALID_ARG", 2: "UNSUPPORTED", 3: "CUDA", 4: "WORKSPACE",
                5: "TIMEOUT", 6: "NONFINITE"}
VARIANTS = {"hoyer": 0, "nuclear": 1}
COMPUTES = {"fp16": 0, "bf16": 1, "fp32": 2, "bf16_split": 3}
DTYPES = {"f32": 0, "bf16": 1}
FLAG_SIMT_GEMM = 1
FLAG_TEST_STALL = 16
FLAG_WRITE_GRAD = 32
FLAG_NO_PDL = 512
FLAG_SEPARATE_NORM = 1024
FLAG_NO_SPLIT_K = 2048
FLAG_GRAPH = 4096
FLAG_PHASE_LAUNCHES = 16384
FLAG_DATAFLOW = 32768


class SlorrError(RuntimeError):
    def __init__(self, status: int, message: str):
        self.status = status
        super().__init__(f"libslorr: {STATUS_NAMES.get(status, status)}: {message}")


class Shape(ctypes.Structure):
    _fields_ = [("m", ctypes.c_int64), ("n", ctypes.c_int64)]


class Options(ctypes.Structure):
    _fields_ = [("variant", ctypes.c_int32), ("compute", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("iters", ctypes.c_int32), ("ell", ctypes.c_double), ("cushion", ctypes.c_double),
                ("safety", ctypes.c_double), ("lambda_", ctypes.c_float), ("eps", ctypes.c_float),
                ("grad_scale", ctypes.c_float), ("flags", ctypes.c_int32), ("timeout_s", ctypes.c_double)]


class MatrixView(ctypes.Structure):
    _fields_ = [("x", ctypes.c_void_p), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("ld", ctypes.c_int64), ("elem", ctypes.c_int32), ("transposed", ctypes.c_int32),
                ("frob_sq", ctypes.c_void_p), ("n_hat", ctypes.c_void_p), ("x0_scale", ctypes.c_void_p)]


_lib = None


def load_library(path: str | None = None) -> ctypes.CDLL:
    """Load libslorr.so (built in-tree by ``paper_2607_08754_gb300.build``)."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise ImportError(f"libslorr.so not found at {p}: run __graft_entry__.build() first")
    lib = ctypes.CDLL(p)
    vp, i32, i64, dbl = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
    sig = {
        "slorr_default_options": (None, [ctypes.POINTER(Options)]),
        "slorr_create": (i32, [ctypes.POINTER(vp), ctypes.POINTER(Shape), i32, ctypes.POINTER(Options)]),
        "slorr_workspace_size": (i32, [vp, ctypes.POINTER(ctypes.c_size_t)]),
        "slorr_reg_forward_backward": (i32, [vp, ctypes.POINTER(vp), ctypes.POINTER(vp), vp, vp, vp,
                                             ctypes.c_size_t, vp]),
        "slorr_reg_descent_step": (i32, [vp, ctypes.POINTER(vp), ctypes.c_float, vp, vp, vp, ctypes.c_size_t,
                                         vp]),
        "slorr_reset_workspace": (i32, [vp]),
        "slorr_get_status": (i32, [vp, vp, vp]),
        "slorr_run_steps": (i32, [vp, ctypes.POINTER(vp), vp, ctypes.c_size_t, i32, vp]),
        "slorr_iterate_view": (i32, [vp, vp, i32, i32, ctypes.POINTER(MatrixView)]),
        "slorr_get_coefficients": (i32, [vp, ctypes.POINTER(dbl), i32]),
        "slorr_pe_coefficients": (i32, [i32, dbl, dbl, dbl, ctypes.POINTER(dbl)]),
        "slorr_cushion_ratio": (dbl, []),
        "slorr_flops": (i64, [ctypes.POINTER(Shape), i32, i32]),
        "slorr_partition": (i32, [ctypes.POINTER(Shape), i32, i32, i32, ctypes.POINTER(i32),
                                  ctypes.POINTER(i32)]),
        "slorr_executed_flops": (i32, [vp, ctypes.POINTER(dbl)]),
        "slorr_gemm_items": (i32, [vp, i32, ctypes.POINTER(i32)]),
        "slorr_gemm_pair_load": (i32, [vp, i32, i32, ctypes.POINTER(i64), ctypes.POINTER(i64)]),
        "slorr_gemm_item_list": (i32, [vp, i32, ctypes.POINTER(i32), i32]),
        "slorr_dataflow_items": (i32, [vp, ctypes.POINTER(i32), i32, ctypes.POINTER(i32), ctypes.POINTER(i32),
                                       ctypes.POINTER(dbl)]),
        "slorr_set_timing": (i32, [vp, i32]),
        "slorr_read_timing": (i32, [vp, ctypes.POINTER(dbl), ctypes.POINTER(i64), i32]),
        "slorr_frob_sq_noalloc": (i32, [vp, i64, i64, i32, vp, vp]),
        "slorr_pipeline_create": (i32, [ctypes.POINTER(vp), ctypes.POINTER(Shape), i32, ctypes.POINTER(Options),
                                        i32]),
        "slorr_pipeline_workspace_size": (i32, [vp, ctypes.POINTER(ctypes.c_size_t)]),
        "slorr_pipeline_forward_backward": (i32, [vp, ctypes.POINTER(vp), ctypes.POINTER(vp), vp, vp,
                                                  ctypes.POINTER(vp), ctypes.POINTER(vp), vp, ctypes.c_size_t, vp]),
        "slorr_pipeline_get_status": (i32, [vp, vp, vp]),
        "slorr_pipeline_destroy": (None, [vp]),
        "slorr_destroy": (None, [vp]),
        "slorr_status_string": (ctypes.c_char_p, [i32]),
        "slorr_last_error": (ctypes.c_char_p, []),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    if path is None:
        _lib = lib
    return lib


def declared_symbols(header: str = HEADER) -> list[str]:
    """Names of the functions include/slorr.h declares."""
    text = open(header).read()
    return sorted(set(re.findall(r"SLORR_API[^;(]*?\b(slorr_\w+)\s*\(", text)))


def _check(status: int) -> None:
    if status != SLORR_OK:
        msg = load_library().slorr_last_error()
        raise SlorrError(status, msg.decode() if msg else "")


def _shapes(shapes) -> tuple[ctypes.Array, int]:
    arr = (Shape * len(shapes))(*[Shape(int(m), int(n)) for m, n in shapes])
    return arr, len(shapes)


def _ptr_array(ptrs) -> ctypes.Array:
    return (ctypes.c_void_p * len(ptrs))(*[ctypes.c_void_p(int(p)) for p in ptrs])


# ---- functions with the C ABI's names ------------------------------------------

def slorr_default_options() -> Options:
    o = Options()
    load_library().slorr_default_options(ctypes.byref(o))
    return o


def slorr_create(shapes, options: Options | None = None) -> ctypes.c_void_p:
    arr, n = _shapes(shapes)
    h = ctypes.c_void_p()
    _check(load_library().slorr_create(ctypes.byref(h), arr, n,
                                       ctypes.byref(options) if options is not None else None))
    return h


def slorr_workspace_size(handle) -> int:
    out = ctypes.c_size_t()
    _check(load_library().slorr_workspace_size(handle, ctypes.byref(out)))
    return out.value


def slorr_reg_forward_backward(handle, weight_ptrs, grad_ptrs, loss_ptr, per_matrix_ptr, workspace_ptr,
                               workspace_bytes, stream) -> None:
    _check(load_library().slorr_reg_forward_backward(
        handle, _ptr_array(weight_ptrs), _ptr_array(grad_ptrs), ctypes.c_void_p(loss_ptr),
        ctypes.c_void_p(per_matrix_ptr or 0), ctypes.c_void_p(workspace_ptr), workspace_bytes,
        ctypes.c_void_p(stream or 0)))


def slorr_reg_descent_step(handle, weight_ptrs, eta, loss_ptr, per_matrix_ptr, workspace_ptr, workspace_bytes,
                           stream) -> None:
    _check(load_library().slorr_reg_descent_step(
        handle, _ptr_array(weight_ptrs), float(eta), ctypes.c_void_p(loss_ptr), ctypes.c_void_p(per_matrix_ptr or 0),
        ctypes.c_void_p(workspace_ptr), workspace_bytes, ctypes.c_void_p(stream or 0)))


def slorr_reset_workspace(handle) -> None:
    _check(load_library().slorr_reset_workspace(handle))


def slorr_get_status(handle, workspace_ptr, stream) -> int:
    """Returns the status code (does not raise for device-side errors)."""
    return int(load_library().slorr_get_status(handle, ctypes.c_void_p(workspace_ptr),
                                               ctypes.c_void_p(stream or 0)))


def slorr_run_steps(handle, weight_ptrs, workspace_ptr, workspace_bytes, steps, stream) -> None:
    _check(load_library().slorr_run_steps(handle, _ptr_array(weight_ptrs), ctypes.c_void_p(workspace_ptr),
                                          workspace_bytes, int(steps), ctypes.c_void_p(stream or 0)))


def slorr_iterate_view(handle, workspace_ptr, i, after_steps) -> MatrixView:
    v = MatrixView()
    _check(load_library().slorr_iterate_view(handle, ctypes.c_void_p(workspace_ptr), int(i),
                                             int(after_steps), ctypes.byref(v)))
    return v


def slorr_get_coefficients(handle, iters: int) -> np.ndarray:
    buf = (ctypes.c_double * (3 * iters))()
    _check(load_library().slorr_get_coefficients(handle, buf, 3 * iters))
    return np.array(buf, dtype=np.float64).reshape(iters, 3)


def slorr_pe_coefficients(iters: int = 6, ell: float = 1e-3, cushion: float = -1.0,
                          safety: float = 1.01) -> np.ndarray:
    buf = (ctypes.c_double * (3 * iters))()
    _check(load_library().slorr_pe_coefficients(int(iters), float(ell), float(cushion), float(safety), buf))
    return np.array(buf, dtype=np.float64).reshape(iters, 3)


def slorr_cushion_ratio() -> float:
    return float(load_library().slorr_cushion_ratio())


def slorr_flops(shapes, iters: int = 6) -> int:
    arr, n = _shapes(shapes)
    return int(load_library().slorr_flops(arr, n, int(iters)))


def slorr_executed_flops(handle) -> float:
    out = ctypes.c_double()
    _check(load_library().slorr_executed_flops(handle, ctypes.byref(out)))
    return out.value


def slorr_gemm_pair_load(handle, phase: int, npairs: int = 76) -> tuple:
    """(largest per-pair total K, total K) of one tensor-core GEMM launch when
    item i goes to pair i mod npairs."""
    mx, tot = ctypes.c_int64(0), ctypes.c_int64(0)
    _check(load_library().slorr_gemm_pair_load(handle, int(phase), int(npairs), ctypes.byref(mx), ctypes.byref(tot)))
    return int(mx.value), int(tot.value)


def slorr_gemm_items(handle, phase: int) -> int:
    """Work items of one GEMM launch of the plan: phase 0 Gram, 1 Poly, 2 Update."""
    out = ctypes.c_int32(0)
    _check(load_library().slorr_gemm_items(handle, int(phase), ctypes.byref(out)))
    return int(out.value)


def slorr_gemm_item_list(handle, phase: int) -> np.ndarray:
    """(items, 7) int32 array: mat, tm, tn, msz, nsz, part, parts per item, in launch order."""
    n = slorr_gemm_items(handle, phase)
    buf = (ctypes.c_int32 * max(1, 7 * n))()
    _check(load_library().slorr_gemm_item_list(handle, int(phase), buf, 7 * n))
    return np.frombuffer(buf, dtype=np.int32, count=7 * n).reshape(n, 7).copy()


def slorr_dataflow_items(handle):
    """(items, npairs, makespan_k): the dataflow plan as an (n, 10) int32 array
    of (pair, seq, step, phase, mat, tm, tn, part, parts, wait), pair by pair."""
    lib = load_library()
    npairs, count, mk = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_double()
    _check(lib.slorr_dataflow_items(handle, None, 0, ctypes.byref(npairs), ctypes.byref(count), ctypes.byref(mk)))
    n = count.value
    buf = (ctypes.c_int32 * max(1, 10 * n))()
    _check(lib.slorr_dataflow_items(handle, buf, 10 * n, ctypes.byref(npairs), ctypes.byref(count), None))
    return np.frombuffer(buf, dtype=np.int32, count=10 * n).reshape(n, 10).copy(), npairs.value, mk.value


def slorr_partition(shapes, world: int, rank: int) -> list[int]:
    arr, n = _shapes(shapes)
    out = (ctypes.c_int32 * max(n, 1))()
    cnt = ctypes.c_int32()
    _check(load_library().slorr_partition(arr, n, int(world), int(rank), out, ctypes.byref(cnt)))
    return [int(out[i]) for i in range(cnt.value)]


KERNEL_KINDS = ("sumsq", "cast", "gram", "poly", "update", "dot", "combine", "normcast", "gemm")


def slorr_set_timing(handle, enable: bool) -> None:
    _check(load_library().slorr_set_timing(handle, 1 if enable else 0))


def slorr_read_timing(handle) -> dict:
    """{kind: (milliseconds, launches)} accumulated since the last read."""
    n = len(KERNEL_KINDS)
    ms = (ctypes.c_double * n)()
    cnt = (ctypes.c_int64 * n)()
    _check(load_library().slorr_read_timing(handle, ms, cnt, n))
    return {k: (float(ms[i]), int(cnt[i])) for i, k in enumerate(KERNEL_KINDS)}


def slorr_frob_sq_noalloc(weight_ptr, m, n, dtype, out_ptr, stream) -> None:
    """||W||_F^2 of one device matrix into a device double, with no device
    allocation (fixed in-library scratch; see include/slorr.h)."""
    _check(load_library().slorr_frob_sq_noalloc(ctypes.c_void_p(weight_ptr), int(m), int(n), int(dtype),
                                                 ctypes.c_void_p(out_ptr), ctypes.c_void_p(stream or 0)))


def slorr_destroy(handle) -> None:
    load_library().slorr_destroy(handle)


def slorr_status_string(status: int) -> str:
    return load_library().slorr_status_string(int(status)).decode()


def slorr_pipeline_create(shapes, options: Options | None = None, groups: int = 8) -> ctypes.c_void_p:
    arr, n = _shapes(shapes)
    p = ctypes.c_void_p()
    _check(load_library().slorr_pipeline_create(ctypes.byref(p), arr, n,
                                                ctypes.byref(options) if options is not None else None, int(groups)))
    return p


def slorr_pipeline_workspace_size(pipe) -> int:
    out = ctypes.c_size_t()
    _check(load_library().slorr_pipeline_workspace_size(pipe, ctypes.byref(out)))
    return out.value


def slorr_pipeline_forward_backward(pipe, host_weight_ptrs, host_grad_ptrs, host_loss_ptr, host_per_matrix_ptr,
                                    dev_weight_ptrs, dev_grad_ptrs, workspace_ptr, workspace_bytes, stream) -> None:
    _check(load_library().slorr_pipeline_forward_backward(
        pipe, _ptr_array(host_weight_ptrs), _ptr_array(host_grad_ptrs), ctypes.c_void_p(host_loss_ptr),
        ctypes.c_void_p(host_per_matrix_ptr or 0), _ptr_array(dev_weight_ptrs), _ptr_array(dev_grad_ptrs),
        ctypes.c_void_p(workspace_ptr), workspace_bytes, ctypes.c_void_p(stream or 0)))


def slorr_pipeline_get_status(pipe, workspace_ptr, stream) -> int:
    return int(load_library().slorr_pipeline_get_status(pipe, ctypes.c_void_p(workspace_ptr),
                                                        ctypes.c_void_p(stream or 0)))


def slorr_pipeline_destroy(pipe) -> None:
    load_library().slorr_pipeline_destroy(pipe)


# ---- torch-facing convenience ----------------------------------------------------

def make_options(variant: str = "hoyer", compute: str = "fp16", dtype: str = "f32", iters: int = 6,
                 lam: float = 1.0, eps: float = 1e-7, grad_scale: float = 1.0, ell: float = 1e-3,
                 cushion: float = -1.0, safety: float = 1.01, flags: int = 0, timeout_s: float = 2.0) -> Options:
    """slorr_options from keyword arguments (defaults as slorr_default_options)."""
    o = slorr_default_options()
    o.variant = VARIANTS[variant]
    o.compute = COMPUTES[compute]
    o.dtype = DTYPES[dtype]
    o.iters = int(iters)
    o.lambda_ = float(lam)
    o.eps = float(eps)
    o.grad_scale = float(grad_scale)
    o.ell = float(ell)
    o.cushion = float(cushion)
    o.safety = float(safety)
    o.flags = int(flags)
    o.timeout_s = float(timeout_s)
    return o


class _OwnedHandle(ctypes.c_void_p):
    """A slorr_handle* that keeps the Python object owning it alive while the
    handle is referenced, so that ``Regularizer(...).handle`` passed straight
    into a call cannot be destroyed before the call has used it."""


class Regularizer:
    """One planned weight set.  Holds the handle and a torch-allocated workspace.

    ``reg(weights, grads)`` enqueues the forward value and gradient of every
    matrix on the current CUDA stream, accumulating lambda * grad into
    ``grads`` and returning the device loss tensor (lambda * sum_i L_i).
    ``compute`` picks the operand mode of the products: "fp16" (default),
    "bf16", "bf16_split" (bf16 hi/lo pairs, three products per product) or
    "fp32" (three tf32 products per product)."""

    def __init__(self, shapes, variant: str = "hoyer", compute: str = "fp16", dtype: str = "f32",
                 iters: int = 6, lam: float = 1.0, eps: float = 1e-7, grad_scale: float = 1.0,
                 ell: float = 1e-3, cushion: float = -1.0, safety: float = 1.01, flags: int = 0,
                 timeout_s: float = 2.0):
        o = make_options(variant, compute, dtype, iters, lam, eps, grad_scale, ell, cushion, safety, flags,
                         timeout_s)
        self.shapes = [(int(m), int(n)) for m, n in shapes]
        self.iters = int(iters)
        self.options = o
        self._raw = slorr_create(self.shapes, o)
        self.workspace_bytes = slorr_workspace_size(self._raw)
        self._ws = None

    @property
    def handle(self) -> _OwnedHandle:
        h = _OwnedHandle(self._raw.value)
        h.owner = self
        return h

    def __del__(self):
        h = getattr(self, "_raw", None)
        if h is not None and _lib is not None:
            slorr_destroy(h)
            self._raw = None

    def workspace(self, device):
        import torch
        if self._ws is None or self._ws.device != torch.device(device):
            self._ws = torch.empty(self.workspace_bytes + 256, dtype=torch.uint8, device=device)
        base = self._ws.data_ptr()
        return base + (-base) % 256

    def coefficients(self) -> np.ndarray:
        return slorr_get_coefficients(self.handle, self.iters)

    def _loss_buffer(self, dev):
        """A fresh loss tensor per call, or with FLAG_GRAPH one reused by every
        call (the graph replays while the output pointer stays the same)."""
        import torch
        if not (self.options.flags & FLAG_GRAPH):
            return torch.empty(1, dtype=torch.float32, device=dev)
        if getattr(self, "_loss", None) is None or self._loss.device != dev:
            self._loss = torch.empty(1, dtype=torch.float32, device=dev)
        return self._loss

    def __call__(self, weights, grads, loss=None, per_matrix=None, stream=None):
        import torch
        dev = weights[0].device
        ws = self.workspace(dev)
        if loss is None:
            loss = self._loss_buffer(dev)
        s = stream if stream is not None else torch.cuda.current_stream(dev).cuda_stream
        slorr_reg_forward_backward(self.handle, [w.data_ptr() for w in weights], [g.data_ptr() for g in grads],
                                   loss.data_ptr(), per_matrix.data_ptr() if per_matrix is not None else 0,
                                   ws, self.workspace_bytes, s)
        return loss

    def descent_step(self, weights, eta: float, loss=None, per_matrix=None, stream=None):
        """W_i -= eta * lambda * grad_scale * G_i(W_i) in place; returns the loss at the old weights."""
        import torch
        dev = weights[0].device
        ws = self.workspace(dev)
        if loss is None:
            loss = self._loss_buffer(dev)
        s = stream if stream is not None else torch.cuda.current_stream(dev).cuda_stream
        slorr_reg_descent_step(self.handle, [w.data_ptr() for w in weights], eta, loss.data_ptr(),
                               per_matrix.data_ptr() if per_matrix is not None else 0, ws, self.workspace_bytes, s)
        return loss

    def run_steps(self, weights, steps: int, stream=None):
        import torch
        dev = weights[0].device
        ws = self.workspace(dev)
        s = stream if stream is not None else torch.cuda.current_stream(dev).cuda_stream
        slorr_run_steps(self.handle, [w.data_ptr() for w in weights], ws, self.workspace_bytes, steps, s)

    def iterate(self, i: int, after_steps: int):
        """Copy of matrix i's Polar Express iterate X (P x Q) after `after_steps` steps, fp32."""
        import torch
        dev = self._ws.device
        v = slorr_iterate_view(self.handle, self.workspace(dev), i, after_steps)
        typestr = {0: "<f4", 1: "<f2", 2: "<u2"}[v.elem]
        raw = device_view(v.x, (v.rows, v.ld), typestr, dev).clone()
        if v.elem == 2:
            raw = raw.view(torch.bfloat16)
        x = raw[:, : v.cols].float()
        if after_steps == 0:  # 16-bit iterates hold W unscaled: X_0 = x0_scale * buffer
            x = x * device_view(v.x0_scale, (1,), "<f4", dev).clone()
        return x.t().contiguous() if v.transposed else x

    def scalars(self, i: int):
        """(||W_i||_F^2, n_hat_i) read back from the workspace."""
        dev = self._ws.device
        v = slorr_iterate_view(self.handle, self.workspace(dev), i, 0)
        out = device_view(v.frob_sq, (2,), "<f8", dev).clone().cpu()
        return float(out[0]), float(out[1])

    def status(self, stream=None) -> int:
        import torch
        dev = self._ws.device
        s = stream if stream is not None else torch.cuda.current_stream(dev).cuda_stream
        return slorr_get_status(self.handle, self.workspace(dev), s)


class Pipeline:
    """A weight set whose weights and grads live in (page-locked) host memory.

    ``pipe(host_w, host_g, dev_w, dev_g, host_loss)`` enqueues the pipelined
    forward + backward on the current CUDA stream: copies in, kernels and
    copies out of consecutive groups of matrices overlap.  ``host_g`` is
    accumulated into (+=); ``host_loss`` (a page-locked 1-element float tensor)
    receives lambda * sum_i L_i.  Keyword options as for ``Regularizer``."""

    @staticmethod
    def auto_groups(shapes, dtype: str = "f32", compute: str = "fp16") -> int:
        """About 64 MiB of weights per group, 1 to 16 groups: enough groups for the
        copies to overlap the kernels, few enough that a group's launches stay
        cheap next to its copies.  With bf16 hi/lo operands, whose kernels take
        2.4 times as long, about 128 MiB (ViT-L/16 on GB300: 18.0 ms with 8
        groups, 31.7 ms with 16)."""
        esz = 4 if dtype == "f32" else 2
        total = sum(int(m) * int(n) for m, n in shapes) * esz
        per = (128 << 20) if compute == "bf16_split" else (64 << 20)
        return max(1, min(16, total // per))

    def __init__(self, shapes, groups: int | None = None, **kw):
        self.shapes = [(int(m), int(n)) for m, n in shapes]
        if groups is None:
            groups = self.auto_groups(self.shapes, kw.get("dtype", "f32"), kw.get("compute", "fp16"))
        self.groups = int(groups)
        self.options = make_options(**kw)
        self.handle = slorr_pipeline_create(self.shapes, self.options, groups)
        self.workspace_bytes = slorr_pipeline_workspace_size(self.handle)
        self._ws = None

    def __del__(self):
        h = getattr(self, "handle", None)
        if h is not None and _lib is not None:
            slorr_pipeline_destroy(h)
            self.handle = None

    def workspace(self, device):
        import torch
        if self._ws is None or self._ws.device != torch.device(device):
            self._ws = torch.empty(self.workspace_bytes + 256, dtype=torch.uint8, device=device)
        base = self._ws.data_ptr()
        return base + (-base) % 256

    def __call__(self, host_weights, host_grads, dev_weights, dev_grads, host_loss, host_per_matrix=None,
                 stream=None):
        import torch
        dev = dev_weights[0].device
        ws = self.workspace(dev)
        s = stream if stream is not None else torch.cuda.current_stream(dev).cuda_stream
        slorr_pipeline_forward_backward(
            self.handle, [w.data_ptr() for w in host_weights], [g.data_ptr() for g in host_grads],
            host_loss.data_ptr(), host_per_matrix.data_ptr() if host_per_matrix is not None else 0,
            [w.data_ptr() for w in dev_weights], [g.data_ptr() for g in dev_grads], ws, self.workspace_bytes, s)

    def status(self, stream=None) -> int:
        import torch
        dev = self._ws.device
        s = stream if stream is not None else torch.cuda.current_stream(dev).cuda_stream
        return slorr_pipeline_get_status(self.handle, self.workspace(dev), s)


class _DeviceArray:
    def __init__(self, ptr: int, shape, typestr: str):
        self.__cuda_array_interface__ = {"shape": tuple(int(d) for d in shape), "typestr": typestr,
                                         "data": (int(ptr), False), "version": 2, "strides": None}


def device_view(ptr: int, shape, typestr: str, device):
    """A torch tensor aliasing device memory at `ptr` (test introspection only)."""
    import torch
    return torch.as_tensor(_DeviceArray(ptr, shape, typestr), device=device)

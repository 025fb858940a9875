"""ctypes binding of ``libnoble.so`` (include/noble.h), plus thin torch helpers.

Argument marshalling only: every step of the layer runs in the library's
kernels.  There is no fallback: if the library is missing or cannot run on the
current device the call raises.

Functions with the C names take device pointers given as ints, torch tensors
or None.  ``NobleLinearBuffers`` / ``forward`` / ``backward`` allocate the
caller-owned buffers with torch and call the same entry points.
"""
from __future__ import annotations

import ctypes
import os
import re
import threading

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libnoble.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "noble.h")

NOBLE_BF16, NOBLE_FP32 = 0, 1
NOBLE_FLAG_SIMT_ONLY, NOBLE_FLAG_INFERENCE = 1, 2
NOBLE_FLAG_SIGMA_COS1, NOBLE_FLAG_SIGMA_IDENTITY = 4, 8
NOBLE_FLAG_FUSED_BRANCH = 16
NOBLE_FLAG_ACT_TANH, NOBLE_FLAG_ACT_LEAKYRELU, NOBLE_FLAG_ACT_GELU = 32, 64, 96
NOBLE_FLAG_SIGMA_SINGLE = NOBLE_FLAG_SIGMA_COS1
NOBLE_FLAG_SIGMA_COS3 = 128
# bottleneck variants by name (Section 4.4, Table 5): flags of the descriptor
SIGMA_FLAGS = {"cosnet": 0, "cos1": NOBLE_FLAG_SIGMA_COS1, "identity": NOBLE_FLAG_SIGMA_IDENTITY,
               "tanh1": NOBLE_FLAG_ACT_TANH | NOBLE_FLAG_SIGMA_SINGLE, "tanh2": NOBLE_FLAG_ACT_TANH,
               "leaky1": NOBLE_FLAG_ACT_LEAKYRELU | NOBLE_FLAG_SIGMA_SINGLE, "leaky2": NOBLE_FLAG_ACT_LEAKYRELU,
               "gelu1": NOBLE_FLAG_ACT_GELU | NOBLE_FLAG_SIGMA_SINGLE, "gelu2": NOBLE_FLAG_ACT_GELU}
# parameters a variant does not read (may be passed as None)
SIGMA_UNUSED = {"cosnet": (), "cos1": ("M", "omega2", "phi2"),
                "identity": ("omega1", "phi1", "M", "omega2", "phi2")}
for _n in ("tanh", "leaky", "gelu"):
    SIGMA_UNUSED[_n + "1"] = ("omega1", "phi1", "M", "omega2", "phi2")
    SIGMA_UNUSED[_n + "2"] = ("omega1", "phi1", "omega2", "phi2")
STATUS = {0: "NOBLE_OK", 1: "NOBLE_ERR_INVALID_ARG", 2: "NOBLE_ERR_MISALIGNED",
          3: "NOBLE_ERR_UNSUPPORTED", 4: "NOBLE_ERR_BUFFER_TOO_SMALL", 5: "NOBLE_ERR_CUDA",
          6: "NOBLE_ERR_TIMEOUT", 7: "NOBLE_ERR_NO_DEVICE"}


class NobleError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


class Desc(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int64), ("d_in", ctypes.c_int64), ("d_out", ctypes.c_int64),
                ("r", ctypes.c_int64), ("dtype", ctypes.c_int32), ("flags", ctypes.c_uint32)]


class AdamwTensor(ctypes.Structure):
    _fields_ = [("param", ctypes.c_void_p), ("param_bf16", ctypes.c_void_p), ("grad", ctypes.c_void_p),
                ("exp_avg", ctypes.c_void_p), ("exp_avg_sq", ctypes.c_void_p), ("n", ctypes.c_int64),
                ("lr_mult", ctypes.c_float), ("decay", ctypes.c_int32)]


class AdamwHparams(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_float), ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
                ("eps", ctypes.c_float), ("weight_decay", ctypes.c_float), ("step", ctypes.c_int64)]


GRAD_COUNT, GRAD_ALIGN = 12, 256
# slots of the gradient bucket, in the order noble_linear_grad_bucket gives
BUCKET_SLOTS = ("dW", "dbias", "dW_down", "dW_up", "dM", "domega1", "dphi1", "domega2", "dphi2",
                "dM2", "domega3", "dphi3")


class GradBucket(ctypes.Structure):
    _fields_ = [("offset", ctypes.c_size_t * GRAD_COUNT), ("count", ctypes.c_size_t * GRAD_COUNT),
                ("total_bytes", ctypes.c_size_t)]


class Cos3Params(ctypes.Structure):
    _fields_ = [("M2", ctypes.c_void_p), ("omega3", ctypes.c_void_p), ("phi3", ctypes.c_void_p)]


class Cos3Grads(ctypes.Structure):
    _fields_ = [("dM2", ctypes.c_void_p), ("domega3", ctypes.c_void_p), ("dphi3", ctypes.c_void_p)]


def make_desc(T, d_in, d_out, r, dtype, flags=0) -> Desc:
    if isinstance(dtype, str):
        dtype = {"bf16": NOBLE_BF16, "fp32": NOBLE_FP32}[dtype]
    return Desc(T, d_in, d_out, r, dtype, flags)


_lib = None
_lock = threading.Lock()


def declared_functions() -> list[str]:
    """Names of the functions include/noble.h declares."""
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(noble_[a-z_0-9]+)\s*\(", src)))


def load(path: str | None = None) -> ctypes.CDLL:
    """Load the library (once).  Raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = path or LIB_PATH
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is missing: build it with paper_2603_06492_gb300.build.build()")
        lib = ctypes.CDLL(path)
        P, S, D = ctypes.c_void_p, ctypes.c_size_t, ctypes.POINTER(Desc)
        lib.noble_linear_saved_bytes.argtypes = [D]
        lib.noble_linear_saved_bytes.restype = S
        lib.noble_linear_bwd_workspace_bytes.argtypes = [D]
        lib.noble_linear_bwd_workspace_bytes.restype = S
        lib.noble_linear_fwd.argtypes = [D] + [P] * 12 + [S, P]
        lib.noble_linear_fwd.restype = ctypes.c_int
        lib.noble_linear_bwd.argtypes = [D] + [P] * 11 + [S] + [P] * 11 + [S, P]
        lib.noble_linear_bwd.restype = ctypes.c_int
        C3P, C3G = ctypes.POINTER(Cos3Params), ctypes.POINTER(Cos3Grads)
        lib.noble_linear_fwd_cos3.argtypes = [D] + [P] * 9 + [C3P] + [P] * 3 + [S, P]
        lib.noble_linear_fwd_cos3.restype = ctypes.c_int
        lib.noble_linear_bwd_cos3.argtypes = [D] + [P] * 9 + [C3P] + [P] * 2 + [S] + [P] * 9 + [C3G] + [P] * 2 + [S, P]
        lib.noble_linear_bwd_cos3.restype = ctypes.c_int
        lib.noble_linear_bwd_noalloc.argtypes = [D] + [P] * 11 + [S] + [P] * 10 + [P]
        lib.noble_linear_bwd_noalloc.restype = ctypes.c_int
        lib.noble_get_device_status.argtypes = [P]
        lib.noble_get_device_status.restype = ctypes.c_int
        lib.noble_status_string.argtypes = [ctypes.c_int]
        lib.noble_status_string.restype = ctypes.c_char_p
        lib.noble_last_error.argtypes = []
        lib.noble_last_error.restype = ctypes.c_char_p
        lib.noble_kernel_launch_count.argtypes = []
        lib.noble_kernel_launch_count.restype = ctypes.c_uint64
        lib.noble_debug_raise_device_status.argtypes = [ctypes.c_uint32]
        lib.noble_debug_raise_device_status.restype = ctypes.c_int
        lib.noble_debug_wait_expiry.argtypes = [ctypes.c_uint64, P, P]
        lib.noble_debug_wait_expiry.restype = ctypes.c_int
        i64, ci = ctypes.c_int64, ctypes.c_int
        lib.noble_test_gemm_bf16.argtypes = [i64] * 4 + [ci] * 3 + [P] * 6 + [ci] * 3 + [P]
        lib.noble_test_gemm_bf16.restype = ctypes.c_int
        lib.noble_profile_enable.argtypes = [ctypes.c_int]
        lib.noble_profile_enable.restype = None
        lib.noble_profile_reset.argtypes = []
        lib.noble_profile_reset.restype = None
        lib.noble_profile_count.argtypes = []
        lib.noble_profile_count.restype = ctypes.c_int
        lib.noble_profile_entry.argtypes = [ctypes.c_int, ctypes.c_char_p, ctypes.c_size_t] + [P] * 5
        lib.noble_profile_entry.restype = ctypes.c_int
        lib.noble_adamw_step.argtypes = [ctypes.POINTER(AdamwTensor), ctypes.c_int,
                                         ctypes.POINTER(AdamwHparams), P]
        lib.noble_adamw_step.restype = ctypes.c_int
        lib.noble_linear_lr_multipliers.argtypes = [D] + [ctypes.c_float] * 4 + [ctypes.POINTER(ctypes.c_float)]
        lib.noble_linear_lr_multipliers.restype = ctypes.c_int
        lib.noble_linear_grad_bucket.argtypes = [D, ctypes.POINTER(GradBucket)]
        lib.noble_linear_grad_bucket.restype = ctypes.c_int
        _lib = lib
        return lib


def _p(a):
    """Pointer value of a torch tensor, an int or None."""
    if a is None:
        return None
    if isinstance(a, int):
        return a
    return a.data_ptr()


def _check(status: int):
    if status != 0:
        lib = load()
        raise NobleError(status, lib.noble_last_error().decode() or
                         lib.noble_status_string(status).decode())


def noble_linear_saved_bytes(desc: Desc) -> int:
    return load().noble_linear_saved_bytes(ctypes.byref(desc))


def noble_linear_bwd_workspace_bytes(desc: Desc) -> int:
    return load().noble_linear_bwd_workspace_bytes(ctypes.byref(desc))


def noble_linear_fwd(desc, x, W, bias, W_down, omega1, phi1, M, omega2, phi2, W_up, y, saved,
                     saved_bytes, stream):
    _check(load().noble_linear_fwd(ctypes.byref(desc), _p(x), _p(W), _p(bias), _p(W_down),
                                   _p(omega1), _p(phi1), _p(M), _p(omega2), _p(phi2), _p(W_up),
                                   _p(y), _p(saved), saved_bytes, stream))


def noble_linear_bwd(desc, dy, x, W, W_down, omega1, phi1, M, omega2, phi2, W_up, saved,
                     saved_bytes, dx, dW, dbias, dW_down, dM, domega1, dphi1, domega2, dphi2,
                     dW_up, workspace, workspace_bytes, stream):
    _check(load().noble_linear_bwd(ctypes.byref(desc), _p(dy), _p(x), _p(W), _p(W_down),
                                   _p(omega1), _p(phi1), _p(M), _p(omega2), _p(phi2), _p(W_up),
                                   _p(saved), saved_bytes, _p(dx), _p(dW), _p(dbias), _p(dW_down),
                                   _p(dM), _p(domega1), _p(dphi1), _p(domega2), _p(dphi2),
                                   _p(dW_up), _p(workspace), workspace_bytes, stream))


def noble_linear_fwd_cos3(desc, x, W, bias, W_down, omega1, phi1, M, omega2, phi2, M2, omega3, phi3, W_up,
                          y, saved, saved_bytes, stream):
    p3 = Cos3Params(_p(M2), _p(omega3), _p(phi3))
    _check(load().noble_linear_fwd_cos3(ctypes.byref(desc), _p(x), _p(W), _p(bias), _p(W_down),
                                        _p(omega1), _p(phi1), _p(M), _p(omega2), _p(phi2),
                                        ctypes.byref(p3), _p(W_up), _p(y), _p(saved), saved_bytes, stream))


def noble_linear_bwd_cos3(desc, dy, x, W, W_down, omega1, phi1, M, omega2, phi2, M2, omega3, phi3, W_up,
                          saved, saved_bytes, dx, dW, dbias, dW_down, dM, domega1, dphi1, domega2, dphi2,
                          dM2, domega3, dphi3, dW_up, workspace, workspace_bytes, stream):
    p3 = Cos3Params(_p(M2), _p(omega3), _p(phi3))
    g3 = Cos3Grads(_p(dM2), _p(domega3), _p(dphi3))
    _check(load().noble_linear_bwd_cos3(ctypes.byref(desc), _p(dy), _p(x), _p(W), _p(W_down),
                                        _p(omega1), _p(phi1), _p(M), _p(omega2), _p(phi2),
                                        ctypes.byref(p3), _p(W_up), _p(saved), saved_bytes, _p(dx),
                                        _p(dW), _p(dbias), _p(dW_down), _p(dM), _p(domega1), _p(dphi1),
                                        _p(domega2), _p(dphi2), ctypes.byref(g3), _p(dW_up),
                                        _p(workspace), workspace_bytes, stream))


def noble_test_gemm_bf16(M, N, K0, K1, a_mn, b_mn, bn, A0, B0, A1, B1, bias, C, c_fp32,
                         kb_per_split, nsplit, stream):
    _check(load().noble_test_gemm_bf16(M, N, K0, K1, a_mn, b_mn, bn, _p(A0), _p(B0), _p(A1),
                                       _p(B1), _p(bias), _p(C), c_fp32, kb_per_split, nsplit,
                                       stream))


def noble_linear_bwd_noalloc(desc, dy, x, W, W_down, omega1, phi1, M, omega2, phi2, W_up, saved,
                             saved_bytes, dx, dW, dbias, dW_down, dM, domega1, dphi1, domega2,
                             dphi2, dW_up, stream):
    """Backward pass using the library's static scratch (no workspace argument)."""
    _check(load().noble_linear_bwd_noalloc(ctypes.byref(desc), _p(dy), _p(x), _p(W), _p(W_down),
                                           _p(omega1), _p(phi1), _p(M), _p(omega2), _p(phi2),
                                           _p(W_up), _p(saved), saved_bytes, _p(dx), _p(dW),
                                           _p(dbias), _p(dW_down), _p(dM), _p(domega1),
                                           _p(dphi1), _p(domega2), _p(dphi2), _p(dW_up), stream))


NOALLOC_SCRATCH_BYTES = 64 << 20


def noble_adamw_step(tensors, lr, beta1=0.9, beta2=0.98, eps=1e-8, weight_decay=0.01, step=1,
                     stream=None):
    """One fused AdamW step.  ``tensors``: dicts with param, grad, exp_avg,
    exp_avg_sq (fp32 device tensors or pointers), optional param_bf16,
    lr_mult (default 1) and decay (default True)."""
    arr = (AdamwTensor * max(1, len(tensors)))()
    for i, t in enumerate(tensors):
        n = t["n"] if "n" in t else t["param"].numel()
        arr[i] = AdamwTensor(_p(t["param"]), _p(t.get("param_bf16")), _p(t["grad"]), _p(t["exp_avg"]),
                             _p(t["exp_avg_sq"]), n, float(t.get("lr_mult", 1.0)), int(t.get("decay", True)))
    hp = AdamwHparams(lr, beta1, beta2, eps, weight_decay, step)
    _check(load().noble_adamw_step(arr, len(tensors), ctypes.byref(hp), stream))


def noble_linear_lr_multipliers(desc, gamma=0.3, gamma_M=0.45, omega_mult=3.0, phi_mult=5.0):
    """Per-group learning-rate multipliers [W|bias|W_down, W_up, M, omega, phi]."""
    out = (ctypes.c_float * 5)()
    _check(load().noble_linear_lr_multipliers(ctypes.byref(desc), gamma, gamma_M, omega_mult, phi_mult, out))
    return list(out)


def noble_linear_grad_bucket(desc) -> dict:
    """Layout of the layer's flat fp32 gradient bucket: {slot: (byte offset,
    element count)} for the slots the descriptor has, and "total_bytes"."""
    b = GradBucket()
    _check(load().noble_linear_grad_bucket(ctypes.byref(desc), ctypes.byref(b)))
    out = {name: (b.offset[i], b.count[i]) for i, name in enumerate(BUCKET_SLOTS) if b.count[i] > 0}
    out["total_bytes"] = b.total_bytes
    return out


def bucket_views(bucket, layout: dict, shapes: dict) -> dict:
    """Views of a flat fp32 bucket tensor (torch) as the layer's gradients."""
    out = {}
    for name, slot in layout.items():
        if name != "total_bytes":
            off, n = slot
            out[name] = bucket[off // 4: off // 4 + n].view(shapes[name])
    return out


def grad_shapes(d_in, d_out, r) -> dict:
    return {"dW": (d_out, d_in), "dbias": (d_out,), "dW_down": (r, d_in), "dW_up": (d_out, r), "dM": (r, r),
            "domega1": (r,), "dphi1": (r,), "domega2": (r,), "dphi2": (r,), "dM2": (r, r), "domega3": (r,),
            "dphi3": (r,)}


def noble_get_device_status(stream=None):
    _check(load().noble_get_device_status(stream))


def noble_kernel_launch_count() -> int:
    return load().noble_kernel_launch_count()


def noble_debug_raise_device_status(bits: int):
    _check(load().noble_debug_raise_device_status(bits))


def noble_debug_wait_expiry(limit_ns: int, result, stream=None):
    _check(load().noble_debug_wait_expiry(limit_ns, _p(result), _stream_handle(stream)))


def profile_read() -> dict:
    """Per-kernel-class totals recorded since the last reset (see noble.h)."""
    lib = load()
    n = lib.noble_profile_count()
    out = {}
    for i in range(n):
        name = ctypes.create_string_buffer(128)
        launches, bound = ctypes.c_uint64(), ctypes.c_int()
        ms, flops, nbytes = ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
        _check(lib.noble_profile_entry(i, name, 128, ctypes.byref(launches), ctypes.byref(ms),
                                       ctypes.byref(flops), ctypes.byref(nbytes), ctypes.byref(bound)))
        out[name.value.decode()] = {"name": name.value.decode(), "launches": launches.value,
                                    "ms": ms.value, "flops": flops.value, "bytes": nbytes.value,
                                    "bound": {0: "tensor", 1: "hbm", 2: "alu"}[bound.value]}
    return out


# ---------------------------------------------------------------- torch side
PARAM_NAMES = ("W", "bias", "W_down", "omega1", "phi1", "M", "omega2", "phi2", "W_up")
GRAD_NAMES = ("dW", "dbias", "dW_down", "dM", "domega1", "dphi1", "domega2", "dphi2", "dW_up")


def _stream_handle(stream):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


class NobleLinearBuffers:
    """Caller-owned device buffers for one layer shape (allocated with torch)."""

    def __init__(self, T, d_in, d_out, r, dtype, device="cuda", with_grads=True, flags=0):
        """With gradients, they are views of one flat fp32 bucket (``self.bucket``,
        laid out by noble_linear_grad_bucket), which a data-parallel step
        all-reduces in one collective."""
        import torch
        self.desc = make_desc(T, d_in, d_out, r, dtype, flags)
        tdt = torch.bfloat16 if self.desc.dtype == NOBLE_BF16 else torch.float32
        self.saved_bytes = noble_linear_saved_bytes(self.desc)
        self.workspace_bytes = noble_linear_bwd_workspace_bytes(self.desc)
        self.y = torch.empty((T, d_out), dtype=tdt, device=device)
        self.saved = (torch.empty(self.saved_bytes, dtype=torch.uint8, device=device)
                      if self.saved_bytes else None)
        if with_grads:
            f32 = dict(dtype=torch.float32, device=device)
            self.dx = torch.empty((T, d_in), dtype=tdt, device=device)
            self.workspace = torch.empty(self.workspace_bytes, dtype=torch.uint8, device=device)
            self.layout = noble_linear_grad_bucket(self.desc)
            self.bucket = torch.zeros(self.layout["total_bytes"] // 4, **f32)
            self.grads = bucket_views(self.bucket, self.layout, grad_shapes(d_in, d_out, r))


def forward(buf: NobleLinearBuffers, x, params: dict, stream=None):
    """y = NOBLE(x) into ``buf.y``; saves activations in ``buf.saved``."""
    p = params
    if buf.desc.flags & NOBLE_FLAG_SIGMA_COS3:
        noble_linear_fwd_cos3(buf.desc, x, p["W"], p.get("bias"), p.get("W_down"), p.get("omega1"),
                              p.get("phi1"), p.get("M"), p.get("omega2"), p.get("phi2"), p.get("M2"),
                              p.get("omega3"), p.get("phi3"), p.get("W_up"), buf.y, buf.saved,
                              buf.saved_bytes, _stream_handle(stream))
        return buf.y
    noble_linear_fwd(buf.desc, x, p["W"], p.get("bias"), p.get("W_down"), p.get("omega1"),
                     p.get("phi1"), p.get("M"), p.get("omega2"), p.get("phi2"), p.get("W_up"),
                     buf.y, buf.saved, buf.saved_bytes, _stream_handle(stream))
    return buf.y


def backward(buf: NobleLinearBuffers, x, dy, params: dict, stream=None, with_dbias=True):
    """dx into ``buf.dx`` and parameter gradients into ``buf.grads``."""
    p, g = params, buf.grads
    if buf.desc.flags & NOBLE_FLAG_SIGMA_COS3:
        noble_linear_bwd_cos3(buf.desc, dy, x, p["W"], p.get("W_down"), p.get("omega1"), p.get("phi1"),
                              p.get("M"), p.get("omega2"), p.get("phi2"), p.get("M2"), p.get("omega3"),
                              p.get("phi3"), p.get("W_up"), buf.saved, buf.saved_bytes, buf.dx, g["dW"],
                              g["dbias"] if with_dbias else None, g.get("dW_down"), g.get("dM"),
                              g.get("domega1"), g.get("dphi1"), g.get("domega2"), g.get("dphi2"),
                              g.get("dM2"), g.get("domega3"), g.get("dphi3"), g.get("dW_up"),
                              buf.workspace, buf.workspace_bytes, _stream_handle(stream))
        return buf.dx, g
    noble_linear_bwd(buf.desc, dy, x, p["W"], p.get("W_down"), p.get("omega1"), p.get("phi1"),
                     p.get("M"), p.get("omega2"), p.get("phi2"), p.get("W_up"), buf.saved,
                     buf.saved_bytes, buf.dx, g["dW"], g["dbias"] if with_dbias else None,
                     g.get("dW_down"), g.get("dM"), g.get("domega1"), g.get("dphi1"),
                     g.get("domega2"), g.get("dphi2"), g.get("dW_up"), buf.workspace,
                     buf.workspace_bytes, _stream_handle(stream))
    return buf.dx, g


def params_to_device(inp: dict, dtype: str, device="cuda") -> dict:
    """Move numpy inputs (library layout, see inputs.py) to device tensors:
    operands in ``dtype``, omega/phi/M/bias in fp32."""
    import numpy as np
    import torch
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    out = {}
    for k, v in inp.items():
        t = torch.from_numpy(np.ascontiguousarray(v, dtype=np.float32))
        if k in ("x", "W", "W_down", "W_up", "dy"):
            t = t.to(tdt)
        out[k] = t.to(device)
    return out

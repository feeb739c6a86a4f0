"""Thin Python binding of libsparoa (include/sparoa.h): argument marshalling only.

Every function here forwards to the C ABI of the same name; tensors are torch
CUDA tensors (device memory and streams come from PyTorch), and the calls run
on the current torch stream.  There is no fallback: if ``libsparoa.so`` is
missing or fails to load, importing this module raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libsparoa.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"libsparoa.so is not built ({LIB_PATH}); run __graft_entry__.build()")
_lib = ctypes.CDLL(LIB_PATH)

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_OOM, ERR_CUDA, ERR_TIMEOUT = range(6)
BF16, F32 = 0, 1
PATH_NONE, PATH_DENSE, PATH_SKIP, PATH_DEPTHWISE = 0, 1, 2, 3
ACT_NONE, ACT_RELU, ACT_RELU6, ACT_GELU = 0, 1, 2, 3
OP_CONV2D, OP_FC, OP_MAXPOOL, OP_AVGPOOL, OP_BN_ACT = 1, 2, 3, 4, 5
OP_LAYERNORM, OP_ATTENTION, OP_TOKENS, OP_SELECT = 6, 7, 8, 9

_P = ctypes.c_void_p
_I64 = ctypes.c_int64
_I32 = ctypes.c_int32


class Thresholds(ctypes.Structure):
    _fields_ = [("s_thr", ctypes.c_double), ("c_thr", ctypes.c_double),
                ("intensity_mode", _I32), ("force_path", _I32)]


class Stats(ctypes.Structure):
    _fields_ = [("numel", ctypes.c_uint64), ("nnz", ctypes.c_uint64), ("sparsity", ctypes.c_double),
                ("flops", ctypes.c_uint64), ("macs_eq2", ctypes.c_uint64),
                ("input_bytes", ctypes.c_uint64), ("flops_per_byte", ctypes.c_double),
                ("B", _I32), ("C_in", _I32), ("H", _I32), ("W", _I32), ("path", _I32),
                ("reserved", _I32)]

    def as_dict(self):
        return {k: getattr(self, k) for k, _ in self._fields_ if k != "reserved"}


class Occupancy(ctypes.Structure):
    _fields_ = [("nnz", _P), ("col_nnz", _P), ("tile_nnz", _P), ("row_bm", _P), ("blk_mask", _P),
                ("R", _I64), ("C", _I64), ("bytes", ctypes.c_uint64)]


class Epilogue(ctypes.Structure):
    _fields_ = [("bias", _P), ("bn", _P), ("bn_eps", ctypes.c_float), ("act", _I32),
                ("residual", _P)]


class Op(ctypes.Structure):
    _fields_ = [("kind", _I32), ("input", _I32), ("residual", _I32), ("c_in", _I32), ("c_out", _I32),
                ("kh", _I32), ("kw", _I32), ("stride", _I32), ("pad", _I32), ("groups", _I32),
                ("act", _I32), ("reserved", _I32), ("weight", _P), ("weight_kn", _P), ("bias", _P),
                ("bn", _P), ("bn_eps", ctypes.c_float), ("reserved2", ctypes.c_float),
                ("thr", Thresholds)]


class Record(ctypes.Structure):
    _fields_ = [("stats", Stats), ("output", _P), ("out_shape", _I64 * 4),
                ("out_occ", ctypes.POINTER(Occupancy))]


def _sig(name, args):
    f = getattr(_lib, name)
    f.restype = ctypes.c_int
    f.argtypes = args
    return f


_sig("sparoa_create", [ctypes.POINTER(_P), ctypes.c_int, _P])
_sig("sparoa_destroy", [_P])
_sig("sparoa_set_stream", [_P, _P])
_sig("sparoa_set_overlap", [_P, _I32])
_sig("sparoa_graph_workspace", [_P, _P, _I32, _I64, _I64, _I64, _I64, ctypes.POINTER(ctypes.c_uint64)])
_sig("sparoa_gemm_split", [_P, _P, _I64, _I64, _P, _P, _I64, _P, ctypes.c_double, _P, _I32, _P, _P])
_sig("sparoa_sync", [_P])
_sig("sparoa_last_path", [_P, ctypes.POINTER(_I32)])
_sig("sparoa_set_wait_limit", [_P, ctypes.c_int64])
_sig("sparoa_set_fault", [_P, ctypes.c_int32])
_lib.sparoa_status_str.restype = ctypes.c_char_p
_lib.sparoa_status_str.argtypes = [ctypes.c_int]
_lib.sparoa_last_error.restype = ctypes.c_char_p
_lib.sparoa_last_error.argtypes = [_P]
_lib.sparoa_occupancy_bytes.restype = ctypes.c_uint64
_lib.sparoa_occupancy_bytes.argtypes = [_I64, _I64]
_sig("sparoa_occupancy_init", [_P, ctypes.c_uint64, _I64, _I64, ctypes.POINTER(Occupancy)])
_sig("sparoa_op_stats", [_P, _P, _I64, _I64, _I64, _I64, ctypes.POINTER(Op),
                         ctypes.POINTER(Occupancy), ctypes.POINTER(Stats)])
_sig("sparoa_gemm", [_P, _P, _I64, _I64, _P, _P, _I64, ctypes.POINTER(Epilogue),
                     ctypes.POINTER(Thresholds), _P, _I32, ctypes.POINTER(Occupancy),
                     ctypes.POINTER(Occupancy), ctypes.POINTER(Stats)])
_sig("sparoa_conv2d", [_P, _P, _I64, _I64, _I64, _I64, _P, _I64, _I32, _I32, _I32, _I32, _I32,
                       ctypes.POINTER(Epilogue), ctypes.POINTER(Thresholds), _P,
                       ctypes.POINTER(Occupancy), ctypes.POINTER(Occupancy), ctypes.POINTER(Stats)])
_sig("sparoa_maxpool2d", [_P, _P, _I64, _I64, _I64, _I64, _I32, _I32, _I32, _P,
                          ctypes.POINTER(Occupancy)])
_sig("sparoa_avgpool_global", [_P, _P, _I64, _I64, _I64, _I64, _P, ctypes.POINTER(Occupancy)])
_sig("sparoa_bn_act", [_P, _P, _I64, _I64, ctypes.POINTER(Epilogue), _P, ctypes.POINTER(Occupancy)])
_sig("sparoa_layernorm", [_P, _P, _I64, _I64, _P, ctypes.c_float, _P, ctypes.POINTER(Occupancy)])
_sig("sparoa_attention", [_P, _P, _I64, _I64, _I32, _I32, _P, ctypes.POINTER(Occupancy)])
_sig("sparoa_run_graph", [_P, ctypes.POINTER(Op), _I32, _P, _I64, _I64, _I64, _I64, _P,
                          ctypes.c_uint64, ctypes.POINTER(Record)])
_sig("sparoa_gemm_noalloc", [_P, _P, _I64, _I64, _P, _P, _I64, ctypes.POINTER(Epilogue),
                             ctypes.POINTER(Thresholds), _P, _I32, ctypes.POINTER(Stats)])

EXPORTED = ["sparoa_create", "sparoa_destroy", "sparoa_set_stream", "sparoa_set_overlap", "sparoa_sync",
            "sparoa_last_path",
            "sparoa_set_wait_limit", "sparoa_set_fault",
            "sparoa_status_str", "sparoa_last_error", "sparoa_occupancy_bytes",
            "sparoa_occupancy_init", "sparoa_op_stats", "sparoa_gemm", "sparoa_conv2d",
            "sparoa_maxpool2d", "sparoa_avgpool_global", "sparoa_bn_act", "sparoa_run_graph",
            "sparoa_graph_workspace", "sparoa_gemm_split", "sparoa_layernorm", "sparoa_attention",
            "sparoa_gemm_noalloc"]


class SparoaError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{_lib.sparoa_status_str(status).decode()}: {msg}")
        self.status = status


def _ptr(t):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def thresholds(s_thr=0.5, c_thr=32.0, intensity_mode=0, force_path=0) -> Thresholds:
    return Thresholds(float(s_thr), float(c_thr), int(intensity_mode), int(force_path))


class Context:
    """A libsparoa context on one device; calls follow the current torch stream."""

    def __init__(self, device: int = 0):
        self.device = device
        h = ctypes.c_void_p()
        with torch.cuda.device(device):
            st = _lib.sparoa_create(ctypes.byref(h), device, ctypes.c_void_p(self._stream()))
        if st != OK:
            raise SparoaError(st, "sparoa_create")
        self.h = h

    def _stream(self):
        return torch.cuda.current_stream(self.device).cuda_stream

    def _check(self, st):
        if st != OK:
            raise SparoaError(st, _lib.sparoa_last_error(self.h).decode())

    def _bind(self):
        self._check(_lib.sparoa_set_stream(self.h, ctypes.c_void_p(self._stream())))

    def close(self):
        if getattr(self, "h", None):
            _lib.sparoa_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def sync(self):
        self._check(_lib.sparoa_sync(self.h))

    def last_path(self) -> int:
        """The path the last sparoa_gemm / sparoa_conv2d call took (synchronises)."""
        p = _I32(0)
        self._check(_lib.sparoa_last_path(self.h, ctypes.byref(p)))
        return int(p.value)

    def set_overlap(self, enable: bool):
        """Programmatic dependent launch between consecutive kernels (default on)."""
        self._check(_lib.sparoa_set_overlap(self.h, 1 if enable else 0))

    def set_wait_limit(self, cycles: int):
        """SM cycles before a kernel's bounded wait gives up (0 = default)."""
        self._check(_lib.sparoa_set_wait_limit(self.h, int(cycles)))

    def set_fault(self, code: int):
        """Error-path tests: 1 = withhold the first accumulator signal
        (timeout), 2 = fail the next workspace allocation, 0 = off."""
        self._check(_lib.sparoa_set_fault(self.h, int(code)))


class OccupancyBuffer:
    """Device occupancy block of a [R, C] tensor (caller-owned torch storage)."""

    def __init__(self, R: int, C: int, device="cuda"):
        nbytes = int(_lib.sparoa_occupancy_bytes(R, C))
        self.buf = torch.zeros(max(nbytes, 16), dtype=torch.uint8, device=device)
        self.occ = Occupancy()
        st = _lib.sparoa_occupancy_init(ctypes.c_void_p(self.buf.data_ptr()), nbytes, R, C,
                                        ctypes.byref(self.occ))
        if st != OK:
            raise SparoaError(st, "sparoa_occupancy_init")
        self.R, self.C = R, C

    def to_host(self) -> dict:
        """Copy the block back: nnz, col_nnz, tile_nnz, row_bm, blk_mask (numpy)."""
        R, C = self.R, self.C
        T = (C + 63) // 64
        W64 = (T + 63) // 64
        RB = (R + 127) // 128
        C32 = (C + 31) // 32
        raw = self.buf.cpu().numpy()
        base = self.occ.nnz

        def view(ptr, dtype, n):
            off = ptr - base
            return raw[off:off + n * np.dtype(dtype).itemsize].view(dtype).copy()

        return {"nnz": int(view(self.occ.nnz, np.uint64, 1)[0]),
                "col_nnz": view(self.occ.col_nnz, np.uint32, C),
                "tile_nnz": view(self.occ.tile_nnz, np.uint32, T),
                "row_bm": view(self.occ.row_bm, np.uint64, R * W64).reshape(R, W64),
                "blk_mask": view(self.occ.blk_mask, np.uint32, RB * C32).reshape(RB, C32)}


def _occ(o):
    return None if o is None else ctypes.byref(o.occ)


def _epi(bias=None, bn=None, eps=1e-5, act=ACT_NONE, residual=None):
    return Epilogue(_ptr(bias), _ptr(bn), float(eps), int(act), _ptr(residual))


def sparoa_op_stats(ctx: Context, x, shape, consumer: Op | None = None, occ=None, host=True):
    """Eq. 1 statistics of x (NHWC shape (N, H, W, C) or (M, K))."""
    N, H, W, C = (shape[0], 1, 1, shape[1]) if len(shape) == 2 else shape
    ctx._bind()
    st = Stats() if host else None
    ctx._check(_lib.sparoa_op_stats(ctx.h, _ptr(x), N, H, W, C,
                                    ctypes.byref(consumer) if consumer is not None else None,
                                    _occ(occ), ctypes.byref(st) if host else None))
    return st


def sparoa_gemm(ctx: Context, x, W, y, W_kn=None, bias=None, bn=None, eps=1e-5, act=ACT_NONE,
                residual=None, thr: Thresholds | None = None, x_occ=None, y_occ=None, host=False):
    """y[M, N] = epilogue(x[M, K] W[N, K]^T) with threshold dispatch."""
    M, K = x.shape
    N = W.shape[0]
    ctx._bind()
    ep = _epi(bias, bn, eps, act, residual)
    st = Stats() if host else None
    ydt = F32 if y.dtype == torch.float32 else BF16
    ctx._check(_lib.sparoa_gemm(ctx.h, _ptr(x), M, K, _ptr(W), _ptr(W_kn), N, ctypes.byref(ep),
                                ctypes.byref(thr) if thr is not None else None, _ptr(y), ydt,
                                _occ(x_occ), _occ(y_occ), ctypes.byref(st) if host else None))
    return st


def sparoa_gemm_split(ctx: Context, x, W, y, xi, W_kn=None, bias=None, bn=None, eps=1e-5,
                      act=ACT_NONE, residual=None, x_occ=None, y_occ=None):
    """y = epilogue(x W^T) with rows [0, xi*M) (whole 128-row blocks) on the
    zero-skip kernel and the rest on the dense kernel, on two streams."""
    M, K = x.shape
    N = W.shape[0]
    ctx._bind()
    ep = _epi(bias, bn, eps, act, residual)
    ydt = F32 if y.dtype == torch.float32 else BF16
    ctx._check(_lib.sparoa_gemm_split(ctx.h, _ptr(x), M, K, _ptr(W), _ptr(W_kn), N, ctypes.byref(ep),
                                      float(xi), _ptr(y), ydt, _occ(x_occ), _occ(y_occ)))


def sparoa_conv2d(ctx: Context, x, w, y, stride=1, pad=0, groups=1, bias=None, bn=None, eps=1e-5,
                  act=ACT_NONE, residual=None, thr: Thresholds | None = None, x_occ=None,
                  y_occ=None, host=False):
    """NHWC conv: x [N, H, W, C_in], w [C_out, kh, kw, C_in/groups], y [N, Ho, Wo, C_out]."""
    N, H, Wd, Cin = x.shape
    Cout, kh, kw, _ = w.shape
    ctx._bind()
    ep = _epi(bias, bn, eps, act, residual)
    st = Stats() if host else None
    ctx._check(_lib.sparoa_conv2d(ctx.h, _ptr(x), N, H, Wd, Cin, _ptr(w), Cout, kh, kw, stride, pad,
                                  groups, ctypes.byref(ep),
                                  ctypes.byref(thr) if thr is not None else None, _ptr(y),
                                  _occ(x_occ), _occ(y_occ), ctypes.byref(st) if host else None))
    return st


def sparoa_maxpool2d(ctx: Context, x, y, k=3, stride=2, pad=1, y_occ=None):
    N, H, W, C = x.shape
    ctx._bind()
    ctx._check(_lib.sparoa_maxpool2d(ctx.h, _ptr(x), N, H, W, C, k, stride, pad, _ptr(y), _occ(y_occ)))


def sparoa_avgpool_global(ctx: Context, x, y, y_occ=None):
    N, H, W, C = x.shape
    ctx._bind()
    ctx._check(_lib.sparoa_avgpool_global(ctx.h, _ptr(x), N, H, W, C, _ptr(y), _occ(y_occ)))


def sparoa_bn_act(ctx: Context, x, y, bias=None, bn=None, eps=1e-5, act=ACT_NONE, residual=None,
                  y_occ=None):
    R = int(np.prod(x.shape[:-1]))
    C = x.shape[-1]
    ctx._bind()
    ep = _epi(bias, bn, eps, act, residual)
    ctx._check(_lib.sparoa_bn_act(ctx.h, _ptr(x), R, C, ctypes.byref(ep), _ptr(y), _occ(y_occ)))


def sparoa_layernorm(ctx: Context, x, y, gamma_beta=None, eps=1e-6, y_occ=None):
    """y = LN(x) over the last dimension; gamma_beta fp32 [2, C] or None."""
    R = int(np.prod(x.shape[:-1]))
    C = x.shape[-1]
    ctx._bind()
    ctx._check(_lib.sparoa_layernorm(ctx.h, _ptr(x), R, C, _ptr(gamma_beta), float(eps), _ptr(y),
                                     _occ(y_occ)))


def sparoa_attention(ctx: Context, qkv, y, heads, y_occ=None):
    """Multi-head self-attention: qkv [N, T, 3 D] (q | k | v per token), y [N, T, D]."""
    N, T, C3 = qkv.shape
    D = C3 // 3
    ctx._bind()
    ctx._check(_lib.sparoa_attention(ctx.h, _ptr(qkv), N, T, int(heads), D // int(heads), _ptr(y),
                                     _occ(y_occ)))


def sparoa_gemm_noalloc(x, W, y, W_kn=None, bias=None, bn=None, eps=1e-5, act=ACT_NONE,
                        residual=None, thr: Thresholds | None = None, host=False):
    """sparoa_gemm for callers that cannot allocate: no context, the input's
    occupancy lives in the library's static device array (see sparoa.h).
    Runs on the current torch stream of the current device."""
    M, K = x.shape
    N = W.shape[0]
    ep = _epi(bias, bn, eps, act, residual)
    st = Stats() if host else None
    ydt = F32 if y.dtype == torch.float32 else BF16
    rc = _lib.sparoa_gemm_noalloc(ctypes.c_void_p(torch.cuda.current_stream().cuda_stream),
                                  _ptr(x), M, K, _ptr(W), _ptr(W_kn), N, ctypes.byref(ep),
                                  ctypes.byref(thr) if thr is not None else None, _ptr(y), ydt,
                                  ctypes.byref(st) if host else None)
    if rc != OK:
        raise SparoaError(rc, "sparoa_gemm_noalloc")
    return st


# ---------------------------------------------------------------------------
# graphs
# ---------------------------------------------------------------------------
_KIND = {"layernorm": OP_LAYERNORM, "attention": OP_ATTENTION, "tokens": OP_TOKENS, "select": OP_SELECT,
         "conv": OP_CONV2D, "fc": OP_FC, "maxpool": OP_MAXPOOL, "avgpool": OP_AVGPOOL,
         "bn_act": OP_BN_ACT}


def bits_to_device(bits: np.ndarray, device="cuda") -> torch.Tensor:
    """uint16 bf16 bit patterns (numpy) -> torch bf16 tensor on the device."""
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)
    return t.to(device)


def device_to_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


class Graph:
    """Operator list uploaded to the device, ready for sparoa_run_graph."""

    def __init__(self, ops: list, device="cuda"):
        self.keep = []
        arr = (Op * len(ops))()
        for i, d in enumerate(ops):
            o = arr[i]
            o.kind = _KIND[d["kind"]]
            o.input = d.get("input", i)
            r = d.get("residual", -1)
            o.residual = -1 if r is None else r
            o.act = d.get("act", ACT_NONE)
            o.groups = d.get("groups", 1)
            if d["kind"] in ("conv", "fc"):
                o.c_in, o.c_out = d["cin"], d["cout"]
                w = bits_to_device(d["w"], device)
                self.keep.append(w)
                o.weight = w.data_ptr()
                if d.get("w_kn") is not None:
                    wk = bits_to_device(d["w_kn"], device)
                    self.keep.append(wk)
                    o.weight_kn = wk.data_ptr()
            if d["kind"] == "conv":
                o.kh = o.kw = d["k"]
                o.stride, o.pad = d["stride"], d["pad"]
            elif d["kind"] == "maxpool":
                o.kh = o.kw = d["k"]
                o.stride, o.pad = d["stride"], d["pad"]
            elif d["kind"] == "layernorm":
                if d.get("gamma_beta") is not None:
                    t = torch.from_numpy(np.ascontiguousarray(d["gamma_beta"], dtype=np.float32)).to(device)
                    self.keep.append(t)
                    o.bn = t.data_ptr()
                o.bn_eps = d.get("eps", 1e-6)
            elif d["kind"] == "attention":
                o.groups = d["heads"]
            elif d["kind"] == "tokens":
                c = bits_to_device(d["cls"], device)
                pos = torch.from_numpy(np.ascontiguousarray(d["pos"], dtype=np.float32)).to(device)
                self.keep += [c, pos]
                o.weight = c.data_ptr()
                o.bias = pos.data_ptr()
            elif d["kind"] == "select":
                o.pad = d.get("index", 0)
            for name in ("bias", "bn"):
                if d.get(name) is not None:
                    t = torch.from_numpy(np.ascontiguousarray(d[name], dtype=np.float32)).to(device)
                    self.keep.append(t)
                    setattr(o, name, t.data_ptr())
            o.bn_eps = d.get("eps", 1e-5)
            thr = d.get("thr", {}) or {}
            o.thr = Thresholds(thr.get("s_thr", 0.5), thr.get("c_thr", 32.0),
                               thr.get("intensity_mode", 0), thr.get("force_path", 0))
        self.ops = arr
        self.n = len(ops)


def sparoa_graph_workspace(ctx: Context, graph: Graph, x_shape) -> int:
    """Bytes of device workspace sparoa_run_graph needs for this input shape."""
    N, H, W, C = (int(v) for v in x_shape)
    out = ctypes.c_uint64(0)
    ctx._check(_lib.sparoa_graph_workspace(ctx.h, graph.ops, graph.n, N, H, W, C, ctypes.byref(out)))
    return int(out.value)


def sparoa_run_graph(ctx: Context, graph: Graph, x, y=None, records=False):
    """Run the graph on x (bf16 NHWC); returns the list of Record (records=True) or None."""
    N, H, W, C = x.shape
    ctx._bind()
    recs = (Record * graph.n)() if records else None
    ctx._check(_lib.sparoa_run_graph(ctx.h, graph.ops, graph.n, _ptr(x), N, H, W, C, _ptr(y),
                                     0 if y is None else y.numel() * y.element_size(), recs))
    return list(recs) if records else None


class _DevView:
    def __init__(self, ptr, shape, typestr):
        self.__cuda_array_interface__ = {"shape": tuple(shape), "typestr": typestr,
                                         "data": (int(ptr), False), "version": 2}


def view_device(ptr: int, shape, dtype=torch.bfloat16) -> torch.Tensor:
    """A torch view (no copy) of device memory owned by the library, e.g. a
    graph record's output; valid only as long as the library keeps it."""
    if dtype == torch.bfloat16:
        t = torch.as_tensor(_DevView(ptr, shape, "<i2"), device="cuda")
        return t.view(torch.bfloat16)
    typestr = {torch.float32: "<f4", torch.int32: "<i4", torch.uint8: "|u1"}[dtype]
    return torch.as_tensor(_DevView(ptr, shape, typestr), device="cuda")


def record_occupancy(rec: Record) -> dict:
    """Copy a graph record's output occupancy to the host (same layout as
    OccupancyBuffer.to_host)."""
    o = rec.out_occ.contents
    R, C = o.R, o.C
    raw = view_device(o.nnz, (int(o.bytes),), torch.uint8).cpu().numpy()
    base = o.nnz
    T = (C + 63) // 64
    W64 = (T + 63) // 64
    RB = (R + 127) // 128
    C32 = (C + 31) // 32

    def view(ptr, dt, n):
        off = ptr - base
        return raw[off:off + n * np.dtype(dt).itemsize].view(dt).copy()

    return {"nnz": int(view(o.nnz, np.uint64, 1)[0]), "col_nnz": view(o.col_nnz, np.uint32, C),
            "tile_nnz": view(o.tile_nnz, np.uint32, T),
            "row_bm": view(o.row_bm, np.uint64, R * W64).reshape(R, W64),
            "blk_mask": view(o.blk_mask, np.uint32, RB * C32).reshape(RB, C32)}

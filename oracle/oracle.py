"""Python face of the SparOA oracle (``sparoa_oracle.c``).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` use this module to check and time the CUDA
path.  It never imports the product package's CUDA binding and the product
never imports it.

Everything here is a thin ctypes wrapper around the plain C functions, plus
``run_graph``, which walks a topologically ordered operator list in Python
(the paper's operator execution order, Sec. 4.1 "layer execution order") and
rounds every operator output to bf16, the storage type of an activation.
Tensors are numpy arrays: bf16 values travel as their uint16 bit patterns.

Citations are to sections and equations of the SparOA paper (arXiv 2511.19457).

Pins: every operator is pinned by tests/test_oracle_pins.py and
tests/test_oracle_vit_pins.py (closed forms, brute force, textbook values,
Table 2's MAC counts).  ``run_graph``'s chained output is the composition of
those operators with bf16 rounding between them; networks with random weights
have no published outputs, so beyond that composition its parity is
unpinned ("parity unpinned").
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "sparoa_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

PATH_NONE, PATH_DENSE, PATH_SKIP, PATH_DEPTHWISE = 0, 1, 2, 3
ACT_NONE, ACT_RELU, ACT_RELU6, ACT_GELU = 0, 1, 2, 3


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (C11, OpenMP, no FP contraction)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fopenmp",
               "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        I64 = ctypes.c_int64
        D = ctypes.c_double
        I = ctypes.c_int
        lib.orc_bf16_to_f64.restype = D
        lib.orc_bf16_to_f64.argtypes = [ctypes.c_uint16]
        lib.orc_f64_to_bf16.restype = ctypes.c_uint16
        lib.orc_f64_to_bf16.argtypes = [D]
        lib.orc_f64_to_bf16_array.argtypes = [P, P, I64]
        lib.orc_bf16_to_f64_array.argtypes = [P, P, I64]
        lib.orc_stats.argtypes = [P, I64, I64, P, P, P, P, P]
        lib.orc_conv_work.argtypes = [I64] * 10 + [P] * 5
        lib.orc_fc_work.argtypes = [I64, I64, I64, P, P, P]
        lib.orc_decide.restype = I
        lib.orc_decide.argtypes = [ctypes.c_uint64, ctypes.c_uint64, D, ctypes.c_uint64, D, D, I, I]
        lib.orc_conv2d.argtypes = [P, I64, I64, I64, I64, P, I64, I64, I64, I64, I64, I64,
                                   P, P, D, P, I, I, P]
        lib.orc_fc.argtypes = [P, I64, I64, P, I64, P, P, D, P, I, I, P]
        lib.orc_maxpool.argtypes = [P, I64, I64, I64, I64, I64, I64, I64, P]
        lib.orc_avgpool_global.argtypes = [P, I64, I64, I64, I64, P]
        lib.orc_bn_act.argtypes = [P, I64, I64, P, P, D, P, I, P]
        lib.orc_num_threads.restype = I
        lib.orc_set_num_threads.argtypes = [I]
        _lib = lib
        return lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _u16(a):
    a = np.ascontiguousarray(a)
    assert a.dtype == np.uint16, a.dtype
    return a


def _f32(a):
    return None if a is None else np.ascontiguousarray(a, dtype=np.float32)


def num_threads() -> int:
    return _load().orc_num_threads()


def set_num_threads(n: int) -> None:
    _load().orc_set_num_threads(int(n))


# --------------------------------------------------------------------------
# bf16 conversion
# --------------------------------------------------------------------------
def bf16_to_f64(bits) -> np.ndarray:
    """Exact value of each bf16 bit pattern."""
    b = _u16(np.asarray(bits, dtype=np.uint16))
    out = np.empty(b.shape, dtype=np.float64)
    _load().orc_bf16_to_f64_array(_ptr(b), _ptr(out), b.size)
    return out


def f64_to_bf16(values) -> np.ndarray:
    """Round doubles to bf16 (round to nearest, ties to even)."""
    v = np.ascontiguousarray(values, dtype=np.float64)
    out = np.empty(v.shape, dtype=np.uint16)
    _load().orc_f64_to_bf16_array(_ptr(v), _ptr(out), v.size)
    return out


# --------------------------------------------------------------------------
# Eq. 1 statistics
# --------------------------------------------------------------------------
@dataclass
class Stats:
    """Eq. 1 count and the occupancy bitmaps of a tensor viewed as [R, C]."""
    R: int
    C: int
    nnz: int
    col_nnz: np.ndarray
    tile_nnz: np.ndarray
    row_bm: np.ndarray
    blk_mask: np.ndarray

    @property
    def numel(self) -> int:
        return self.R * self.C

    @property
    def sparsity(self) -> float:
        """rho = 1 - c(O)/n(O) (Eq. 1)."""
        return 1.0 - self.nnz / self.numel if self.numel else 0.0


def stats(x_bits, R: int, C: int) -> Stats:
    x = _u16(np.asarray(x_bits).reshape(-1))
    assert x.size == R * C
    T = (C + 63) // 64
    W64 = (T + 63) // 64
    RB = (R + 127) // 128
    C32 = (C + 31) // 32
    nnz = np.zeros(1, dtype=np.uint64)
    col = np.zeros(max(C, 1), dtype=np.uint32)
    tile = np.zeros(max(T, 1), dtype=np.uint32)
    row = np.zeros(max(R * W64, 1), dtype=np.uint64)
    blk = np.zeros(max(RB * C32, 1), dtype=np.uint32)
    _load().orc_stats(_ptr(x), R, C, _ptr(nnz), _ptr(col), _ptr(tile), _ptr(row), _ptr(blk))
    return Stats(R, C, int(nnz[0]), col[:C], tile[:T], row[:R * W64].reshape(R, W64),
                 blk[:RB * C32].reshape(RB, C32))


# --------------------------------------------------------------------------
# Eq. 2 work and the threshold rule
# --------------------------------------------------------------------------
@dataclass
class Work:
    flops: int
    macs_eq2: int
    input_bytes: int
    Ho: int = 1
    Wo: int = 1

    @property
    def flops_per_byte(self) -> float:
        return self.flops / self.input_bytes if self.input_bytes else 0.0


def conv_work(N, H, W, Cin, Cout, kh, kw, stride, pad, groups=1) -> Work:
    out = [np.zeros(1, dtype=np.uint64) for _ in range(3)] + [np.zeros(1, dtype=np.int64) for _ in range(2)]
    _load().orc_conv_work(N, H, W, Cin, Cout, kh, kw, stride, pad, groups, *[_ptr(o) for o in out])
    return Work(int(out[0][0]), int(out[1][0]), int(out[2][0]), int(out[3][0]), int(out[4][0]))


def fc_work(M, K, N) -> Work:
    out = [np.zeros(1, dtype=np.uint64) for _ in range(3)]
    _load().orc_fc_work(M, K, N, *[_ptr(o) for o in out])
    return Work(int(out[0][0]), int(out[1][0]), int(out[2][0]))


def decide(numel: int, nnz: int, fpb: float, macs_eq2: int, s_thr: float, c_thr: float,
           intensity_mode: int = 0, force_path: int = 0) -> int:
    return int(_load().orc_decide(numel, nnz, float(fpb), macs_eq2, float(s_thr), float(c_thr),
                                  int(intensity_mode), int(force_path)))


# --------------------------------------------------------------------------
# Operators (fp64 results; round with f64_to_bf16 when the storage type is bf16)
# --------------------------------------------------------------------------
def conv2d(x_bits, N, H, W, Cin, w_bits, Cout, kh, kw, stride, pad, groups=1, bias=None,
           bn=None, eps=1e-5, residual_bits=None, act=ACT_NONE, skip_zeros=False) -> np.ndarray:
    """NHWC conv; returns y[N, Ho, Wo, Cout] in fp64."""
    x = _u16(np.asarray(x_bits).reshape(-1))
    w = _u16(np.asarray(w_bits).reshape(-1))
    assert x.size == N * H * W * Cin and w.size == Cout * kh * kw * (Cin // groups)
    Ho = (H + 2 * pad - kh) // stride + 1
    Wo = (W + 2 * pad - kw) // stride + 1
    y = np.empty((N, Ho, Wo, Cout), dtype=np.float64)
    b = _f32(bias)
    bnv = _f32(bn)
    res = None if residual_bits is None else _u16(np.asarray(residual_bits).reshape(-1))
    _load().orc_conv2d(_ptr(x), N, H, W, Cin, _ptr(w), Cout, kh, kw, stride, pad, groups,
                       _ptr(b), _ptr(bnv), float(eps), _ptr(res), int(act), int(bool(skip_zeros)),
                       _ptr(y))
    return y


def fc(x_bits, M, K, w_bits, N, bias=None, bn=None, eps=1e-5, residual_bits=None,
       act=ACT_NONE, skip_zeros=False) -> np.ndarray:
    """y[M, N] = x[M, K] W[N, K]^T + epilogue, in fp64."""
    x = _u16(np.asarray(x_bits).reshape(-1))
    w = _u16(np.asarray(w_bits).reshape(-1))
    assert x.size == M * K and w.size == N * K
    y = np.empty((M, N), dtype=np.float64)
    b = _f32(bias)
    bnv = _f32(bn)
    res = None if residual_bits is None else _u16(np.asarray(residual_bits).reshape(-1))
    _load().orc_fc(_ptr(x), M, K, _ptr(w), N, _ptr(b), _ptr(bnv), float(eps), _ptr(res), int(act),
                   int(bool(skip_zeros)), _ptr(y))
    return y


def maxpool(x_bits, N, H, W, C, k, stride, pad) -> np.ndarray:
    x = _u16(np.asarray(x_bits).reshape(-1))
    Ho = (H + 2 * pad - k) // stride + 1
    Wo = (W + 2 * pad - k) // stride + 1
    y = np.empty((N, Ho, Wo, C), dtype=np.float64)
    _load().orc_maxpool(_ptr(x), N, H, W, C, k, stride, pad, _ptr(y))
    return y


def avgpool_global(x_bits, N, H, W, C) -> np.ndarray:
    x = _u16(np.asarray(x_bits).reshape(-1))
    y = np.empty((N, C), dtype=np.float64)
    _load().orc_avgpool_global(_ptr(x), N, H, W, C, _ptr(y))
    return y


def bn_act(x_bits, R, C, bias=None, bn=None, eps=1e-5, residual_bits=None, act=ACT_NONE):
    x = _u16(np.asarray(x_bits).reshape(-1))
    y = np.empty((R, C), dtype=np.float64)
    res = None if residual_bits is None else _u16(np.asarray(residual_bits).reshape(-1))
    _load().orc_bn_act(_ptr(x), R, C, _ptr(_f32(bias)), _ptr(_f32(bn)), float(eps), _ptr(res),
                       int(act), _ptr(y))
    return y


# --------------------------------------------------------------------------
# Vision-transformer operators (the attention-based models of Sec. 6, Table 2:
# ViT-B16).  Plain fp64 definitions on the bf16 input values.
# --------------------------------------------------------------------------
def gelu(v):
    """GELU, exact form: v * Phi(v), Phi the standard normal CDF."""
    v = np.asarray(v, dtype=np.float64)
    erf = np.vectorize(__import__("math").erf, otypes=[np.float64])
    return 0.5 * v * (1.0 + erf(v / np.sqrt(2.0)))


def layernorm(x_bits, R, C, gamma_beta=None, eps=1e-6):
    """Layer normalisation (the LN of Sec. 3.2's encoder): per row, the C values
    minus their mean, over sqrt(biased variance + eps); then gamma * . + beta
    (gamma_beta fp32 [2, C]; None = 1, 0)."""
    x = bf16_to_f64(x_bits).reshape(R, C)
    mu = x.mean(axis=1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=1, keepdims=True)
    y = (x - mu) / np.sqrt(var + eps)
    if gamma_beta is not None:
        gb = np.asarray(gamma_beta, dtype=np.float64).reshape(2, C)
        y = y * gb[0] + gb[1]
    return y


def attention(qkv_bits, N, T, heads, hd):
    """Multi-head self-attention (the MHSA of Sec. 3.2's encoder) on the token
    rows of one projection: row t of image n holds q | k | v, each of heads x hd
    values; per head, out = softmax(Q K^T / sqrt(hd)) V; heads concatenated."""
    x = bf16_to_f64(qkv_bits).reshape(N, T, 3, heads, hd)
    q, k, v = x[:, :, 0], x[:, :, 1], x[:, :, 2]
    s = np.einsum("nthd,nshd->nhts", q, k) / np.sqrt(hd)
    s = s - s.max(axis=-1, keepdims=True)
    e = np.exp(s)
    p = e / e.sum(axis=-1, keepdims=True)
    return np.einsum("nhts,nshd->nthd", p, v).reshape(N, T, heads * hd)


def tokens(x_bits, N, P, D, cls_bits, pos):
    """Token sequence of a patch embedding: row 0 the class token, rows 1..P the
    P patch vectors, each plus its position embedding (pos fp32 [1 + P, D])."""
    x = bf16_to_f64(x_bits).reshape(N, P, D)
    cls = bf16_to_f64(cls_bits).reshape(1, 1, D)
    seq = np.concatenate([np.broadcast_to(cls, (N, 1, D)), x], axis=1)
    return seq + np.asarray(pos, dtype=np.float64).reshape(1, P + 1, D)


def select_token(x_bits, N, T, D, index):
    """Token `index` of every image: [N, T, D] -> [N, D]."""
    return bf16_to_f64(x_bits).reshape(N, T, D)[:, index, :]


# --------------------------------------------------------------------------
# Graph walk
# --------------------------------------------------------------------------
@dataclass
class OpRecord:
    """What the oracle decided and produced for one operator."""
    kind: str
    path: int
    in_stats: Stats
    work: Work | None
    out_shape: tuple
    out_f64: np.ndarray = field(repr=False)
    out_bits: np.ndarray = field(repr=False)


def run_op(op: dict, x_bits: np.ndarray, x_shape: tuple, residual_bits=None,
           skip_zeros_on_skip_path: bool = True) -> OpRecord:
    """Run one operator of a graph description on a bf16 input.

    ``op`` is a plain dict (see the workload builders): kind in
    {"conv", "fc", "maxpool", "avgpool", "bn_act", "layernorm", "attention",
    "tokens", "select"}, plus the layer geometry,
    bf16 weights (uint16), fp32 bias / bn, activation and thresholds.
    """
    kind = op["kind"]
    thr = op.get("thr", {})
    s_thr = thr.get("s_thr", 0.5)
    c_thr = thr.get("c_thr", 32.0)
    mode = thr.get("intensity_mode", 0)
    force = thr.get("force_path", 0)
    if kind == "conv":
        N, H, W, Cin = x_shape
        st = stats(x_bits, N * H * W, Cin)
        g = op.get("groups", 1)
        wk = conv_work(N, H, W, Cin, op["cout"], op["k"], op["k"], op["stride"], op["pad"], g)
        if g == 1:
            path = decide(st.numel, st.nnz, wk.flops_per_byte, wk.macs_eq2, s_thr, c_thr, mode, force)
        else:
            path = PATH_DEPTHWISE
        y = conv2d(x_bits, N, H, W, Cin, op["w"], op["cout"], op["k"], op["k"], op["stride"],
                   op["pad"], g, op.get("bias"), op.get("bn"), op.get("eps", 1e-5), residual_bits,
                   op.get("act", ACT_NONE), skip_zeros=(path == PATH_SKIP and skip_zeros_on_skip_path))
        shape = (N, wk.Ho, wk.Wo, op["cout"])
    elif kind == "fc":
        if len(x_shape) == 4:
            M = x_shape[0]
            K = int(np.prod(x_shape[1:]))
        else:
            M, K = x_shape
        st = stats(x_bits, M, K)
        wk = fc_work(M, K, op["cout"])
        path = decide(st.numel, st.nnz, wk.flops_per_byte, wk.macs_eq2, s_thr, c_thr, mode, force)
        y = fc(x_bits, M, K, op["w"], op["cout"], op.get("bias"), op.get("bn"), op.get("eps", 1e-5),
               residual_bits, op.get("act", ACT_NONE),
               skip_zeros=(path == PATH_SKIP and skip_zeros_on_skip_path))
        shape = (M, op["cout"])
    elif kind == "maxpool":
        N, H, W, C = x_shape
        st = stats(x_bits, N * H * W, C)
        wk = None
        path = PATH_NONE
        y = maxpool(x_bits, N, H, W, C, op["k"], op["stride"], op["pad"])
        shape = y.shape
    elif kind == "avgpool":
        N, H, W, C = x_shape
        st = stats(x_bits, N * H * W, C)
        wk = None
        path = PATH_NONE
        y = avgpool_global(x_bits, N, H, W, C)
        shape = y.shape
    elif kind == "bn_act":
        R = int(np.prod(x_shape[:-1]))
        C = x_shape[-1]
        st = stats(x_bits, R, C)
        wk = None
        path = PATH_NONE
        y = bn_act(x_bits, R, C, op.get("bias"), op.get("bn"), op.get("eps", 1e-5), residual_bits,
                   op.get("act", ACT_NONE)).reshape(x_shape)
        shape = tuple(x_shape)
    elif kind == "layernorm":
        R = int(np.prod(x_shape[:-1]))
        C = x_shape[-1]
        st = stats(x_bits, R, C)
        wk = None
        path = PATH_NONE
        y = layernorm(x_bits, R, C, op.get("gamma_beta"), op.get("eps", 1e-6))
        shape = tuple(x_shape)
    elif kind == "attention":
        N, H, W, C3 = x_shape
        T = H * W
        heads = op["heads"]
        hd = C3 // 3 // heads
        st = stats(x_bits, N * T, C3)
        wk = None
        path = PATH_NONE
        y = attention(x_bits, N, T, heads, hd)
        shape = (N, H, W, C3 // 3)
    elif kind == "tokens":
        N, H, W, D = x_shape
        st = stats(x_bits, N * H * W, D)
        wk = None
        path = PATH_NONE
        y = tokens(x_bits, N, H * W, D, op["cls"], op["pos"])
        shape = (N, 1, H * W + 1, D)
    elif kind == "select":
        N, H, W, D = x_shape
        st = stats(x_bits, N * H * W, D)
        wk = None
        path = PATH_NONE
        y = select_token(x_bits, N, H * W, D, op.get("index", 0))
        shape = (N, 1, 1, D)
    else:
        raise ValueError(f"unknown operator kind {kind!r}")
    bits = f64_to_bf16(y).reshape(shape)
    return OpRecord(kind, path, st, wk, tuple(shape), y.reshape(shape), bits)


def run_graph(ops: list, x_bits: np.ndarray, x_shape: tuple, teacher=None) -> list:
    """Walk ``ops`` in order.  Value 0 is the graph input and value i+1 the
    output of op i; ``op["input"]`` and ``op.get("residual")`` name values.

    ``teacher`` (optional) maps a value index to bf16 bits to use instead of
    the oracle's own value; parity tests feed the GPU's activations here so
    that each operator is checked on exactly the tensor the GPU saw.
    """
    values = {0: (np.asarray(x_bits), tuple(x_shape))}
    records = []
    for i, op in enumerate(ops):
        src = op.get("input", i)
        xb, xs = values[src]
        if teacher is not None and src in teacher:
            xb = teacher[src]
        res = None
        if op.get("residual", -1) is not None and op.get("residual", -1) >= 0:
            r = op["residual"]
            res = values[r][0] if teacher is None or r not in teacher else teacher[r]
        rec = run_op(op, xb, xs, res)
        records.append(rec)
        values[i + 1] = (rec.out_bits, rec.out_shape)
    return records

"""Python binding of libseedq.so: argument marshalling only.

Every function forwards to the C ABI declared in include/seedq.h under the same
name; all computation happens in the library's CUDA kernels.  Device buffers
are passed as torch tensors (their data_ptr) or raw integer addresses, and the
CUDA stream as torch.cuda.Stream / raw handle / None (torch's current stream).
If the library is missing this module raises at import of the handle: there is
no fallback path.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libseedq.so")
_lib = None

STATUS = {0: "SEEDQ_OK", 1: "SEEDQ_ERR_INVALID_ARG", 2: "SEEDQ_ERR_STREAM",
          3: "SEEDQ_ERR_SCHEDULE", 4: "SEEDQ_ERR_CUDA", 5: "SEEDQ_ERR_NOMEM",
          6: "SEEDQ_ERR_UNSUPPORTED", 7: "SEEDQ_ERR_IO", 8: "SEEDQ_ERR_FORMAT"}


class SeedQError(RuntimeError):
    def __init__(self, status: int, where: str):
        msg = lib().seedq_status_string(status).decode()
        if status == 4:
            msg += ": " + lib().seedq_last_cuda_error_string().decode()
        super().__init__(f"{where}: {STATUS.get(status, status)} ({msg})")
        self.status = status


class Rung(C.Structure):
    _fields_ = [("S", C.c_int32), ("k", C.c_int32)]


class Schedule(C.Structure):
    _fields_ = [("J", C.c_int32), ("rungs", C.POINTER(Rung)), ("theta", C.POINTER(C.c_double)),
                ("j_tie", C.c_int32), ("q", C.c_double)]


class LayerDesc(C.Structure):
    _fields_ = [("rows", C.c_int64), ("cols", C.c_int64), ("a", C.POINTER(C.c_float)),
                ("rho", C.POINTER(C.c_float)), ("tie_count", C.c_int64),
                ("n_outliers", C.c_int32), ("outlier_cols", C.POINTER(C.c_int32)),
                ("outlier_vals", C.c_void_p), ("max_batch", C.c_int32)]


class ContainerTensor(C.Structure):
    _fields_ = [("name", C.c_char_p), ("rows", C.c_int64), ("cols", C.c_int64),
                ("a", C.POINTER(C.c_float)), ("rho", C.POINTER(C.c_float)), ("tie_count", C.c_int64),
                ("n_outliers", C.c_int32), ("outlier_cols", C.POINTER(C.c_int32)),
                ("outlier_vals", C.POINTER(C.c_uint16)), ("stream", C.POINTER(C.c_uint8)),
                ("stream_bits", C.c_uint64)]


class LlamaLayer(C.Structure):
    _fields_ = [("attn_norm", C.c_void_p), ("mlp_norm", C.c_void_p), ("wq", C.c_void_p),
                ("wk", C.c_void_p), ("wv", C.c_void_p), ("wo", C.c_void_p), ("wgate", C.c_void_p),
                ("wup", C.c_void_p), ("wdown", C.c_void_p)]


class LlamaModel(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("d_model", C.c_int32), ("n_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("d_ff", C.c_int32),
                ("vocab", C.c_int64), ("layers", C.POINTER(LlamaLayer)),
                ("final_norm", C.c_void_p), ("lm_head", C.c_void_p)]


class ImportanceOut(C.Structure):
    _fields_ = [("a_o", C.c_void_p), ("a_down", C.c_void_p), ("rho_o", C.c_void_p),
                ("rho_down", C.c_void_p), ("dyn_range", C.c_void_p), ("act_ratio", C.c_void_p)]


class Outlier(C.Structure):
    _fields_ = [("tensor", C.c_int32), ("column", C.c_int32)]


class FactorDesc(C.Structure):
    _fields_ = [("rows", C.c_int64), ("cols", C.c_int64), ("a", C.POINTER(C.c_float)),
                ("rho", C.POINTER(C.c_float))]


# Every symbol include/seedq.h declares, with its ctypes signature.
SIGNATURES = {
    "seedq_layer_prepare": (C.c_int, [C.POINTER(LayerDesc), C.POINTER(Schedule), C.c_void_p,
                                      C.POINTER(C.c_void_p)]),
    "seedq_layer_stream_bits": (C.c_int, [C.c_void_p, C.POINTER(C.c_uint64)]),
    "seedq_stream_bytes_required": (C.c_uint64, [C.c_uint64]),
    "seedq_layer_bind_stream": (C.c_int, [C.c_void_p, C.c_void_p, C.c_uint64, C.c_uint64]),
    "seedq_layer_limit_stream_bytes": (C.c_int, [C.c_void_p, C.c_uint64]),
    "seedq_fp64_fma_probe": (C.c_int, [C.c_int64, C.c_int32, C.c_void_p, C.c_void_p,
                                       C.POINTER(C.c_int64)]),
    "seedq_layer_release": (C.c_int, [C.c_void_p]),
    "seedq_decode_weights": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p]),
    "seedq_decode_rows": (C.c_int, [C.c_void_p, C.c_int64, C.c_int64, C.c_void_p, C.c_void_p]),
    "seedq_gemv": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "seedq_gemm_small_batch": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p]),
    "seedq_gemm_multi": (C.c_int, [C.POINTER(C.c_void_p), C.c_int32, C.POINTER(C.c_void_p),
                                   C.c_int32, C.POINTER(C.c_void_p), C.c_void_p]),
    "seedq_layer_rung_map": (C.c_int, [C.c_void_p, C.c_int64, C.c_int64, C.c_void_p]),
    "seedq_layer_perm": (C.c_int, [C.c_void_p, C.c_void_p]),
    "seedq_layer_row_offsets": (C.c_int, [C.c_void_p, C.c_void_p]),
    "seedq_last_device_error": (C.c_int, [C.c_void_p, C.POINTER(C.c_uint32)]),
    "seedq_lfsr_taps": (C.c_uint32, [C.c_int32]),
    "seedq_synth_stream": (C.c_int, [C.c_void_p, C.c_uint64, C.c_void_p, C.c_uint64, C.c_void_p]),
    "seedq_row_plan_static": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int64, C.c_int32,
                                        C.POINTER(Schedule), C.c_int64, C.c_void_p, C.c_void_p,
                                        C.c_void_p, C.c_void_p]),
    "seedq_encode_blocks": (C.c_int, [C.c_int32, C.c_int32, C.c_void_p, C.c_int64, C.c_void_p,
                                      C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "seedq_encode_layer": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                     C.c_void_p, C.c_void_p]),
    "seedq_pack_stream": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                    C.c_uint64, C.c_void_p]),
    "seedq_container_write": (C.c_int, [C.c_char_p, C.POINTER(Schedule), C.c_int32,
                                        C.POINTER(ContainerTensor)]),
    "seedq_container_open": (C.c_int, [C.c_char_p, C.POINTER(C.c_void_p)]),
    "seedq_container_schedule": (C.c_int, [C.c_void_p, C.POINTER(Schedule)]),
    "seedq_container_count": (C.c_int, [C.c_void_p, C.POINTER(C.c_int32)]),
    "seedq_container_get": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(ContainerTensor)]),
    "seedq_container_close": (C.c_int, [C.c_void_p]),
    "seedq_layer_set_create": (C.c_int, [C.POINTER(C.c_void_p), C.c_int32, C.POINTER(C.c_void_p)]),
    "seedq_layer_set_layout": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p]),
    "seedq_gemm_set": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p]),
    "seedq_layer_set_release": (C.c_int, [C.c_void_p]),
    "seedq_importance": (C.c_int, [C.POINTER(LlamaModel), C.POINTER(ImportanceOut),
                                   C.POINTER(Outlier), C.c_int32, C.POINTER(C.c_int32), C.c_void_p]),
    "seedq_column_stats": (C.c_int, [C.c_void_p, C.c_int64, C.c_int64, C.c_void_p, C.c_void_p,
                                     C.c_void_p, C.c_void_p]),
    "seedq_synth_fp16": (C.c_int, [C.c_uint64, C.c_int64, C.c_int64, C.c_int32, C.c_int32,
                                   C.c_void_p, C.c_void_p]),
    "seedq_allocate": (C.c_int, [C.POINTER(FactorDesc), C.c_int32, C.c_int32, C.c_void_p,
                                 C.c_void_p, C.c_void_p, C.c_double, C.c_double, C.c_void_p,
                                 C.POINTER(C.c_int32), C.POINTER(C.c_double), C.c_void_p,
                                 C.c_void_p, C.c_void_p]),
    "seedq_status_string": (C.c_char_p, [C.c_int]),
    "seedq_last_cuda_error_string": (C.c_char_p, []),
}


def lib():
    """The loaded libseedq.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: run __graft_entry__.build() "
                              "(there is no CPU fallback)")
        L = C.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _check(status: int, where: str):
    if status != 0:
        raise SeedQError(status, where)


def _ptr(t) -> int:
    if t is None:
        return 0
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(s) -> int:
    if s is None:
        import torch

        return torch.cuda.current_stream().cuda_stream
    if isinstance(s, int):
        return s
    return s.cuda_stream


def stream_bytes_required(bits: int) -> int:
    return lib().seedq_stream_bytes_required(bits)


def lfsr_taps(S: int) -> int:
    return lib().seedq_lfsr_taps(S)


class Layer:
    """One prepared tensor (seedq_layer_prepare ... seedq_layer_release)."""

    def __init__(self, rows, cols, a, rho, rungs, theta, j_tie, q, tie_count,
                 outlier_cols=None, outlier_vals=None, max_batch=0, stream=None):
        self.rows, self.cols = int(rows), int(cols)
        self._a = np.ascontiguousarray(a, np.float32)
        self._rho = None if rho is None else np.ascontiguousarray(rho, np.float32)
        self._rungs = (Rung * len(rungs))(*[Rung(int(S), int(k)) for S, k in rungs])
        self._theta = np.ascontiguousarray(theta, np.float64)
        if self._theta.size == 0:
            self._theta = np.zeros(1, np.float64)
        self._ocols = (np.zeros(1, np.int32) if outlier_cols is None
                       else np.ascontiguousarray(outlier_cols, np.int32))
        self._ovals = outlier_vals  # device tensor, kept alive with the layer
        n_out = 0 if outlier_cols is None else len(outlier_cols)
        desc = LayerDesc(self.rows, self.cols, self._a.ctypes.data_as(C.POINTER(C.c_float)),
                         None if self._rho is None else self._rho.ctypes.data_as(C.POINTER(C.c_float)),
                         int(tie_count), n_out, self._ocols.ctypes.data_as(C.POINTER(C.c_int32)),
                         _ptr(outlier_vals), int(max_batch))
        sched = Schedule(len(rungs), self._rungs, self._theta.ctypes.data_as(C.POINTER(C.c_double)),
                         int(j_tie), float(q))
        h = C.c_void_p()
        _check(lib().seedq_layer_prepare(C.byref(desc), C.byref(sched), _stream(stream), C.byref(h)),
               "seedq_layer_prepare")
        self.h = h
        self._stream_buf = None

    # -- lifetime ---------------------------------------------------------
    def release(self):
        if self.h is not None and self.h.value:
            _check(lib().seedq_layer_release(self.h), "seedq_layer_release")
        self.h = None

    def __del__(self):
        try:
            self.release()
        except Exception:
            pass

    # -- stream -----------------------------------------------------------
    @property
    def stream_bits(self) -> int:
        b = C.c_uint64()
        _check(lib().seedq_layer_stream_bits(self.h, C.byref(b)), "seedq_layer_stream_bits")
        return b.value

    def bind_stream(self, buf, bits: int, nbytes: int):
        _check(lib().seedq_layer_bind_stream(self.h, _ptr(buf), bits, nbytes), "seedq_layer_bind_stream")
        self._stream_buf = buf

    def limit_stream_bytes(self, nbytes: int):
        _check(lib().seedq_layer_limit_stream_bytes(self.h, nbytes), "seedq_layer_limit_stream_bytes")

    def synth_stream(self, key: int, buf, nbytes: int, stream=None):
        _check(lib().seedq_synth_stream(self.h, key, _ptr(buf), nbytes, _stream(stream)),
               "seedq_synth_stream")

    # -- hot calls --------------------------------------------------------
    def decode_weights(self, W, stream=None):
        _check(lib().seedq_decode_weights(self.h, _ptr(W), _stream(stream)), "seedq_decode_weights")

    def decode_rows(self, row0: int, nrows: int, W, stream=None):
        _check(lib().seedq_decode_rows(self.h, row0, nrows, _ptr(W), _stream(stream)), "seedq_decode_rows")

    def gemv(self, x, y, stream=None):
        _check(lib().seedq_gemv(self.h, _ptr(x), _ptr(y), _stream(stream)), "seedq_gemv")

    def gemm_small_batch(self, X, n: int, Y, stream=None):
        _check(lib().seedq_gemm_small_batch(self.h, _ptr(X), n, _ptr(Y), _stream(stream)),
               "seedq_gemm_small_batch")

    def encode(self, W, seed, E, t, err=None, stream=None):
        _check(lib().seedq_encode_layer(self.h, _ptr(W), _ptr(seed), _ptr(E), _ptr(t), _ptr(err),
                                        _stream(stream)), "seedq_encode_layer")

    def pack_stream(self, seed, E, t, buf, nbytes: int, stream=None):
        _check(lib().seedq_pack_stream(self.h, _ptr(seed), _ptr(E), _ptr(t), _ptr(buf), nbytes,
                                       _stream(stream)), "seedq_pack_stream")

    # -- introspection (synchronous) --------------------------------------
    def rung_map(self, row0: int = 0, nrows: int | None = None) -> np.ndarray:
        nrows = self.rows - row0 if nrows is None else nrows
        out = np.zeros((nrows, self.cols // 8), np.uint8)
        _check(lib().seedq_layer_rung_map(self.h, row0, nrows, out.ctypes.data), "seedq_layer_rung_map")
        return out

    def perm(self) -> np.ndarray:
        out = np.zeros(self.cols, np.int32)
        _check(lib().seedq_layer_perm(self.h, out.ctypes.data), "seedq_layer_perm")
        return out

    def row_offsets(self) -> np.ndarray:
        out = np.zeros(self.rows + 1, np.uint64)
        _check(lib().seedq_layer_row_offsets(self.h, out.ctypes.data), "seedq_layer_row_offsets")
        return out

    def device_error(self) -> int:
        f = C.c_uint32()
        _check(lib().seedq_last_device_error(self.h, C.byref(f)), "seedq_last_device_error")
        return f.value


STATIC_PLAN_MAX_ROWS = 1 << 17


def row_plan_static(abar, rho, rows: int, nb: int, rungs, theta, j_tie: int, q: float,
                    tie_count: int, brk, row_off, summary, stream=None):
    """seedq_row_plan_static: the allocation-free row pass (device buffers in/out)."""
    rr = (Rung * len(rungs))(*[Rung(int(S), int(k)) for S, k in rungs])
    th = np.ascontiguousarray(theta if len(theta) else [0.0], np.float64)
    sched = Schedule(len(rungs), rr, th.ctypes.data_as(C.POINTER(C.c_double)), int(j_tie), float(q))
    _check(lib().seedq_row_plan_static(_ptr(abar), _ptr(rho), rows, nb, C.byref(sched), tie_count,
                                       _ptr(brk), _ptr(row_off), _ptr(summary), _stream(stream)),
           "seedq_row_plan_static")


def gemm_multi(layers, X, n: int, Y, stream=None):
    """seedq_gemm_multi: Y[i] = X[i] W_hat_i^T for several layers in one launch."""
    cnt = len(layers)
    lh = (C.c_void_p * cnt)(*[l.h.value for l in layers])
    xh = (C.c_void_p * cnt)(*[_ptr(x) for x in X])
    yh = (C.c_void_p * cnt)(*[_ptr(y) for y in Y])
    _check(lib().seedq_gemm_multi(lh, cnt, xh, n, yh, _stream(stream)), "seedq_gemm_multi")


def encode_blocks(S: int, k: int, w, nblocks: int, seed, E, t, err=None, stream=None):
    """seedq_encode_blocks: exhaustive seed search of nblocks blocks at rung (S, k)."""
    _check(lib().seedq_encode_blocks(S, k, _ptr(w), nblocks, _ptr(seed), _ptr(E), _ptr(t), _ptr(err),
                                     _stream(stream)), "seedq_encode_blocks")


def fp64_fma_probe(iters: int, blocks_per_sm: int, out, stream=None) -> int:
    """seedq_fp64_fma_probe: launch the fp64 FMA rate probe; returns its FMA count."""
    n = C.c_int64()
    _check(lib().seedq_fp64_fma_probe(iters, blocks_per_sm, _ptr(out), _stream(stream), C.byref(n)),
           "seedq_fp64_fma_probe")
    return n.value


def synth_fp16(key: int, first: int, n: int, m: int, e: int, out, stream=None):
    """seedq_synth_fp16: n generated FP16 values into a device buffer."""
    _check(lib().seedq_synth_fp16(key & ((1 << 64) - 1), first, n, m, e, _ptr(out), _stream(stream)),
           "seedq_synth_fp16")


def column_stats(W, R: int, Cc: int, dyn_range, g=None, col_sq=None, stream=None):
    """seedq_column_stats: dynamic-range statistic (and weighted column sums of squares)."""
    _check(lib().seedq_column_stats(_ptr(W), R, Cc, _ptr(g), _ptr(dyn_range), _ptr(col_sq),
                                    _stream(stream)), "seedq_column_stats")


def importance(dims: dict, layers, final_norm, lm_head, out: dict, max_outliers: int = 4,
               stream=None):
    """seedq_importance over a resident FP16 model.

    dims: n_layers, d_model, n_heads, n_kv_heads, head_dim, d_ff, vocab.
    layers: per layer a dict of device buffers attn_norm, mlp_norm, wq, wk, wv,
    wo, wgate, wup, wdown.  out: device buffers a_o, a_down, rho_o, rho_down
    and optionally dyn_range, act_ratio.  Returns the outlier (tensor, column)
    pairs."""
    L = len(layers)
    arr = (LlamaLayer * L)(*[LlamaLayer(*[_ptr(y[k]) for k in (
        "attn_norm", "mlp_norm", "wq", "wk", "wv", "wo", "wgate", "wup", "wdown")]) for y in layers])
    m = LlamaModel(dims["n_layers"], dims["d_model"], dims["n_heads"], dims["n_kv_heads"],
                   dims["head_dim"], dims["d_ff"], dims["vocab"], arr, _ptr(final_norm), _ptr(lm_head))
    o = ImportanceOut(_ptr(out["a_o"]), _ptr(out["a_down"]), _ptr(out["rho_o"]), _ptr(out["rho_down"]),
                      _ptr(out.get("dyn_range")), _ptr(out.get("act_ratio")))
    res = (Outlier * max(max_outliers, 1))()
    n = C.c_int32(0)
    _check(lib().seedq_importance(C.byref(m), C.byref(o), res, max_outliers, C.byref(n),
                                  _stream(stream)), "seedq_importance")
    return [(res[i].tensor, res[i].column) for i in range(n.value)]


def allocate(factors, rungs, slopes, rbar: float, floor_f: float, stream=None):
    """seedq_allocate: Alg. 1's floor, multiplier bisection and tie pass over
    a list of (rows, cols, a, rho or None) host arrays.  Returns
    (theta, j_tie, q, tie_count, stream_bits)."""
    keep = []
    descs = (FactorDesc * len(factors))()
    for i, (R, Cc, a, rho) in enumerate(factors):
        a32 = np.ascontiguousarray(a, np.float32)
        keep.append(a32)
        rp = None
        if rho is not None:
            r32 = np.ascontiguousarray(rho, np.float32)
            keep.append(r32)
            rp = r32.ctypes.data_as(C.POINTER(C.c_float))
        descs[i] = FactorDesc(R, Cc, a32.ctypes.data_as(C.POINTER(C.c_float)), rp)
    J = len(rungs)
    S = np.asarray([r[0] for r in rungs], np.int32)
    k = np.asarray([r[1] for r in rungs], np.int32)
    sl = np.ascontiguousarray(slopes if len(slopes) else [1.0], np.float64)
    theta = np.zeros(max(J - 1, 1), np.float64)
    jt, q = C.c_int32(), C.c_double()
    T = np.zeros(len(factors), np.int64)
    bits = np.zeros(len(factors), np.uint64)
    _check(lib().seedq_allocate(descs, len(factors), J, S.ctypes.data, k.ctypes.data, sl.ctypes.data,
                                rbar, floor_f, theta.ctypes.data, C.byref(jt), C.byref(q),
                                T.ctypes.data, bits.ctypes.data, _stream(stream)), "seedq_allocate")
    return theta[:J - 1], jt.value, q.value, T, bits


class LayerSet:
    """seedq_layer_set_create ... _release: every layer of a model behind one
    launch per call; x / y of all tensors in one buffer each (see layout())."""

    def __init__(self, layers):
        self.layers = list(layers)  # kept alive with the set
        arr = (C.c_void_p * len(self.layers))(*[l.h.value for l in self.layers])
        h = C.c_void_p()
        _check(lib().seedq_layer_set_create(arr, len(self.layers), C.byref(h)), "seedq_layer_set_create")
        self.h = h
        co = np.zeros(len(self.layers) + 1, np.int64)
        ro = np.zeros(len(self.layers) + 1, np.int64)
        _check(lib().seedq_layer_set_layout(self.h, co.ctypes.data, ro.ctypes.data), "seedq_layer_set_layout")
        self.col_offsets, self.row_offsets = co, ro

    def gemm(self, X, n: int, Y, stream=None):
        _check(lib().seedq_gemm_set(self.h, _ptr(X), n, _ptr(Y), _stream(stream)), "seedq_gemm_set")

    def release(self):
        if self.h is not None and self.h.value:
            _check(lib().seedq_layer_set_release(self.h), "seedq_layer_set_release")
        self.h = None

    def __del__(self):
        try:
            self.release()
        except Exception:
            pass


# ------------------------------------------------------------ container

def container_write(path: str, rungs, theta, j_tie: int, q: float, tensors):
    """seedq_container_write.  tensors: dicts with name, a, rho (or None),
    tie_count, outlier_cols, outlier_vals (rows x n uint16) and the host
    stream bytes with its bit length."""
    rr = (Rung * len(rungs))(*[Rung(int(S), int(k)) for S, k in rungs])
    th = np.ascontiguousarray(theta if len(theta) else [0.0], np.float64)
    sched = Schedule(len(rungs), rr, th.ctypes.data_as(C.POINTER(C.c_double)), int(j_tie), float(q))
    keep, arr = [], (ContainerTensor * max(1, len(tensors)))()
    for i, t in enumerate(tensors):
        a = np.ascontiguousarray(t["a"], np.float32)
        rho = None if t.get("rho") is None else np.ascontiguousarray(t["rho"], np.float32)
        oc = np.ascontiguousarray(t.get("outlier_cols", np.zeros(0)), np.int32)
        ov = np.ascontiguousarray(t.get("outlier_vals", np.zeros(0)), np.uint16)
        st = np.ascontiguousarray(t["stream"], np.uint8)
        name = t.get("name", "").encode()
        keep += [a, rho, oc, ov, st, name]
        arr[i] = ContainerTensor(name, int(t["rows"]), int(t["cols"]),
                                 a.ctypes.data_as(C.POINTER(C.c_float)),
                                 None if rho is None else rho.ctypes.data_as(C.POINTER(C.c_float)),
                                 int(t["tie_count"]), int(oc.size),
                                 oc.ctypes.data_as(C.POINTER(C.c_int32)),
                                 ov.ctypes.data_as(C.POINTER(C.c_uint16)),
                                 st.ctypes.data_as(C.POINTER(C.c_uint8)), int(t["stream_bits"]))
    _check(lib().seedq_container_write(path.encode(), C.byref(sched), len(tensors), arr),
           "seedq_container_write")


class Container:
    """seedq_container_open ... seedq_container_close: a read-only view."""

    def __init__(self, path: str):
        h = C.c_void_p()
        _check(lib().seedq_container_open(path.encode(), C.byref(h)), "seedq_container_open")
        self.h = h
        s = Schedule()
        _check(lib().seedq_container_schedule(self.h, C.byref(s)), "seedq_container_schedule")
        self.rungs = [(s.rungs[j].S, s.rungs[j].k) for j in range(s.J)]
        self.theta = [s.theta[j] for j in range(s.J - 1)]
        self.j_tie, self.q = s.j_tie, s.q
        n = C.c_int32()
        _check(lib().seedq_container_count(self.h, C.byref(n)), "seedq_container_count")
        self.count = n.value

    def tensor(self, i: int) -> dict:
        t = ContainerTensor()
        _check(lib().seedq_container_get(self.h, i, C.byref(t)), "seedq_container_get")
        R, Cc, no = t.rows, t.cols, t.n_outliers
        nbytes = (t.stream_bits + 7) // 8
        return {
            "name": t.name.decode(), "rows": R, "cols": Cc,
            "a": np.ctypeslib.as_array(t.a, (Cc,)).copy(),
            "rho": None if not t.rho else np.ctypeslib.as_array(t.rho, (R,)).copy(),
            "tie_count": t.tie_count,
            "outlier_cols": np.ctypeslib.as_array(t.outlier_cols, (no,)).copy() if no else np.zeros(0, np.int32),
            "outlier_vals": (np.ctypeslib.as_array(t.outlier_vals, (R * no,)).reshape(R, no).copy()
                             if no else np.zeros((R, 0), np.uint16)),
            "stream": np.ctypeslib.as_array(t.stream, (nbytes,)).copy() if nbytes else np.zeros(0, np.uint8),
            "stream_bits": t.stream_bits,
        }

    def close(self):
        if self.h is not None and self.h.value:
            _check(lib().seedq_container_close(self.h), "seedq_container_close")
        self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def load_layers(path: str, max_batch: int = 1, stream=None):
    """Open a container and prepare one bound Layer per tensor (streams and
    outlier values uploaded to the current CUDA device).  Returns a list of
    (name, Layer)."""
    import torch

    c = Container(path)
    out = []
    try:
        for i in range(c.count):
            t = c.tensor(i)
            ov = None
            if len(t["outlier_cols"]):
                ov = torch.from_numpy(t["outlier_vals"].view(np.int16)).cuda()
            L = Layer(t["rows"], t["cols"], t["a"], t["rho"], c.rungs, c.theta, c.j_tie, c.q,
                      t["tie_count"], t["outlier_cols"] if len(t["outlier_cols"]) else None, ov,
                      max_batch=max_batch, stream=stream)
            L._ovals_keep = ov
            nbytes = stream_bytes_required(t["stream_bits"])
            buf = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
            if t["stream"].size:
                buf[:t["stream"].size].copy_(torch.from_numpy(t["stream"]))
            L.bind_stream(buf, t["stream_bits"], nbytes)
            out.append((t["name"], L))
    finally:
        c.close()
    return out

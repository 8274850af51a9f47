"""ctypes front end of the Seed-Q CPU oracle (``liboracle.so``).

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this module.  The product path
(the CUDA library and its binding) never does; the two share no code.

Every function here is a thin marshalling layer over the C oracle, whose
functions cite the passage of the paper they restate (see seedq_oracle.h).
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = ["codec.c", "schedule.c", "decode.c"]
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile liboracle.so in place (gcc, fp contraction off)."""
    srcs = [os.path.join(_HERE, s) for s in _SRC]
    hdr = os.path.join(_HERE, "seedq_oracle.h")
    if not force and os.path.exists(_LIB_PATH):
        newest = max(os.path.getmtime(p) for p in srcs + [hdr])
        if os.path.getmtime(_LIB_PATH) >= newest:
            return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
           "-o", tmp] + srcs + ["-lm", "-lpthread"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class Factors(C.Structure):
    _fields_ = [("R", C.c_int64), ("C", C.c_int64),
                ("perm", C.POINTER(C.c_int32)), ("abar", C.POINTER(C.c_double)),
                ("rho", C.POINTER(C.c_double)), ("rho_uniform", C.c_int)]


class Schedule(C.Structure):
    _fields_ = [("J", C.c_int), ("S", C.POINTER(C.c_int)), ("k", C.POINTER(C.c_int)),
                ("theta", C.POINTER(C.c_double)), ("j_tie", C.c_int), ("q", C.c_double)]


def _p(arr, ctype):
    return arr.ctypes.data_as(C.POINTER(ctype))


def lib():
    global _lib
    if _lib is None:
        build()
        L = C.CDLL(_LIB_PATH)
        u8p, u16p, i32p = C.POINTER(C.c_uint8), C.POINTER(C.c_uint16), C.POINTER(C.c_int32)
        u32p, u64p, i64p = C.POINTER(C.c_uint32), C.POINTER(C.c_uint64), C.POINTER(C.c_int64)
        dp, fp, ip = C.POINTER(C.c_double), C.POINTER(C.c_float), C.POINTER(C.c_int)
        FP, SP = C.POINTER(Factors), C.POINTER(Schedule)
        sig = {
            "or_block_bits": (C.c_int, [C.c_int, C.c_int]),
            "or_lfsr_bits": (None, [C.c_int, C.c_uint32, C.c_uint32, C.c_int, u8p]),
            "or_lfsr_period": (C.c_int64, [C.c_int, C.c_uint32]),
            "or_find_taps": (C.c_uint32, [C.c_int]),
            "or_reconstruct_block": (None, [C.c_int, C.c_int, C.c_uint32, C.c_uint32, C.c_int, ip, fp]),
            "or_read_bits": (C.c_uint64, [u8p, C.c_uint64, C.c_int]),
            "or_write_bits": (None, [u8p, C.c_uint64, C.c_int, C.c_uint64]),
            "or_factors_init": (C.c_int, [FP, C.c_int64, C.c_int64, fp, fp]),
            "or_factors_free": (None, [FP]),
            "or_imp": (C.c_double, [FP, SP, C.c_int64, C.c_int64]),
            "or_ladder": (C.c_int, [SP, C.c_double]),
            "or_rung_rows": (None, [FP, SP, C.c_int64, C.c_int64, C.c_int64, u8p]),
            "or_tied_blocks": (C.c_int64, [FP, SP]),
            "or_row_bit_offset": (C.c_uint64, [FP, SP, C.c_int64, C.c_int64]),
            "or_decode_rows": (C.c_int, [FP, SP, C.c_int64, u8p, C.c_uint64, u32p, C.c_int,
                                         i32p, u16p, C.c_int64, C.c_int64, fp]),
            "or_gemv_f64": (None, [C.c_int64, C.c_int64, fp, C.c_int, u16p, dp]),
            "or_decode_gemv_threads": (C.c_int, [FP, SP, C.c_int64, u8p, C.c_uint64, u32p,
                                                 C.c_int, u16p, C.c_int64, C.c_int64, dp, C.c_int]),
            "or_splitmix64_at": (C.c_uint64, [C.c_uint64, C.c_uint64]),
            "or_synth_fields": (None, [C.c_uint64, C.c_uint64, C.c_int, C.c_int, u32p, ip, ip]),
            "or_synth_pack": (C.c_uint64, [FP, SP, C.c_int64, C.c_uint64, u8p]),
            "or_synth_rows": (None, [FP, SP, C.c_int64, C.c_uint64, u32p, C.c_int, i32p, u16p,
                                     C.c_int64, C.c_int64, fp]),
            "or_synth_gemv_threads": (C.c_int, [FP, SP, C.c_int64, C.c_uint64, u32p, C.c_int, u16p,
                                                C.c_int64, C.c_int64, dp, dp, C.c_int]),
            "or_synth_pack_rows": (C.c_uint64, [FP, SP, C.c_int64, C.c_uint64, C.c_int64,
                                                C.c_int64, u8p]),
            "or_hull": (C.c_int, [C.c_int, ip, ip, dp, ip]),
            "or_allocate": (C.c_int, [C.c_int, C.POINTER(FP), C.c_int, ip, ip, dp, C.c_double,
                                      C.c_double, dp, ip, dp, i64p, u64p]),
            "or_encode_block": (C.c_double, [C.c_int, C.c_int, C.c_uint32, dp, u32p, ip, ip]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


# ----------------------------------------------------------------- codec

def block_bits(S: int, k: int) -> int:
    return lib().or_block_bits(S, k)


def lfsr_bits(S: int, taps: int, seed: int, n: int) -> np.ndarray:
    o = np.zeros(n, np.uint8)
    lib().or_lfsr_bits(S, taps, seed, n, _p(o, C.c_uint8))
    return o


def lfsr_period(S: int, taps: int) -> int:
    return lib().or_lfsr_period(S, taps)


def find_taps(S: int) -> int:
    return lib().or_find_taps(S)


_TAPS_CACHE: dict[int, int] = {}


def taps_table() -> np.ndarray:
    """uint32[17]: entry S is the tap mask the oracle's search picks for width S."""
    out = np.zeros(17, np.uint32)
    for S in range(8, 17):
        if S not in _TAPS_CACHE:
            _TAPS_CACHE[S] = find_taps(S)
        out[S] = _TAPS_CACHE[S]
    return out


def reconstruct_block(S, k, taps, seed, E, t) -> np.ndarray:
    tt = np.asarray(list(t) + [0] * (6 - len(t)), np.int32).astype(np.intc)
    w = np.zeros(8, np.float32)
    lib().or_reconstruct_block(S, k, taps, seed, E, _p(tt, C.c_int), _p(w, C.c_float))
    return w


def read_bits(stream: np.ndarray, pos: int, n: int) -> int:
    return lib().or_read_bits(_p(stream, C.c_uint8), pos, n)


def write_bits(stream: np.ndarray, pos: int, n: int, value: int) -> None:
    lib().or_write_bits(_p(stream, C.c_uint8), pos, n, value)


def splitmix64_at(key: int, i: int) -> int:
    return lib().or_splitmix64_at(key, i)


def synth_fields(key, b, S, k):
    seed = C.c_uint32()
    E = C.c_int()
    t = (C.c_int * 6)()
    lib().or_synth_fields(key, b, S, k, C.byref(seed), C.byref(E), t)
    return seed.value, E.value, list(t)[:k]


def encode_block(S, k, taps, w):
    w = np.ascontiguousarray(w, np.float64)
    seed, E = C.c_uint32(), C.c_int()
    t = (C.c_int * 6)()
    err = lib().or_encode_block(S, k, taps, _p(w, C.c_double), C.byref(seed), C.byref(E), t)
    return seed.value, E.value, list(t)[:k], err


# -------------------------------------------------------------- schedule

class Sched:
    """A decoder schedule (hull rungs, thresholds, tie threshold, floor)."""

    def __init__(self, rungs, theta, j_tie, q):
        self.S = np.asarray([r[0] for r in rungs], np.intc)
        self.k = np.asarray([r[1] for r in rungs], np.intc)
        self.theta = np.ascontiguousarray(theta, np.float64)
        self.j_tie = int(j_tie)
        self.q = float(q)
        assert len(self.theta) == len(self.S) - 1
        self.c = Schedule(len(self.S), _p(self.S, C.c_int), _p(self.k, C.c_int),
                          _p(self.theta, C.c_double), self.j_tie, self.q)

    @property
    def rungs(self):
        return [(int(s), int(k)) for s, k in zip(self.S, self.k)]


class Tensor:
    """Per-tensor factors of Eq. imp (perm, unit-mean abar and rho)."""

    def __init__(self, R, Cc, a, rho=None):
        self.a = np.ascontiguousarray(a, np.float32)
        self.rho_in = None if rho is None else np.ascontiguousarray(rho, np.float32)
        self.f = Factors()
        rc = lib().or_factors_init(C.byref(self.f), R, Cc, _p(self.a, C.c_float),
                                   None if self.rho_in is None else _p(self.rho_in, C.c_float))
        if rc != 0:
            raise ValueError("or_factors_init failed")
        self.R, self.C = R, Cc

    def __del__(self):
        try:
            lib().or_factors_free(C.byref(self.f))
        except Exception:
            pass

    @property
    def perm(self):
        return np.ctypeslib.as_array(self.f.perm, shape=(self.C,)).copy()

    @property
    def abar(self):
        return np.ctypeslib.as_array(self.f.abar, shape=(self.C // 8,)).copy()

    @property
    def rho(self):
        return np.ctypeslib.as_array(self.f.rho, shape=(self.R,)).copy()

    def imp(self, s: Sched, r: int, c: int) -> float:
        return lib().or_imp(C.byref(self.f), C.byref(s.c), r, c)

    def rung_rows(self, s: Sched, T: int, r0: int = 0, nrows: int | None = None):
        nrows = self.R - r0 if nrows is None else nrows
        out = np.zeros((nrows, self.C // 8), np.uint8)
        lib().or_rung_rows(C.byref(self.f), C.byref(s.c), T, r0, nrows, _p(out, C.c_uint8))
        return out

    def tied_blocks(self, s: Sched) -> int:
        return lib().or_tied_blocks(C.byref(self.f), C.byref(s.c))

    def row_bit_offset(self, s: Sched, T: int, r: int) -> int:
        return lib().or_row_bit_offset(C.byref(self.f), C.byref(s.c), T, r)

    def decode_rows(self, s, T, stream, stream_bits, r0=0, nrows=None,
                    outlier_cols=None, outlier_vals=None):
        nrows = self.R - r0 if nrows is None else nrows
        W = np.zeros((nrows, self.C), np.float32)
        cols, vals, n_out = _outliers(outlier_cols, outlier_vals)
        taps = taps_table()
        rc = lib().or_decode_rows(C.byref(self.f), C.byref(s.c), T, _p(stream, C.c_uint8),
                                  stream_bits, _p(taps, C.c_uint32), n_out,
                                  _p(cols, C.c_int32), _p(vals, C.c_uint16), r0, nrows,
                                  _p(W, C.c_float))
        if rc != 0:
            raise ValueError("stream too short")
        return W

    def synth_pack(self, s, T, key):
        bits = self.row_bit_offset(s, T, self.R)
        nbytes = (bits + 7) // 8
        stream = np.zeros(((nbytes + 15) // 16) * 16 + 16, np.uint8)
        got = lib().or_synth_pack(C.byref(self.f), C.byref(s.c), T, key, _p(stream, C.c_uint8))
        assert got == bits
        return stream, bits

    def synth_rows(self, s, T, key, r0=0, nrows=None, outlier_cols=None, outlier_vals=None):
        nrows = self.R - r0 if nrows is None else nrows
        W = np.zeros((nrows, self.C), np.float32)
        cols, vals, n_out = _outliers(outlier_cols, outlier_vals)
        taps = taps_table()
        lib().or_synth_rows(C.byref(self.f), C.byref(s.c), T, key, _p(taps, C.c_uint32), n_out,
                            _p(cols, C.c_int32), _p(vals, C.c_uint16), r0, nrows,
                            _p(W, C.c_float))
        return W

    def synth_gemv(self, s, T, key, x_bf16, r0=0, nrows=None, nthreads=None):
        """fp64 y = W_hat x and sum |W_hat| |x| for rows [r0, r0+nrows) of the
        synthetic tensor (nb x nrows arrays)."""
        nrows = self.R - r0 if nrows is None else nrows
        x = np.ascontiguousarray(x_bf16, np.uint16)
        nb = x.size // self.C
        y = np.zeros((nb, self.R), np.float64)
        ya = np.zeros((nb, self.R), np.float64)
        nthreads = nthreads or max(1, min(os.cpu_count() or 1, 64))
        taps = taps_table()
        lib().or_synth_gemv_threads(C.byref(self.f), C.byref(s.c), T, key, _p(taps, C.c_uint32), nb,
                                    _p(x, C.c_uint16), r0, nrows, _p(y, C.c_double),
                                    _p(ya, C.c_double), nthreads)
        return y[:, r0:r0 + nrows], ya[:, r0:r0 + nrows]

    def synth_pack_rows(self, s, T, key, r0, nrows, nbits_hint):
        out = np.zeros((nbits_hint + 7) // 8 + 16, np.uint8)
        bits = lib().or_synth_pack_rows(C.byref(self.f), C.byref(s.c), T, key, r0, nrows,
                                        _p(out, C.c_uint8))
        return out, bits

    def decode_gemv_threads(self, s, T, stream, stream_bits, x_bf16, nthreads, r0=0, nrows=None):
        nrows = self.R - r0 if nrows is None else nrows
        x = np.ascontiguousarray(x_bf16, np.uint16)
        nb = x.size // self.C
        y = np.zeros((nb, self.R), np.float64)
        taps = taps_table()
        n = lib().or_decode_gemv_threads(C.byref(self.f), C.byref(s.c), T, _p(stream, C.c_uint8),
                                         stream_bits, _p(taps, C.c_uint32), nb,
                                         _p(x, C.c_uint16), r0, nrows, _p(y, C.c_double), nthreads)
        if n < 0:
            raise ValueError("stream too short")
        return y, n


def _outliers(cols, vals):
    if cols is None or len(cols) == 0:
        return np.zeros(1, np.int32), np.zeros(1, np.uint16), 0
    cols = np.ascontiguousarray(cols, np.int32)
    vals = np.ascontiguousarray(vals, np.uint16)
    return cols, vals, len(cols)


def gemv_f64(W: np.ndarray, x_bf16: np.ndarray) -> np.ndarray:
    W = np.ascontiguousarray(W, np.float32)
    x = np.ascontiguousarray(x_bf16, np.uint16)
    nrows, Cc = W.shape
    nb = x.size // Cc
    y = np.zeros((nb, nrows), np.float64)
    lib().or_gemv_f64(nrows, Cc, _p(W, C.c_float), nb, _p(x, C.c_uint16), _p(y, C.c_double))
    return y


def hull(points):
    """points: list of (S, k, e).  Returns the hull as a list of indices."""
    n = len(points)
    S = np.asarray([p[0] for p in points], np.intc)
    k = np.asarray([p[1] for p in points], np.intc)
    e = np.asarray([p[2] for p in points], np.float64)
    idx = np.zeros(n, np.intc)
    J = lib().or_hull(n, _p(S, C.c_int), _p(k, C.c_int), _p(e, C.c_double), _p(idx, C.c_int))
    return [int(i) for i in idx[:J]]


def allocate(tensors, rungs, slopes, rbar, floor_f=0.06):
    """Alg. 1 allocation over a set of Tensor objects sharing one budget."""
    nt, J = len(tensors), len(rungs)
    arr = (C.POINTER(Factors) * nt)(*[C.pointer(t.f) for t in tensors])
    S = np.asarray([r[0] for r in rungs], np.intc)
    k = np.asarray([r[1] for r in rungs], np.intc)
    sl = np.ascontiguousarray(slopes, np.float64)
    theta = np.zeros(max(J - 1, 1), np.float64)
    j_tie, q = C.c_int(), C.c_double()
    T = np.zeros(nt, np.int64)
    bits = np.zeros(nt, np.uint64)
    rc = lib().or_allocate(nt, arr, J, _p(S, C.c_int), _p(k, C.c_int), _p(sl, C.c_double),
                           rbar, floor_f, _p(theta, C.c_double), C.byref(j_tie), C.byref(q),
                           _p(T, C.c_int64), _p(bits, C.c_uint64))
    if rc != 0:
        raise RuntimeError(f"or_allocate failed ({rc})")
    return Sched(rungs, theta[:J - 1], j_tie.value, q.value), T, bits


def hull_rungs(damage: dict, rbar: float, band=(1.0, 1.5)):
    """Hull of a damage table (Sec. 3.4) confined to the rate band of App. A.5
    (rungs within band[0] bits/weight below and band[1] above rbar).

    Returns (rungs, e, slopes) with slopes s_j = (e_j - e_{j+1}) / (r_{j+1} - r_j)."""
    pts = [(S, k, e) for (S, k), e in sorted(damage.items())]
    idx = hull(pts)
    rungs = [(pts[i][0], pts[i][1]) for i in idx]
    es = [pts[i][2] for i in idx]
    keep = [j for j, (S, k) in enumerate(rungs)
            if rbar - band[0] <= block_bits(S, k) / 8.0 <= rbar + band[1]]
    rungs = [rungs[j] for j in keep]
    es = [es[j] for j in keep]
    rates = [block_bits(S, k) / 8.0 for S, k in rungs]
    slopes = [(es[j] - es[j + 1]) / (rates[j + 1] - rates[j]) for j in range(len(rungs) - 1)]
    return rungs, es, slopes


# ------------------------------------------------------------ container file
# The oracle's own reader and writer of the container layout (the model file
# holding the Sec. 3.6 table and, per tensor, the inputs of Alg. 2 and the
# stream): little-endian fields in this order, then a 64-bit FNV-1a hash of
# all preceding bytes.  Written independently of the library's C++ version.

import struct as _st

_MAGIC = b"SEEDQ\x00v1"


def _fnv1a(data: bytes) -> int:
    h = 0xCBF29CE484222325
    for b in data:
        h ^= b
        h = (h * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h


def write_container(path, rungs, theta, j_tie, q, tensors) -> None:
    out = bytearray(_MAGIC)
    out += _st.pack("<II", 1, len(rungs))
    for S, k in rungs:
        out += _st.pack("<ii", S, k)
    for th in theta:
        out += _st.pack("<d", th)
    out += _st.pack("<id", j_tie, q)
    taps = taps_table()
    for S in range(8, 17):
        out += _st.pack("<I", int(taps[S]))
    out += _st.pack("<I", len(tensors))
    for t in tensors:
        name = t.get("name", "").encode()
        out += _st.pack("<I", len(name)) + name
        out += _st.pack("<qq", t["rows"], t["cols"])
        out += np.ascontiguousarray(t["a"], "<f4").tobytes()
        if t.get("rho") is None:
            out += _st.pack("<I", 0)
        else:
            out += _st.pack("<I", 1) + np.ascontiguousarray(t["rho"], "<f4").tobytes()
        out += _st.pack("<q", t["tie_count"])
        cols = np.ascontiguousarray(t.get("outlier_cols", np.zeros(0)), "<i4")
        out += _st.pack("<i", cols.size) + cols.tobytes()
        out += np.ascontiguousarray(t.get("outlier_vals", np.zeros(0)), "<u2").tobytes()
        nbytes = (int(t["stream_bits"]) + 7) // 8
        out += _st.pack("<QQ", int(t["stream_bits"]), nbytes)
        out += np.ascontiguousarray(t["stream"], np.uint8)[:nbytes].tobytes()
    out += _st.pack("<Q", _fnv1a(bytes(out)))
    with open(path, "wb") as f:
        f.write(bytes(out))


def read_container(path) -> dict:
    data = open(path, "rb").read()
    if data[:8] != _MAGIC:
        raise ValueError("not a container")
    if _st.unpack("<Q", data[-8:])[0] != _fnv1a(data[:-8]):
        raise ValueError("hash mismatch")
    at = 8

    def take(fmt):
        nonlocal at
        v = _st.unpack_from(fmt, data, at)
        at += _st.calcsize(fmt)
        return v

    version, J = take("<II")
    if version != 1:
        raise ValueError("version")
    rungs = [take("<ii") for _ in range(J)]
    theta = [take("<d")[0] for _ in range(J - 1)]
    j_tie, q = take("<id")
    taps = [take("<I")[0] for _ in range(9)]
    (nt,) = take("<I")
    tensors = []
    for _ in range(nt):
        (nl,) = take("<I")
        name = data[at:at + nl].decode()
        at += nl
        R, Cc = take("<qq")
        a = np.frombuffer(data, "<f4", Cc, at).copy()
        at += 4 * Cc
        (has_rho,) = take("<I")
        rho = None
        if has_rho:
            rho = np.frombuffer(data, "<f4", R, at).copy()
            at += 4 * R
        (T,) = take("<q")
        (no,) = take("<i")
        cols = np.frombuffer(data, "<i4", no, at).copy()
        at += 4 * no
        vals = np.frombuffer(data, "<u2", R * no, at).copy().reshape(R, no)
        at += 2 * R * no
        bits, nbytes = take("<QQ")
        stream = np.frombuffer(data, np.uint8, nbytes, at).copy()
        at += nbytes
        tensors.append({"name": name, "rows": R, "cols": Cc, "a": a, "rho": rho, "tie_count": T,
                        "outlier_cols": cols, "outlier_vals": vals, "stream": stream,
                        "stream_bits": bits})
    if at != len(data) - 8:
        raise ValueError("trailing bytes")
    return {"rungs": [tuple(r) for r in rungs], "theta": theta, "j_tie": j_tie, "q": q,
            "taps": taps, "tensors": tensors}

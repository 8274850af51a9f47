"""Seeded synthetic workloads shaped like the paper's LLM layers.

This module only draws inputs: layer shapes, the importance factors a and rho,
activation vectors x, the keys from which each tensor's synthetic payload is
derived, and the published damage tables.  It holds none of the method's
arithmetic (no hull, no schedule, no codec), so the oracle and the CUDA
library can both consume what it produces without sharing code.

Determinism across machines: every random number comes from splitmix64
(Steele, Lea, Flood 2014) evaluated with exact uint64 arithmetic; normals are
Irwin-Hall sums of twelve 24-bit uniforms (exact in fp64) and exponentials are
(1 + y/1024)^1024 by ten IEEE squarings, so the same bits come out on x86 and
Arm without relying on libm.
"""
from __future__ import annotations

import dataclasses
import hashlib
from functools import lru_cache

import numpy as np

_M64 = (1 << 64) - 1
_GAMMA = 0x9E3779B97F4A7C15


def splitmix64_at(key: int, i):
    """Output number i (0-based) of splitmix64 started at state `key`.

    Works on a Python int or a numpy uint64 array of indices."""
    if isinstance(i, (int, np.integer)):
        z = (key + (int(i) + 1) * _GAMMA) & _M64
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _M64
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _M64
        return z ^ (z >> 31)
    idx = np.asarray(i, np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(key) + (idx + np.uint64(1)) * np.uint64(_GAMMA)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
    return z ^ (z >> np.uint64(31))


def derive_key(seed: int, *parts: int) -> int:
    k = seed & _M64
    for p in parts:
        k = splitmix64_at(k, p)
    return k


def uniform24(key: int, n: int, offset: int = 0) -> np.ndarray:
    """n uniforms on [0, 1) with 24 random bits each (exact in fp64)."""
    h = splitmix64_at(key, np.arange(offset, offset + n, dtype=np.uint64))
    return (h >> np.uint64(40)).astype(np.float64) * (2.0 ** -24)


def normal(key: int, n: int) -> np.ndarray:
    """Approximately N(0,1): Irwin-Hall sum of 12 uniforms minus 6."""
    u = uniform24(key, 12 * n).reshape(n, 12)
    z = np.zeros(n, np.float64)
    for i in range(12):
        z = z + u[:, i]
    return z - 6.0


def exp_det(y: np.ndarray) -> np.ndarray:
    """exp(y) as (1 + y/1024)^1024: only IEEE multiply/add, so bit-reproducible."""
    z = 1.0 + np.asarray(y, np.float64) / 1024.0
    for _ in range(10):
        z = z * z
    return z


def to_bf16_bits(v: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even from float32 to bfloat16 bit patterns (uint16)."""
    f = np.ascontiguousarray(v, np.float32).view(np.uint32).astype(np.uint64)
    r = (f + np.uint64(0x7FFF) + ((f >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, np.uint32) << np.uint32(16)).view(np.float32)


def to_f16_bits(v: np.ndarray) -> np.ndarray:
    return np.ascontiguousarray(v, np.float16).view(np.uint16)


# ---------------------------------------------------------------------------
# Damage tables: the rung-grid table of App. B.3, excess loss e(g) in nats per
# token over FP16 on WikiText-2 test, indexed by rung (S, k).
DAMAGE_LLAMA2_7B = {
    (8, 3): 1.8746, (10, 3): 0.5852, (12, 3): 0.2249, (14, 3): 0.1182,
    (16, 3): 0.0669, (10, 4): 0.1445, (12, 4): 0.0744, (14, 4): 0.0441,
    (16, 4): 0.0340, (12, 5): 0.0367, (14, 5): 0.0239, (16, 5): 0.0131,
    (16, 6): 0.0064,
}
# Llama-3-8B column; (8,3) was measured but excluded from its allocation.
DAMAGE_LLAMA3_8B = {
    (10, 3): 0.7014, (12, 3): 0.3892, (14, 3): 0.2445, (16, 3): 0.1556,
    (14, 4): 0.1173, (16, 5): 0.0446,
}


def damage_synthetic_k2() -> dict:
    """Sub-4-bit grid: the Llama-2-7B column plus e(S,2) := 2 e(S,3) for even S.

    The paper prints no k = 2 damages; App. B.3 reports that each coefficient
    added beyond k = 3 roughly halves the excess loss, and this extends that
    one step down.  Synthetic, used only for the 3.0 bits/weight workloads."""
    d = dict(DAMAGE_LLAMA2_7B)
    for S in (8, 10, 12, 14, 16):
        d[(S, 2)] = 2.0 * DAMAGE_LLAMA2_7B[(S, 3)]
    return d


DAMAGE_TABLES = {
    "llama2_7b": lambda: dict(DAMAGE_LLAMA2_7B),
    "llama3_8b": lambda: dict(DAMAGE_LLAMA3_8B),
    "synthetic_k2": damage_synthetic_k2,
}


# ---------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class TensorSpec:
    name: str
    R: int            # output rows
    C: int            # input channels
    a_group: str      # tensors with the same a_group share one a vector
    has_rho: bool     # rows carry an output-side factor rho


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    seed: int
    rbar: float
    damage: str
    tensors: tuple
    batches: tuple
    description: str

    @property
    def weights(self) -> int:
        return sum(t.R * t.C for t in self.tensors)


def _llama_layer(prefix, d, kv, ff, rho_all=False):
    return [
        TensorSpec(f"{prefix}q", d, d, f"{prefix}attn_in", rho_all),
        TensorSpec(f"{prefix}k", kv, d, f"{prefix}attn_in", rho_all),
        TensorSpec(f"{prefix}v", kv, d, f"{prefix}attn_in", rho_all),
        TensorSpec(f"{prefix}o", d, d, f"{prefix}o_in", True),
        TensorSpec(f"{prefix}gate", ff, d, f"{prefix}mlp_in", rho_all),
        TensorSpec(f"{prefix}up", ff, d, f"{prefix}mlp_in", rho_all),
        TensorSpec(f"{prefix}down", d, ff, f"{prefix}down_in", True),
    ]


def _build():
    w = {}
    w["c0"] = Workload("c0", 0, 4.0, "llama2_7b",
                       (TensorSpec("w", 1024, 1024, "w_in", False),), (1,),
                       "single 1024x1024 linear layer, 4.0 bits/weight, batch 1")
    w["c1"] = Workload("c1", 1, 4.0, "llama2_7b", tuple(_llama_layer("", 4096, 4096, 11008)), (1,),
                       "Llama-2-7B-shaped layer set (q,k,v,o 4096x4096; gate,up 11008x4096; "
                       "down 4096x11008), 4.0 bits/weight, batch 1")
    w["c2"] = Workload("c2", 2, 3.0, "synthetic_k2",
                       tuple(_llama_layer("", 4096, 4096, 11008, rho_all=True)), (1, 2, 4, 8),
                       "Llama-2-7B-shaped layer set, 3.0 bits/weight, rho on every row "
                       "(rung map varies across rows), batch 1/2/4/8")
    t3 = []
    for L in range(32):
        t3 += _llama_layer(f"l{L}.", 4096, 1024, 14336)
    t3.append(TensorSpec("lm_head", 128256, 4096, "lm_head_in", False))
    w["c3"] = Workload("c3", 3, 4.0, "llama3_8b", tuple(t3), (1,),
                       "Llama-3-8B-shaped 32 layers + lm_head, 4.0 bits/weight, batch 1")
    t4 = []
    for L in range(80):
        t4 += _llama_layer(f"l{L}.", 8192, 1024, 28672)
    w["c4"] = Workload("c4", 4, 4.0, "llama2_7b", tuple(t4), (1, 4, 16),
                       "Llama-2-70B-shaped 80 layers, 4.0 bits/weight, batch 1/4/16")
    w["c4_3"] = Workload("c4_3", 4, 3.0, "synthetic_k2", tuple(t4), (1, 4, 16),
                         "Llama-2-70B-shaped 80 layers, 3.0 bits/weight, batch 1/4/16")
    return w


WORKLOADS = _build()

# Domain separators for derive_key.
_D_A, _D_RHO, _D_OUTCH, _D_PAYLOAD, _D_X, _D_OUTVAL = 1, 2, 3, 7, 11, 13


@lru_cache(maxsize=None)
def _group_a(seed: int, group: str, C: int) -> np.ndarray:
    gid = int.from_bytes(hashlib.sha256(group.encode()).digest()[:8], "little")
    key = derive_key(seed, _D_A, gid)
    gamma = exp_det(0.5 * normal(key, C))
    a = gamma * gamma
    # Four channels with a_j = 100x the tensor mean (the activation-outlier
    # scale of the outlier-column rule, Sec. 3.5).
    mean = a.sum() / C
    ch = (splitmix64_at(derive_key(key, _D_OUTCH), np.arange(4, dtype=np.uint64))
          % np.uint64(C)).astype(np.int64)
    a[ch] = 100.0 * mean
    return a.astype(np.float32)


def importance(w: Workload, i: int):
    """(a, rho) for tensor i: float32 arrays, rho None when the rows carry none."""
    t = w.tensors[i]
    a = _group_a(w.seed, t.a_group, t.C)
    rho = None
    if t.has_rho:
        key = derive_key(w.seed, _D_RHO, i)
        rho = exp_det(0.5 * normal(key, t.R)).astype(np.float32)
    return a, rho


def payload_key(w: Workload, i: int) -> int:
    """Key of the counter-based generator for the block fields of tensor i."""
    return derive_key(w.seed, _D_PAYLOAD, i)


def x_bf16(w: Workload, i: int, nb: int = 1) -> np.ndarray:
    """nb activation columns for tensor i, x ~ N(0,1) rounded to bf16 (nb x C)."""
    C = w.tensors[i].C
    out = np.zeros((nb, C), np.uint16)
    for b in range(nb):
        out[b] = to_bf16_bits(normal(derive_key(w.seed, _D_X, i, b), C).astype(np.float32))
    return out


def outlier_case(w: Workload, i: int, n_out: int = 4):
    """n_out distinct outlier columns of tensor i and their fp16 values (R x n_out)."""
    t = w.tensors[i]
    key = derive_key(w.seed, _D_OUTVAL, i)
    cols = []
    j = 0
    while len(cols) < n_out:
        c = int(splitmix64_at(key, j) % t.C)
        j += 1
        if c not in cols:
            cols.append(c)
    vals = 8.0 * normal(derive_key(key, 1), t.R * n_out)
    return np.asarray(cols, np.int32), to_f16_bits(vals.astype(np.float32)).reshape(t.R, n_out)


def a_rho_checksum(w: Workload) -> str:
    """Digest of every tensor's (a, rho) bits, stored beside the schedule so a
    machine that draws different inputs fails loudly instead of silently."""
    h = hashlib.sha256()
    for i in range(len(w.tensors)):
        a, rho = importance(w, i)
        h.update(a.tobytes())
        if rho is not None:
            h.update(rho.tobytes())
    return h.hexdigest()[:32]


# ---------------------------------------------------------------------------
# Synthetic FP16 checkpoints for the data-free importance (Sec. 3.2) and the
# outlier-column rules (Sec. 3.5): Llama-shaped decoders with random weights,
# RMSNorm gains near one with a few massive channels, and planted super
# weights.  Every value is integer-exact before its single rounding to FP16,
# so numpy and a device kernel implementing the same counter-based generator
# produce the same bits.

_D_W, _D_GAIN, _D_MASSIVE, _D_SUPER = 17, 19, 23, 29
MODEL_KINDS = ("q", "k", "v", "o", "gate", "up", "down")


@dataclasses.dataclass(frozen=True)
class ModelSpec:
    name: str
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    d_ff: int
    vocab: int
    seed: int
    description: str

    @property
    def q_dim(self) -> int:
        return self.n_heads * self.head_dim

    @property
    def kv_dim(self) -> int:
        return self.n_kv_heads * self.head_dim

    def shape(self, kind: str):
        d, f = self.d_model, self.d_ff
        return {"q": (self.q_dim, d), "k": (self.kv_dim, d), "v": (self.kv_dim, d),
                "o": (d, self.q_dim), "gate": (f, d), "up": (f, d), "down": (d, f),
                "lm_head": (self.vocab, d)}[kind]

    def tensor_names(self):
        return [f"l{l}.{k}" for l in range(self.n_layers) for k in MODEL_KINDS] + ["lm_head"]

    @property
    def weights(self) -> int:
        per = sum(self.shape(k)[0] * self.shape(k)[1] for k in MODEL_KINDS)
        return self.n_layers * per + self.vocab * self.d_model


MODELS = {
    "tiny": ModelSpec("tiny", 2, 256, 4, 2, 64, 640, 300, 31,
                      "2 layers, d 256, 4 query / 2 key-value heads of 64, d_ff 640, vocab 300"),
    "tiny_mha": ModelSpec("tiny_mha", 3, 256, 4, 4, 64, 512, 272, 37,
                          "3 layers, d 256, 4 heads of 64 (no sharing), d_ff 512, vocab 272"),
    "tiny_odd": ModelSpec("tiny_odd", 2, 160, 5, 1, 32, 96, 77, 47,
                          "2 layers, d 160, 5 query heads of 32 sharing 1 key-value head, "
                          "d_ff 96, vocab 77 (row counts not multiples of 64)"),
    "llama2_7b": ModelSpec("llama2_7b", 32, 4096, 32, 32, 128, 11008, 32000, 41,
                           "Llama-2-7B-shaped: 32 layers, d 4096, 32 heads of 128, d_ff 11008, "
                           "vocab 32000, FP16"),
    "llama3_8b": ModelSpec("llama3_8b", 32, 4096, 32, 8, 128, 14336, 128256, 43,
                           "Llama-3-8B-shaped: 32 layers, d 4096, 32 query / 8 key-value heads, "
                           "d_ff 14336, vocab 128256, FP16"),
}

# Weights: z * m * 2^-e rounded once to FP16, z the centred sum of the four
# 16-bit fields of one splitmix64 output (|z| < 2^17, sd ~37838), m * 2^-e =
# 9 * 2^-24 (sd ~0.0203); exact in fp32 before the rounding.
W_SCALE_M, W_SCALE_E = 9, 24
GAIN_SCALE_E = 19           # gains 1 + z * 2^-19 (sd ~0.072), exact in fp32
MASSIVE_GAIN = 24.0         # gain of the massive channels (layers >= 1)
N_MASSIVE = 1
SUPER_VALUES = (40.0, -36.0)  # planted super weights (~2000 sd), exact in FP16


def _kind_index(kind: str) -> int:
    return MODEL_KINDS.index(kind) if kind in MODEL_KINDS else 7


def weight_key(spec: ModelSpec, layer, kind: str) -> int:
    return derive_key(spec.seed, _D_W, 0xFFFF if layer is None else layer, _kind_index(kind))


def irwin_hall4(key: int, start: int, n: int) -> np.ndarray:
    """Centred sum of the four 16-bit fields of splitmix64 outputs start..start+n-1."""
    h = splitmix64_at(key, np.arange(start, start + n, dtype=np.uint64))
    m = np.uint64(0xFFFF)
    z = (h & m) + ((h >> np.uint64(16)) & m) + ((h >> np.uint64(32)) & m) + (h >> np.uint64(48))
    return z.astype(np.int64) - 131070


def _fp16_of_exact(v32: np.ndarray) -> np.ndarray:
    return np.asarray(v32, np.float32).astype(np.float16).view(np.uint16)


def synth_weight_rows(spec: ModelSpec, layer, kind: str, r0: int, nrows: int) -> np.ndarray:
    """Rows [r0, r0 + nrows) of a weight matrix as FP16 bits (nrows x C),
    planted super weights included."""
    R, C = spec.shape(kind)
    z = irwin_hall4(weight_key(spec, layer, kind), r0 * C, nrows * C)
    v = z.astype(np.float32) * np.float32(W_SCALE_M * 2.0 ** -W_SCALE_E)
    out = _fp16_of_exact(v).reshape(nrows, C)
    for (l, k, r, c, bits) in super_weights(spec):
        if l == layer and k == kind and r0 <= r < r0 + nrows:
            out[r - r0, c] = bits
    return out


def super_weights(spec: ModelSpec):
    """Planted super weights: (layer, kind, row, column, FP16 bits) in the
    down projection of layer 1 (layer 0 for one-layer models)."""
    l = min(1, spec.n_layers - 1)
    R, C = spec.shape("down")
    key = derive_key(spec.seed, _D_SUPER)
    out = []
    for i, val in enumerate(SUPER_VALUES):
        r = int(splitmix64_at(key, 2 * i) % np.uint64(R))
        c = int(splitmix64_at(key, 2 * i + 1) % np.uint64(C))
        out.append((l, "down", r, c, int(_fp16_of_exact(np.float32(val)))))
    return out


def massive_channels(spec: ModelSpec) -> np.ndarray:
    key = derive_key(spec.seed, _D_MASSIVE)
    return (splitmix64_at(key, np.arange(N_MASSIVE, dtype=np.uint64))
            % np.uint64(spec.d_model)).astype(np.int64)


def synth_gain(spec: ModelSpec, layer, which: str) -> np.ndarray:
    """RMSNorm gain as FP16 bits: which = "attn" / "mlp" (layer's input norms)
    or "final" (layer None)."""
    wi = {"attn": 0, "mlp": 1, "final": 2}[which]
    key = derive_key(spec.seed, _D_GAIN, 0xFFFF if layer is None else layer, wi)
    z = irwin_hall4(key, 0, spec.d_model)
    v = np.float32(1.0) + z.astype(np.float32) * np.float32(2.0 ** -GAIN_SCALE_E)
    if which != "final" and layer is not None and layer >= 1:
        v[massive_channels(spec)] = MASSIVE_GAIN
    return _fp16_of_exact(v)


class SynthModel:
    """Host (numpy) view of a synthetic checkpoint; arrays are drawn on demand."""

    def __init__(self, spec: ModelSpec):
        self.spec = spec

    def weight(self, layer, kind: str) -> np.ndarray:
        R, _ = self.spec.shape(kind)
        return synth_weight_rows(self.spec, layer, kind, 0, R)

    def lm_head(self) -> np.ndarray:
        return self.weight(None, "lm_head")

    def gain(self, layer, which: str) -> np.ndarray:
        return synth_gain(self.spec, layer, which)

    def tensor(self, i: int) -> np.ndarray:
        """Tensor i of the model order (per layer q, k, v, o, gate, up, down; the head)."""
        n = len(MODEL_KINDS)
        if i == self.spec.n_layers * n:
            return self.lm_head()
        return self.weight(i // n, MODEL_KINDS[i % n])

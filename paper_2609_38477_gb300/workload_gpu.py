"""Bring a synthetic workload onto the GPU through the C ABI.

For each tensor: prepare the decoder plan (seedq_layer_prepare) from the
workload's importance factors and a schedule table, allocate the stream buffer,
fill it with the synthetic payload on the device (seedq_synth_stream) and bind
it.  Torch only allocates device memory here.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import torch

from . import seedq as Q
from . import workloads as W


@dataclasses.dataclass
class GpuTensor:
    index: int
    spec: W.TensorSpec
    layer: Q.Layer
    stream: torch.Tensor
    bits: int
    nbytes: int


def prepare_tensor(w: W.Workload, i: int, sched: dict, max_batch: int = 1,
                   outliers=None, stream_bytes=None, synth: bool = True) -> GpuTensor:
    t = w.tensors[i]
    a, rho = W.importance(w, i)
    ocols, ovals = (None, None) if outliers is None else outliers
    ovals_dev = None
    if ovals is not None:
        ovals_dev = torch.from_numpy(np.ascontiguousarray(ovals).view(np.int16)).cuda()
    layer = Q.Layer(t.R, t.C, a, rho, [tuple(r) for r in sched["rungs"]], sched["theta"],
                    sched["j_tie"], sched["q"], sched["tie_count"][i], ocols, ovals_dev,
                    max_batch=max_batch)
    layer._ovals_keep = ovals_dev
    bits = layer.stream_bits
    nbytes = Q.stream_bytes_required(bits)
    buf = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    if synth:
        layer.synth_stream(W.payload_key(w, i), buf, nbytes)
    return GpuTensor(i, t, layer, buf, bits, nbytes)


def bind(gt: GpuTensor):
    gt.layer.bind_stream(gt.stream, gt.bits, gt.nbytes)
    return gt


def prepare_workload(w: W.Workload, sched: dict, indices=None, max_batch: int = 1):
    idx = range(len(w.tensors)) if indices is None else indices
    out = []
    for i in idx:
        gt = prepare_tensor(w, i, sched, max_batch=max_batch)
        bind(gt)
        out.append(gt)
    torch.cuda.synchronize()
    return out


def x_device(w: W.Workload, i: int, nb: int = 1) -> torch.Tensor:
    """Activation columns of tensor i as a device int16 tensor of bf16 bits (nb x C)."""
    return torch.from_numpy(W.x_bf16(w, i, nb).view(np.int16)).cuda()


# ------------------------------------------------- synthetic FP16 checkpoints

@dataclasses.dataclass
class GpuModel:
    """A synthetic FP16 checkpoint on the device (int16 tensors holding FP16
    bits) in the layout seedq_importance reads."""
    spec: W.ModelSpec
    layers: list
    final_norm: torch.Tensor
    lm_head: torch.Tensor

    def dims(self) -> dict:
        s = self.spec
        return dict(n_layers=s.n_layers, d_model=s.d_model, n_heads=s.n_heads,
                    n_kv_heads=s.n_kv_heads, head_dim=s.head_dim, d_ff=s.d_ff, vocab=s.vocab)

    def tensors(self):
        """Weight tensors in model order (per layer q, k, v, o, gate, up, down; the head)."""
        out = []
        for y in self.layers:
            out += [y[k] for k in ("wq", "wk", "wv", "wo", "wgate", "wup", "wdown")]
        return out + [self.lm_head]


def synth_weight_device(spec: W.ModelSpec, layer, kind: str) -> torch.Tensor:
    """One weight matrix drawn on the device by seedq_synth_fp16 (the same
    counter-based values as workloads.synth_weight_rows), super weights planted."""
    R, C = spec.shape(kind)
    t = torch.empty((R, C), dtype=torch.int16, device="cuda")
    Q.synth_fp16(W.weight_key(spec, layer, kind), 0, R * C, W.W_SCALE_M, W.W_SCALE_E, t)
    for (l, k, r, c, bits) in W.super_weights(spec):
        if l == layer and k == kind:
            t[r, c] = int(np.uint16(bits).view(np.int16))
    return t


def synth_model_device(spec: W.ModelSpec) -> GpuModel:
    def gain(l, which):
        return torch.from_numpy(W.synth_gain(spec, l, which).view(np.int16)).cuda()

    kinds = {"wq": "q", "wk": "k", "wv": "v", "wo": "o", "wgate": "gate", "wup": "up", "wdown": "down"}
    layers = []
    for l in range(spec.n_layers):
        y = {"attn_norm": gain(l, "attn"), "mlp_norm": gain(l, "mlp")}
        for name, kind in kinds.items():
            y[name] = synth_weight_device(spec, l, kind)
        layers.append(y)
    return GpuModel(spec, layers, gain(None, "final"), synth_weight_device(spec, None, "lm_head"))


def importance_buffers(spec: W.ModelSpec, with_stats: bool = True) -> dict:
    L, d = spec.n_layers, spec.d_model
    dev = dict(device="cuda")
    out = {"a_o": torch.empty(L * spec.q_dim, dtype=torch.float32, **dev),
           "a_down": torch.empty(L * spec.d_ff, dtype=torch.float32, **dev),
           "rho_o": torch.empty(L * d, dtype=torch.float32, **dev),
           "rho_down": torch.empty(L * d, dtype=torch.float32, **dev)}
    if with_stats:
        ncols = sum(spec.shape(k)[1] for k in W.MODEL_KINDS) * L + d
        out["dyn_range"] = torch.empty(ncols, dtype=torch.float64, **dev)
        out["act_ratio"] = torch.empty(ncols, dtype=torch.float64, **dev)
    return out


def run_importance(m: GpuModel, out: dict, max_outliers: int = 4, stream=None):
    return Q.importance(m.dims(), m.layers, m.final_norm, m.lm_head, out, max_outliers, stream)

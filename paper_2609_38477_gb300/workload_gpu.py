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

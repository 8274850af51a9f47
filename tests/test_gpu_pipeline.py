"""The method end to end on the device: FP16 checkpoint -> data-free importance
and outlier columns (Sec. 3.2, 3.5) -> allocation (Alg. 1) -> exhaustive seed
search at each block's rung and packing (Sec. 3.1, Alg. 1 emit) -> decoder plan
(Alg. 2) -> fused reconstruction + GEMV.

No CUDA output is fed to the oracle here; the checks are properties that tie
the steps together: every tensor's packed stream has exactly the bits the
allocator counted for it, the budget holds, outlier columns come back as their
FP16 values, the decoded weights are the encoder's own reconstruction (their
squared error is the error the search reported; outlier entries are searched as
zero because the FP16 columns overwrite them), and the fused product agrees
with the decoded matrix.
"""
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
sys.path.insert(0, os.path.join(ROOT, "oracle"))

import oracle as O  # noqa: E402
from paper_2609_38477_gb300 import workloads as W  # noqa: E402

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _gain_sq(bits):
    g = np.asarray(bits, np.uint16).view(np.float16).astype(np.float32)
    return g * g


@pytest.mark.parametrize("name", ["tiny", "tiny_odd"])
def test_fp16_checkpoint_to_fused_gemv(name):
    from paper_2609_38477_gb300 import build

    build.build()
    from paper_2609_38477_gb300 import seedq as Q
    from paper_2609_38477_gb300 import workload_gpu as G

    spec = W.MODELS[name]
    gm = G.synth_model_device(spec)
    out = G.importance_buffers(spec, with_stats=False)
    outliers = G.run_importance(gm, out)
    torch.cuda.synchronize()
    assert len(outliers) == 4
    L, d, f, qd = spec.n_layers, spec.d_model, spec.d_ff, spec.q_dim
    a_o = out["a_o"].cpu().numpy().reshape(L, qd)
    a_dn = out["a_down"].cpu().numpy().reshape(L, f)
    r_o = out["rho_o"].cpu().numpy().reshape(L, d)
    r_dn = out["rho_down"].cpu().numpy().reshape(L, d)

    # Per-tensor factors as the decoder would hold them (Sec. 3.6): gains for
    # q, k, v, gate, up and the head, the per-tensor table for o and down.
    tensors = gm.tensors()
    factors = []
    for l in range(L):
        a_attn = _gain_sq(gm.layers[l]["attn_norm"].cpu().numpy().view(np.uint16))
        a_mlp = _gain_sq(gm.layers[l]["mlp_norm"].cpu().numpy().view(np.uint16))
        fa = [(a_attn, None), (a_attn, None), (a_attn, None), (a_o[l], r_o[l]),
              (a_mlp, None), (a_mlp, None), (a_dn[l], r_dn[l])]
        for k, (a, rho) in enumerate(fa):
            R, Cc = tensors[7 * l + k].shape
            factors.append((R, Cc, a, rho))
    R, Cc = tensors[-1].shape
    factors.append((R, Cc, _gain_sq(gm.final_norm.cpu().numpy().view(np.uint16)), None))

    rbar = 4.0
    rungs, _, slopes = O.hull_rungs(W.DAMAGE_TABLES["llama2_7b"](), rbar)
    theta, j_tie, q, T, bits = Q.allocate(factors, rungs, slopes, rbar, 0.06)
    nblocks = sum(R * Cc // 8 for R, Cc, _, _ in factors)
    step = max(O.block_bits(*rungs[j + 1]) - O.block_bits(*rungs[j]) for j in range(len(rungs) - 1))
    budget = int(np.floor(8 * rbar * nblocks))
    assert budget - step < int(bits.sum()) <= budget

    by_tensor = {}
    for t, c in outliers:
        by_tensor.setdefault(t, []).append(c)
    rng = np.random.default_rng(7)
    total_err = 0.0
    total_sq = 0.0
    for i, (Wt, (R, Cc, a, rho)) in enumerate(zip(tensors, factors)):
        ocols = sorted(by_tensor.get(i, []))
        ovals = Wt[:, ocols].contiguous() if ocols else None
        layer = Q.Layer(R, Cc, a, rho, rungs, theta, j_tie, q, int(T[i]),
                        ocols if ocols else None, ovals, max_batch=4)
        assert layer.stream_bits == int(bits[i]), i
        Wf = Wt.view(torch.float16).float().contiguous()
        nb = R * (Cc // 8)
        seed = torch.zeros(nb, dtype=torch.int32, device="cuda")
        E = torch.zeros(nb, dtype=torch.int8, device="cuda")
        tt = torch.zeros(nb * 6, dtype=torch.int8, device="cuda")
        err = torch.zeros(nb, dtype=torch.float64, device="cuda")
        layer.encode(Wf, seed, E, tt, err)  # outlier columns searched as zero
        nbytes = Q.stream_bytes_required(int(bits[i]))
        buf = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
        layer.pack_stream(seed, E, tt, buf, nbytes)
        layer.bind_stream(buf, int(bits[i]), nbytes)
        Wh = torch.empty((R, Cc), dtype=torch.float32, device="cuda")
        layer.decode_weights(Wh)
        torch.cuda.synchronize()
        Wn, Whn = Wf.cpu().numpy().astype(np.float64), Wh.cpu().numpy().astype(np.float64)
        # Outlier columns are the FP16 values; elsewhere the squared error is
        # at most what the seed search reported for the blocks (which also
        # counts the zeroed outlier entries), equal to it without outliers.
        if ocols:
            assert np.array_equal(Whn[:, ocols], Wn[:, ocols]), i
        keep = np.setdiff1d(np.arange(Cc), ocols)
        sq = float(((Whn[:, keep] - Wn[:, keep]) ** 2).sum())
        e = float(err.cpu().numpy().sum())
        assert sq <= e * (1 + 1e-9) + 1e-30, i
        if not ocols:
            assert sq == pytest.approx(e, rel=1e-9), i
        total_err += sq
        total_sq += float((Wn[:, keep] ** 2).sum())
        # The fused kernel multiplies the decoded matrix (R15 criterion).
        xf = rng.normal(0, 1, (4, Cc)).astype(np.float32)
        xb = (xf.view(np.uint32) >> 16).astype(np.uint16)
        xd = (xb.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        X = torch.from_numpy(xb.view(np.int16)).cuda()
        Y = torch.empty((4, R), dtype=torch.float32, device="cuda")
        layer.gemm_small_batch(X, 4, Y)
        torch.cuda.synchronize()
        y64 = xd @ Whn.T
        yabs = np.abs(xd) @ np.abs(Whn).T
        assert np.all(np.abs(Y.cpu().numpy() - y64) <= 1e-3 * yabs + 1e-30), i
        assert layer.device_error() == 0
        layer.release()
    # Four bits per weight of a shared-exponent seed codec on Gaussian blocks:
    # the relative squared error is a few percent.
    assert total_err / total_sq < 0.1

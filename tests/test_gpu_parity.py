"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Bar: the plan (permutation, rung map, row offsets), the synthetic stream and
the reconstructed weights are bit-exact; y = W_hat x meets the output tolerance
derived from fp32 accumulation (reading R15): for every row
|y - y64| <= 1e-3 * sum_c |W_hat_rc x_c|, and max |y - y64| <= 1e-3 max |y64|.
"""
import json
import os

import numpy as np
import pytest

import oracle as O
from paper_2609_38477_gb300 import workloads as W

torch = pytest.importorskip("torch")
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
TOL = 1e-3

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_38477_gb300 import build

    build.build()


def Q():
    from paper_2609_38477_gb300 import seedq

    return seedq


def G():
    from paper_2609_38477_gb300 import workload_gpu

    return workload_gpu


def load(name):
    d = json.load(open(os.path.join(GOLDEN, f"schedule_{name}.json")))
    s = O.Sched([tuple(r) for r in d["rungs"]], d["theta"], d["j_tie"], d["q"])
    return d, s


def otensor(w, i):
    t = w.tensors[i]
    return O.Tensor(t.R, t.C, *W.importance(w, i))


def check_y(y, y64, yabs, cols=28672):
    """Reading R15's criterion, then the fp32 accumulation bound, which is far
    tighter: a block adds at most 8 products, a row at most cols/8 block terms
    in sequence, and at most 32 more additions combine partial sums, so
    |y - y64| <= (cols/8 + 32) 2^-24 sum|W_hat x| to first order (cols defaults
    to the widest tensor of the workloads).  A mis-parsed block moves y by about
    8/cols of sum|W_hat x|, above this bound."""
    y = np.asarray(y, np.float64)
    err = np.abs(y - y64)
    assert err.max() <= TOL * max(np.abs(y64).max(), 1e-30), err.max()
    assert np.all(err <= TOL * yabs + 1e-30), (err / np.maximum(yabs, 1e-30)).max()
    acc = (cols // 8 + 32) * 2.0 ** -24
    assert np.all(err <= acc * yabs + 1e-30), (err / np.maximum(yabs, 1e-30)).max()
    return float((err / np.maximum(yabs, 1e-30)).max())


def gpu_bits(buf: "torch.Tensor", start: int, nbits: int) -> np.ndarray:
    """Bits [start, start+nbits) of a device stream, repacked at bit 0 (host)."""
    b0 = start // 8
    raw = buf[b0:b0 + (nbits + 7) // 8 + 2].cpu().numpy()
    bits = np.unpackbits(raw, bitorder="little")[start - 8 * b0:start - 8 * b0 + nbits]
    return np.packbits(bits, bitorder="little")


def oracle_bits(arr: np.ndarray, nbits: int) -> np.ndarray:
    bits = np.unpackbits(arr, bitorder="little")[:nbits]
    return np.packbits(bits, bitorder="little")


def rung_offsets(d, rm):
    L = np.array([O.block_bits(S, k) for S, k in d["rungs"]], np.uint64)
    return np.concatenate([[0], np.cumsum(L[rm].sum(axis=1, dtype=np.uint64))]).astype(np.uint64)


def x_dev(xb):
    return torch.from_numpy(np.ascontiguousarray(xb).view(np.int16)).cuda()


# ----------------------------------------------------------------- c0 (full)

def test_c0_full_parity():
    w = W.WORKLOADS["c0"]
    d, s = load("c0")
    T = d["tie_count"][0]
    ot = otensor(w, 0)
    gt = G().prepare_tensor(w, 0, d, max_batch=16)
    L = gt.layer
    assert gt.bits == d["stream_bits"][0]
    assert np.array_equal(L.perm(), ot.perm)
    rm = ot.rung_rows(s, T)
    assert np.array_equal(L.rung_map(), rm)
    assert np.array_equal(L.row_offsets(), rung_offsets(d, rm))
    # The device-written synthetic stream equals the oracle's packing, bit for bit.
    ost, obits = ot.synth_pack(s, T, W.payload_key(w, 0))
    assert obits == gt.bits
    assert np.array_equal(gpu_bits(gt.stream, 0, obits), oracle_bits(ost, obits))
    G().bind(gt)
    Wg = torch.empty((ot.R, ot.C), dtype=torch.float32, device="cuda")
    L.decode_weights(Wg)
    Wo = ot.decode_rows(s, T, ost, obits)
    assert np.array_equal(Wg.cpu().numpy(), Wo)
    # Same result from the oracle's own stream uploaded to the device.
    up = torch.zeros(gt.nbytes, dtype=torch.uint8, device="cuda")
    up[:ost.size].copy_(torch.from_numpy(ost[:min(ost.size, gt.nbytes)]))
    L.bind_stream(up, gt.bits, gt.nbytes)
    Wg2 = torch.empty_like(Wg)
    L.decode_weights(Wg2)
    assert torch.equal(Wg, Wg2)
    # y = W_hat x and small batches.
    xb = W.x_bf16(w, 0, 16)
    y64 = O.gemv_f64(Wo, xb)
    yabs = np.abs(Wo.astype(np.float64)) @ np.abs(W.bf16_bits_to_f32(xb).astype(np.float64)).T
    y = torch.empty(ot.R, dtype=torch.float32, device="cuda")
    L.gemv(x_dev(xb[:1]), y)
    check_y(y.cpu().numpy(), y64[0], yabs[:, 0])
    for n in (1, 2, 3, 4, 8, 16):
        Y = torch.empty((n, ot.R), dtype=torch.float32, device="cuda")
        L.gemm_small_batch(x_dev(xb[:n]), n, Y)
        for b in range(n):
            check_y(Y[b].cpu().numpy(), y64[b], yabs[:, b])
    torch.cuda.synchronize()
    assert L.device_error() == 0
    L.release()


# ------------------------------------------------------------- c1, c2 tensors

def _sample_rows(R):
    return sorted({0, 1, 2, R // 3, R // 2 + 1, R - 3, R - 2, R - 1})


@pytest.mark.parametrize("name,i", [("c1", i) for i in range(7)] + [("c2", i) for i in range(7)])
def test_layer_set_tensor(name, i):
    w = W.WORKLOADS[name]
    d, s = load(name)
    T = d["tie_count"][i]
    ot = otensor(w, i)
    nbmax = max(w.batches)
    gt = G().prepare_tensor(w, i, d, max_batch=nbmax)
    L = gt.layer
    assert gt.bits == d["stream_bits"][i]
    assert np.array_equal(L.perm(), ot.perm)
    rm = ot.rung_rows(s, T)
    assert np.array_equal(L.rung_map(), rm)
    offs = L.row_offsets()
    assert np.array_equal(offs, rung_offsets(d, rm))
    key = W.payload_key(w, i)
    for r in _sample_rows(ot.R):
        nbits = int(offs[r + 1] - offs[r])
        ob, got = ot.synth_pack_rows(s, T, key, r, 1, nbits)
        assert got == nbits
        assert np.array_equal(gpu_bits(gt.stream, int(offs[r]), nbits), oracle_bits(ob, nbits))
    G().bind(gt)
    rows = _sample_rows(ot.R)
    Wg = torch.empty((1, ot.C), dtype=torch.float32, device="cuda")
    for r in rows:
        L.decode_rows(r, 1, Wg)
        assert np.array_equal(Wg.cpu().numpy(), ot.synth_rows(s, T, key, r, 1)), r
    xb = W.x_bf16(w, i, nbmax)
    y64, yabs = ot.synth_gemv(s, T, key, xb)
    y = torch.empty(ot.R, dtype=torch.float32, device="cuda")
    L.gemv(x_dev(xb[:1]), y)
    check_y(y.cpu().numpy(), y64[0], yabs[0])
    for n in w.batches:
        if n == 1:
            continue
        Y = torch.empty((n, ot.R), dtype=torch.float32, device="cuda")
        L.gemm_small_batch(x_dev(xb[:n]), n, Y)
        for b in range(n):
            check_y(Y[b].cpu().numpy(), y64[b], yabs[b])
    torch.cuda.synchronize()
    assert L.device_error() == 0
    L.release()


# ------------------------------------------------------ full-size, sampled

@pytest.mark.parametrize("name", ["c3", "c4", "c4_3"])
def test_full_size_sampled(name):
    """Every tensor of the full configuration resident on the device, y for all
    tensors computed in the benchmark's launch configuration; sampled rows
    (two per tensor) checked against the oracle, plus the plan's total bits
    against the stored schedule."""
    w = W.WORKLOADS[name]
    d, s = load(name)
    nbmax = max(w.batches)
    gts = []
    for i in range(len(w.tensors)):
        gt = G().prepare_tensor(w, i, d, max_batch=nbmax)
        assert gt.bits == d["stream_bits"][i]
        G().bind(gt)
        gts.append(gt)
    torch.cuda.synchronize()
    rng = np.random.default_rng(sum(map(ord, name)))
    worst = 0.0
    # Every batch size of the workload, each as the benchmark runs it: all
    # tensors through seedq_gemm_multi, eight per launch.
    Ys = {}
    xbs = {i: W.x_bf16(w, i, nbmax) for i in range(len(w.tensors))}
    xds = {i: x_dev(xbs[i]) for i in range(len(w.tensors))}
    for n in w.batches:
        Ys[n] = [torch.empty((n, t.R), dtype=torch.float32, device="cuda") for t in w.tensors]
        for c0 in range(0, len(gts), 8):
            idx = list(range(c0, min(c0 + 8, len(gts))))
            Q().gemm_multi([gts[i].layer for i in idx], [xds[i][:n] for i in idx], n,
                           [Ys[n][i] for i in idx])
    torch.cuda.synchronize()
    for i, gt in enumerate(gts):
        t = w.tensors[i]
        xb = xbs[i]
        rows = sorted({int(rng.integers(0, t.R)), t.R - 1})
        ot = otensor(w, i)
        key = W.payload_key(w, i)
        for r in rows:
            assert np.array_equal(gt.layer.rung_map(r, 1), ot.rung_rows(s, d["tie_count"][i], r, 1))
        for n in w.batches:
            Yh = Ys[n][i].cpu().numpy()
            for r in rows:
                y64, yabs = ot.synth_gemv(s, d["tie_count"][i], key, xb[:n], r, 1)
                worst = max(worst, check_y(Yh[:, r], y64[:, 0], yabs[:, 0]))
        Wg = torch.empty((1, t.C), dtype=torch.float32, device="cuda")
        gt.layer.decode_rows(rows[0], 1, Wg)
        assert np.array_equal(Wg.cpu().numpy(), ot.synth_rows(s, d["tie_count"][i], key, rows[0], 1))
    for gt in gts:
        assert gt.layer.device_error() == 0
        gt.layer.release()
    print(f"{name}: worst |y-y64| / sum|w x| = {worst:.3e}")


# --------------------------------------------------------------- edge cases

def _small_case(R, Cc, rungs, theta, j_tie, q, rho=True, seed=0, T=0, n_out=0):
    rng = np.random.default_rng(seed)
    a = np.exp(rng.normal(0, 1, Cc)).astype(np.float32)
    rh = np.exp(rng.normal(0, 0.5, R)).astype(np.float32) if rho else None
    ot = O.Tensor(R, Cc, a, rh)
    s = O.Sched(rungs, theta, j_tie, q)
    key = int(rng.integers(1, 2 ** 62))
    ost, bits = ot.synth_pack(s, T, key)
    cols = vals = None
    if n_out:
        cols = rng.choice(Cc, n_out, replace=False).astype(np.int32)
        vals = W.to_f16_bits(rng.normal(0, 4, (R, n_out)).astype(np.float32))
    return a, rh, ot, s, ost, bits, cols, vals


def _gpu_layer(R, Cc, a, rh, s, T, ost, bits, cols, vals, max_batch=16):
    vd = None if vals is None else torch.from_numpy(np.ascontiguousarray(vals).view(np.int16)).cuda()
    L = Q().Layer(R, Cc, a, rh, s.rungs, s.theta, s.j_tie, s.q, T, cols, vd, max_batch=max_batch)
    L._keep = vd
    assert L.stream_bits == bits
    nbytes = Q().stream_bytes_required(bits)
    buf = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
    n = min(ost.size, nbytes)
    buf[:n].copy_(torch.from_numpy(ost[:n]))
    L.bind_stream(buf, bits, nbytes)
    L._buf = buf
    return L


EDGE = [
    # R, C, rungs, theta, j_tie, q, rho, T, n_out
    (1, 8, [(16, 3)], [], -1, 0.0, False, 0, 0),                       # one block, one rung
    (7, 296, [(8, 2), (12, 3), (16, 6)], [0.7, 1.3], -1, 0.2, True, 0, 0),  # ragged group
    (33, 1024, [(10, 3), (14, 4), (16, 5)], [0.8, 1.5], 0, 0.0, False, 40, 4),  # ties + outliers
    (5, 65536, [(8, 3), (16, 3)], [1.0], -1, 0.5, True, 0, 0),          # widest rows, split-K
    (300, 64, [(8, 2), (10, 2), (12, 2), (14, 2), (16, 2), (16, 3), (14, 4)],
     [0.3, 0.5, 0.8, 1.1, 1.6, 2.5], -1, 0.1, True, 0, 2),
]


@pytest.mark.parametrize("case", range(len(EDGE)))
def test_edge_cases(case):
    R, Cc, rungs, theta, j_tie, q, rho, T, n_out = EDGE[case]
    a, rh, ot, s, ost, bits, cols, vals = _small_case(R, Cc, rungs, theta, j_tie, q, rho, case, 0, n_out)
    if j_tie >= 0:  # tie the first rung boundary at an attained importance value
        v = ot.imp(s, 0, Cc // 8 // 2)
        theta = [v] + [max(t, 2.0 * v * (j + 1)) for j, t in enumerate(theta[1:])]
        s = O.Sched(rungs, theta, j_tie, q)
        tied = ot.tied_blocks(s)
        T = min(T, max(tied - 1, 1))
        assert 0 < T <= tied
        ost, bits = ot.synth_pack(s, T, 77)
    L = _gpu_layer(R, Cc, a, rh, s, T, ost, bits, cols, vals)
    assert np.array_equal(L.rung_map(), ot.rung_rows(s, T))
    Wo = ot.decode_rows(s, T, ost, bits, 0, R, cols, vals)
    Wg = torch.empty((R, Cc), dtype=torch.float32, device="cuda")
    L.decode_weights(Wg)
    assert np.array_equal(Wg.cpu().numpy(), Wo)
    L.decode_rows(0, 0, Wg)  # empty range is a no-op
    xb = W.to_bf16_bits(np.random.default_rng(case).normal(0, 1, (16, Cc)).astype(np.float32))
    y64 = O.gemv_f64(Wo, xb)
    yabs = np.abs(Wo.astype(np.float64)) @ np.abs(W.bf16_bits_to_f32(xb).astype(np.float64)).T
    for n in (1, 3, 16):
        Y = torch.empty((n, R), dtype=torch.float32, device="cuda")
        if n == 1:
            L.gemv(x_dev(xb[:1]), Y[0])
        else:
            L.gemm_small_batch(x_dev(xb[:n]), n, Y)
        for b in range(n):
            check_y(Y[b].cpu().numpy(), y64[b], yabs[:, b])
    torch.cuda.synchronize()
    assert L.device_error() == 0
    L.release()


TIES = [
    # R, C, number of distinct a values, number of distinct rho values
    (3, 1024, 1, 0),      # every channel tied: identity order, one whole sort chunk
    (1030, 1032, 3, 3),   # one chunk plus a 8-key tail; rows ranked by tied rho
    (257, 3000, 2, 2),    # three chunks, ragged last one
    (64, 4104, 5, 1),     # five chunks; rho all equal after its unit mean
]


@pytest.mark.parametrize("case", range(len(TIES)))
def test_ranking_ties(case):
    """Sec. 3.3 sorts channels ascending by a with ties by channel index, and
    the rows are ordered by rho; with few distinct values nearly every key is
    tied, across the boundaries of the device's 1024-key sort chunks."""
    R, Cc, na, nr = TIES[case]
    rng = np.random.default_rng(100 + case)
    a = rng.choice(np.array([0.5, 1.0, 2.0, 3.0, 0.25], np.float32)[:na], Cc)
    rh = None if nr == 0 else rng.choice(np.array([0.8, 1.0, 1.25], np.float32)[:nr], R)
    ot = O.Tensor(R, Cc, a, rh)
    s = O.Sched([(8, 2), (12, 3), (16, 4)], [0.9, 1.2], -1, 0.1)
    ost, bits = ot.synth_pack(s, 0, 4242 + case)
    L = _gpu_layer(R, Cc, a, rh, s, 0, ost, bits, None, None)
    assert np.array_equal(L.perm(), np.argsort(a, kind="stable"))
    assert np.array_equal(L.rung_map(), ot.rung_rows(s, 0))
    Wo = ot.decode_rows(s, 0, ost, bits)
    Wg = torch.empty((R, Cc), dtype=torch.float32, device="cuda")
    L.decode_weights(Wg)
    assert np.array_equal(Wg.cpu().numpy(), Wo)
    xb = W.to_bf16_bits(rng.normal(0, 1, (3, Cc)).astype(np.float32))
    y64 = O.gemv_f64(Wo, xb)
    yabs = np.abs(Wo.astype(np.float64)) @ np.abs(W.bf16_bits_to_f32(xb).astype(np.float64)).T
    Y = torch.empty((3, R), dtype=torch.float32, device="cuda")
    L.gemv(x_dev(xb[:1]), Y[0])
    check_y(Y[0].cpu().numpy(), y64[0], yabs[:, 0])
    L.gemm_small_batch(x_dev(xb), 3, Y)
    for b in range(3):  # every output row written once, in its own place
        check_y(Y[b].cpu().numpy(), y64[b], yabs[:, b])
    torch.cuda.synchronize()
    assert L.device_error() == 0
    L.release()


def test_seed_zero_and_seed_fault():
    """Reading R12: a zero seed decodes as the all-zero sequence on both sides.
    Sec. 4.3: flipping one seed bit changes at most the 8 weights of its block."""
    R, Cc = 4, 256
    a, rh, ot, s, ost, bits, _, _ = _small_case(R, Cc, [(8, 3), (16, 3)], [1.0], -1, 0.0, False, 9)
    L = _gpu_layer(R, Cc, a, rh, s, 0, ost, bits, None, None)
    rm = ot.rung_rows(s, 0)
    Lb = [O.block_bits(S, k) for S, k in s.rungs]
    off = int(sum(Lb[j] for j in rm[0]) + sum(Lb[j] for j in rm[1][:5]))  # block 5 of row 1
    S5 = s.rungs[rm[1][5]][0]
    zero = ost.copy()
    O.write_bits(zero, off, S5, 0)
    flip = ost.copy()
    flip[(off + 3) >> 3] ^= np.uint8(1 << ((off + 3) & 7))
    Wg = torch.empty((R, Cc), dtype=torch.float32, device="cuda")
    L.decode_weights(Wg)
    clean = Wg.cpu().numpy()
    for bad in (zero, flip):
        L._buf[:bad.size].copy_(torch.from_numpy(bad[:L._buf.numel()]))
        L.decode_weights(Wg)
        got = Wg.cpu().numpy()
        assert np.array_equal(got, ot.decode_rows(s, 0, bad, bits))
        diff = np.argwhere(got != clean)
        assert 1 <= len(diff) <= 8 and set(diff[:, 0]) == {1}
    L.release()


def test_api_errors_and_determinism():
    R, Cc = 16, 512
    a, rh, ot, s, ost, bits, _, _ = _small_case(R, Cc, [(8, 3), (16, 3)], [1.0], -1, 0.0, True, 3)
    Qm = Q()
    L = Qm.Layer(R, Cc, a, rh, s.rungs, s.theta, s.j_tie, s.q, 0, max_batch=4)
    x = torch.zeros((1, Cc), dtype=torch.int16, device="cuda")
    y = torch.empty(R, dtype=torch.float32, device="cuda")
    with pytest.raises(Qm.SeedQError) as e:
        L.gemv(x, y)
    assert e.value.status == 2  # no stream bound
    nbytes = Qm.stream_bytes_required(bits)
    buf = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
    for bb, nn in ((bits + 1, nbytes), (bits, nbytes - 16)):
        with pytest.raises(Qm.SeedQError) as e:
            L.bind_stream(buf, bb, nn)
        assert e.value.status == 2
    buf[:ost.size].copy_(torch.from_numpy(ost[:nbytes]))
    L.bind_stream(buf, bits, nbytes)
    with pytest.raises(Qm.SeedQError) as e:
        L.gemm_small_batch(x, 5, y)  # above max_batch
    assert e.value.status == 1
    with pytest.raises(Qm.SeedQError) as e:
        L.decode_rows(R - 1, 2, y)
    assert e.value.status == 1
    xb = W.to_bf16_bits(np.random.default_rng(1).normal(0, 1, (1, Cc)).astype(np.float32))
    xd = x_dev(xb)
    y2 = torch.empty_like(y)
    L.gemv(xd, y)
    L.gemv(xd, y2)
    assert torch.equal(y, y2)
    L.release()
    # More demotions than tied blocks is a schedule error.
    s2 = O.Sched(s.rungs, [ot.imp(s, 0, 10)], 0, 0.0)
    tied = ot.tied_blocks(s2)
    with pytest.raises(Qm.SeedQError) as e:
        Qm.Layer(R, Cc, a, rh, s2.rungs, s2.theta, 0, 0.0, tied + 1)
    assert e.value.status == 3


@pytest.mark.parametrize("name", ["c1", "c2"])
def test_layer_set_multi_launch(name):
    """The benchmark's step: all seven tensors in one seedq_gemm_multi launch,
    every output row checked against the oracle, at each batch size."""
    w = W.WORKLOADS[name]
    d, s = load(name)
    nbmax = max(w.batches)
    gts = [G().bind(G().prepare_tensor(w, i, d, max_batch=nbmax)) for i in range(len(w.tensors))]
    xbs = [W.x_bf16(w, i, nbmax) for i in range(len(w.tensors))]
    xds = [x_dev(x) for x in xbs]
    ref = [otensor(w, i).synth_gemv(s, d["tie_count"][i], W.payload_key(w, i), xbs[i])
           for i in range(len(w.tensors))]
    for n in w.batches:
        Ys = [torch.empty((n, t.R), dtype=torch.float32, device="cuda") for t in w.tensors]
        Q().gemm_multi([g.layer for g in gts], [x[:n] for x in xds], n, Ys)
        torch.cuda.synchronize()
        for i in range(len(gts)):
            Yh = Ys[i].cpu().numpy()
            for b in range(n):
                check_y(Yh[b], ref[i][0][b], ref[i][1][b])
    for g in gts:
        assert g.layer.device_error() == 0
        g.layer.release()


@pytest.mark.parametrize("name", ["c1", "c2"])
def test_layer_set_one_launch(name):
    """A layer set over all seven tensors: one launch per call, x and y of all
    tensors in one buffer each.  Same partition and arithmetic as the
    multi-tensor launch, so the outputs are bit-identical to it; every row is
    also checked against the oracle, at each batch size."""
    w = W.WORKLOADS[name]
    d, s = load(name)
    nbmax = max(w.batches)
    gts = [G().bind(G().prepare_tensor(w, i, d, max_batch=nbmax)) for i in range(len(w.tensors))]
    layers = [g.layer for g in gts]
    ls = Q().LayerSet(layers)
    co, ro = ls.col_offsets, ls.row_offsets
    assert list(np.diff(co)) == [t.C for t in w.tensors] and list(np.diff(ro)) == [t.R for t in w.tensors]
    xbs = [W.x_bf16(w, i, nbmax) for i in range(len(w.tensors))]
    ref = [otensor(w, i).synth_gemv(s, d["tie_count"][i], W.payload_key(w, i), xbs[i])
           for i in range(len(w.tensors))]
    for n in w.batches:
        X = torch.from_numpy(np.concatenate([x[:n].reshape(-1) for x in xbs]).view(np.int16)).cuda()
        Y = torch.full((n * int(ro[-1]),), float("nan"), dtype=torch.float32, device="cuda")
        ls.gemm(X, n, Y)
        Ym = [torch.empty((n, t.R), dtype=torch.float32, device="cuda") for t in w.tensors]
        Q().gemm_multi(layers, [x_dev(x[:n]) for x in xbs], n, Ym)
        torch.cuda.synchronize()
        Yh = Y.cpu().numpy()
        for i, t in enumerate(w.tensors):
            yi = Yh[n * ro[i]:n * ro[i + 1]].reshape(n, t.R)
            assert np.array_equal(yi, Ym[i].cpu().numpy()), (name, n, t.name)
            for b in range(n):
                check_y(yi[b], ref[i][0][b], ref[i][1][b])
    with pytest.raises(Q().SeedQError):
        ls.gemm(X, nbmax + 1, Y)
    ls.release()
    for g in gts:
        assert g.layer.device_error() == 0
        g.layer.release()


def test_layer_set_full_model_sampled():
    """The Llama-3-8B-shaped set (225 tensors) in one launch per call; sampled
    rows of every tensor against the oracle."""
    name = "c3"
    w = W.WORKLOADS[name]
    d, s = load(name)
    gts = [G().bind(G().prepare_tensor(w, i, d, max_batch=1)) for i in range(len(w.tensors))]
    ls = Q().LayerSet([g.layer for g in gts])
    ro = ls.row_offsets
    xbs = [W.x_bf16(w, i, 1) for i in range(len(w.tensors))]
    X = torch.from_numpy(np.concatenate([x.reshape(-1) for x in xbs]).view(np.int16)).cuda()
    Y = torch.full((int(ro[-1]),), float("nan"), dtype=torch.float32, device="cuda")
    ls.gemm(X, 1, Y)
    torch.cuda.synchronize()
    Yh = Y.cpu().numpy()
    assert not np.isnan(Yh).any()
    rng = np.random.default_rng(4242)
    for i, t in enumerate(w.tensors):
        r = int(rng.integers(0, t.R))
        y64, yabs = otensor(w, i).synth_gemv(s, d["tie_count"][i], W.payload_key(w, i), xbs[i], r0=r, nrows=1)
        err = abs(float(Yh[ro[i] + r]) - y64[0][0])
        assert err <= TOL * yabs[0][0] + 1e-30, (t.name, r)
    ls.release()
    for g in gts:
        g.layer.release()

"""Bit-exact parity of the CUDA path at full size (through the C ABI).

- The fused kernel's own parse and reconstruction: with one-hot activations
  x_b = e_j every output is a single exact product (Eq. codec: W_hat = I 2^(E-S+1),
  times 1.0), so Y[b] must equal column j of the oracle's W_hat bit for bit.
  The columns hit the first and last block, rung breakpoints, stage boundaries
  of every batch template and row groups cut between CTAs.
- Reconstructed weights (seedq_decode_weights) equal the oracle's in full for
  every tensor of the Llama-2-7B-shaped sets, and for one tensor of every
  distinct shape of the 32- and 80-layer models, plus 64 random rows of every
  tensor.
- The device error word: a layer whose readable stream is cut short reports
  bit 0 and the kernels return without reading past the limit.
"""
import concurrent.futures as cf
import json
import os

import numpy as np
import pytest

import oracle as O
from paper_2609_38477_gb300 import workloads as W

torch = pytest.importorskip("torch")
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
THREADS = max(1, min(os.cpu_count() or 1, 32))
ONE_BF16 = 0x3F80  # 1.0

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


def x_dev(xb):
    return torch.from_numpy(np.ascontiguousarray(xb).view(np.int16)).cuda()


def oracle_chunks(ot, s, T, key, rows, chunk=1024):
    """Oracle rows [a, b) for consecutive chunks of `rows` (a range), computed
    in parallel host threads (the C oracle runs without the GIL)."""
    r0, r1 = rows
    starts = list(range(r0, r1, chunk))
    with cf.ThreadPoolExecutor(THREADS) as ex:
        futs = [ex.submit(ot.synth_rows, s, T, key, a, min(chunk, r1 - a)) for a in starts]
        for a, f in zip(starts, futs):
            yield a, f.result()


def compare_full(layer, ot, s, T, key, cols=None, chunk=1024):
    """Decode the whole tensor on the device and compare it with the oracle in
    row chunks; returns W_hat[:, cols] from the oracle if cols is given."""
    R, Cc = ot.R, ot.C
    Wg = torch.empty((min(chunk, R), Cc), dtype=torch.float32, device="cuda")
    picked = None if cols is None else np.zeros((R, len(cols)), np.float32)
    for a, Wo in oracle_chunks(ot, s, T, key, (0, R), chunk):
        n = Wo.shape[0]
        layer.decode_rows(a, n, Wg[:n])
        got = Wg[:n].cpu().numpy()
        if not np.array_equal(got, Wo):
            bad = np.argwhere(got != Wo)[0]
            raise AssertionError(f"row {a + bad[0]} col {bad[1]}: {got[tuple(bad)]} vs {Wo[tuple(bad)]}")
        if picked is not None:
            picked[a:a + n] = Wo[:, cols]
    return picked


def pick_columns(ot, s, T, count, seed):
    """`count` original columns whose blocks cover the first and last block,
    the rung breakpoints of row 0, the stage boundaries of every batch template
    (27, 21, 15, 12, 7 columns) and the middle; random blocks fill the rest."""
    nb = ot.C // 8
    rm0 = ot.rung_rows(s, T, 0, 1)[0]
    brk = [c for c in range(1, nb) if rm0[c] != rm0[c - 1]]
    cands = [0, nb - 1] + [v for b in brk for v in (b - 1, b)]
    cands += [v for st in (27, 21, 15, 12, 7) for v in (st - 1, st, 2 * st)] + [nb // 2]
    blocks = []
    for c in cands:
        if 0 <= c < nb and c not in blocks:
            blocks.append(c)
    rng = np.random.default_rng(seed)
    while len(blocks) < count:
        c = int(rng.integers(0, nb))
        if c not in blocks:
            blocks.append(c)
    blocks = blocks[:count]
    perm = ot.perm
    return [int(perm[8 * c + (c * 5) % 8]) for c in blocks]


def one_hot(cols, C):
    x = np.zeros((len(cols), C), np.uint16)
    for b, j in enumerate(cols):
        x[b, j] = ONE_BF16
    return x


@pytest.mark.parametrize("name", ["c1", "c2"])
def test_full_weights_and_one_hot(name):
    """Every tensor of the set: W_hat in full equals the oracle's; then the whole
    set in one fused launch (seedq_gemm_multi) and in one layer-set launch with
    one-hot activations gives exactly the oracle's columns, at every batch
    template the configuration uses."""
    w = W.WORKLOADS[name]
    d, s = load(name)
    nt = len(w.tensors)
    gts, refs, cols = [], [], []
    for i in range(nt):
        gt = G().prepare_tensor(w, i, d, max_batch=16)
        G().bind(gt)
        gts.append(gt)
        ot = otensor(w, i)
        T = d["tie_count"][i]
        cols.append(pick_columns(ot, s, T, 16, 100 + i))
        refs.append(compare_full(gt.layer, ot, s, T, W.payload_key(w, i), cols[i]))
    layers = [g.layer for g in gts]
    batches = [16, 1] if name == "c1" else [8, 4, 2, 1]
    for n in batches:
        for off in range(0, min(16, 2 * n), n):  # two launches per template (one at n = 16)
            sub = [c[off:off + n] for c in cols]
            xs = [x_dev(one_hot(sub[i], w.tensors[i].C)) for i in range(nt)]
            ys = [torch.empty((n, t.R), dtype=torch.float32, device="cuda") for t in w.tensors]
            Q().gemm_multi(layers, xs, n, ys)
            torch.cuda.synchronize()
            for i in range(nt):
                got = ys[i].cpu().numpy()
                want = refs[i][:, off:off + n].T
                assert np.array_equal(got, want), (name, i, n, off, np.argwhere(got != want)[:3])
    # one layer-set launch over all tensors (descriptors in device memory)
    lset = Q().LayerSet(layers)
    n = 16 if name == "c1" else 8
    xcat = torch.cat([x_dev(one_hot(cols[i][:n], w.tensors[i].C)).reshape(-1) for i in range(nt)])
    ycat = torch.empty(sum(n * t.R for t in w.tensors), dtype=torch.float32, device="cuda")
    lset.gemm(xcat, n, ycat)
    torch.cuda.synchronize()
    yh, oy = ycat.cpu().numpy(), 0
    for i, t in enumerate(w.tensors):
        assert np.array_equal(yh[oy:oy + n * t.R].reshape(n, t.R), refs[i][:, :n].T), (name, "set", i)
        oy += n * t.R
    lset.release()
    for g in gts:
        assert g.layer.device_error() == 0
        g.layer.release()


def check_y(y, y64, yabs, cols):
    """Output criterion (reading R15) plus the fp32 accumulation bound: a block
    adds at most 8 products, a row at most cols/8 block terms in sequence, and
    at most 32 more additions combine partial sums (warps, CTAs, outlier term),
    so |y - y64| <= (cols/8 + 32) 2^-24 sum |W_hat x| (first order)."""
    y = np.asarray(y, np.float64)
    err = np.abs(y - y64)
    assert err.max() <= 1e-3 * max(np.abs(y64).max(), 1e-30), err.max()
    assert np.all(err <= 1e-3 * yabs + 1e-30)
    acc = (cols // 8 + 32) * 2.0 ** -24
    assert np.all(err <= acc * yabs + 1e-30), (err / np.maximum(yabs, 1e-30)).max()
    return float((err / np.maximum(yabs, 1e-30)).max())


@pytest.mark.parametrize("name", ["c3", "c4", "c4_3"])
def test_full_size(name):
    """Every tensor of the model resident; y of all tensors from one layer-set
    launch per batch size (the benchmark's launch).  Per tensor: 64 rows (eight
    random windows of eight) bit-exact against the oracle, their rung map, and
    their y.  For one tensor of every distinct shape: W_hat in full and y of
    every row."""
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
    xbs = [W.x_bf16(w, i, nbmax) for i in range(len(w.tensors))]
    xcat = torch.cat([x_dev(x).reshape(-1) for x in xbs])
    lset = Q().LayerSet([g.layer for g in gts])
    roff = np.concatenate([[0], np.cumsum([t.R for t in w.tensors])])
    Ys = {}
    for n in w.batches:
        xn = torch.cat([x_dev(x[:n]).reshape(-1) for x in xbs])
        y = torch.empty(int(roff[-1]) * n, dtype=torch.float32, device="cuda")
        lset.gemm(xn, n, y)
        torch.cuda.synchronize()
        yh = y.cpu().numpy()
        Ys[n] = [yh[n * roff[i]:n * roff[i + 1]].reshape(n, w.tensors[i].R) for i in range(len(w.tensors))]
    del xcat
    rng = np.random.default_rng(sum(map(ord, name)))
    windows = [sorted({int(v) for v in rng.integers(0, t.R - 8, 8)} | {t.R - 8}) for t in w.tensors]

    # the oracle's factor set-up sorts with a file-scope key: build them here,
    # in one thread, and only run the row generators in the pool
    ots = [otensor(w, i) for i in range(len(w.tensors))]

    def oracle_side(i):
        ot = ots[i]
        T, key = d["tie_count"][i], W.payload_key(w, i)
        out = []
        for a in windows[i]:
            rm = ot.rung_rows(s, T, a, 8)
            Wo = ot.synth_rows(s, T, key, a, 8)
            y64, yabs = ot.synth_gemv(s, T, key, xbs[i], a, 8, nthreads=1)
            out.append((a, rm, Wo, y64, yabs))
        return out

    worst = 0.0
    Wflat = torch.empty(8 * max(t.C for t in w.tensors), dtype=torch.float32, device="cuda")
    with cf.ThreadPoolExecutor(THREADS) as ex:
        for i, res in enumerate(ex.map(oracle_side, range(len(w.tensors)))):
            t, L = w.tensors[i], gts[i].layer
            for a, rm, Wo, y64, yabs in res:
                assert np.array_equal(L.rung_map(a, 8), rm), (i, a)
                Wg = Wflat[:8 * t.C].view(8, t.C)  # contiguous rows of this tensor's width
                L.decode_rows(a, 8, Wg)
                assert np.array_equal(Wg.cpu().numpy(), Wo), (i, a)
                for n in w.batches:
                    for b in range(n):
                        worst = max(worst, check_y(Ys[n][i][b, a:a + 8], y64[b], yabs[b], t.C))
    # one tensor of every distinct shape: all of W_hat, all rows of y
    shapes = {}
    for i, t in enumerate(w.tensors):
        shapes.setdefault((t.R, t.C), i)
    for (R, Cc), i in sorted(shapes.items()):
        ot = ots[i]
        T, key = d["tie_count"][i], W.payload_key(w, i)
        compare_full(gts[i].layer, ot, s, T, key)
        y64, yabs = ot.synth_gemv(s, T, key, xbs[i], nthreads=THREADS)
        for n in w.batches:
            for b in range(n):
                worst = max(worst, check_y(Ys[n][i][b], y64[b], yabs[b], Cc))
    lset.release()
    for g in gts:
        assert g.layer.device_error() == 0
        g.layer.release()
    print(f"{name}: worst |y-y64| / sum|w x| = {worst:.3e}")


def test_device_error_word():
    """Bit 0 of the device error word: a layer whose readable stream is cut
    short of what the plan needs (seedq_layer_limit_stream_bytes) makes the
    fused kernel and the decode kernel stop their reads at the limit and report
    it; rows that never reach the limit keep their exact results, and a layer
    with the full stream reports nothing."""
    w = W.WORKLOADS["c0"]
    d, s = load("c0")
    gt = G().bind(G().prepare_tensor(w, 0, d, max_batch=16))
    ref = G().bind(G().prepare_tensor(w, 0, d, max_batch=16))
    L, R, Cc = gt.layer, w.tensors[0].R, w.tensors[0].C
    xb = x_dev(W.x_bf16(w, 0, 1))
    y0 = torch.empty(R, dtype=torch.float32, device="cuda")
    y1 = torch.empty(R, dtype=torch.float32, device="cuda")
    ref.layer.gemv(xb, y0)
    torch.cuda.synchronize()
    assert L.device_error() == 0 and ref.layer.device_error() == 0
    with pytest.raises(Q().SeedQError):
        L.limit_stream_bytes(gt.nbytes + 16)
    offs = L.row_offsets()
    cut = int(offs[R - 40]) // 8 // 16 * 16  # rows from R - 41 on reach past it
    L.limit_stream_bytes(cut)
    L.gemv(xb, y1)
    torch.cuda.synchronize()  # the kernel returned; the context is intact
    assert L.device_error() & 1
    # rows wholly below the limit (and their stage read-ahead) are unchanged
    safe = int(np.searchsorted(offs, max(0, 8 * cut - 2048), side="right")) - 2
    assert safe > R // 2
    a, b = y0.cpu().numpy(), y1.cpu().numpy()
    np.testing.assert_array_equal(a[:safe], b[:safe])
    # the decode kernel reports the same and writes only readable blocks
    gt2 = G().bind(G().prepare_tensor(w, 0, d, max_batch=1))
    gt2.layer.limit_stream_bytes(cut)
    Wg = torch.zeros((4, Cc), dtype=torch.float32, device="cuda")
    gt2.layer.decode_rows(0, 4, Wg)
    torch.cuda.synchronize()
    assert gt2.layer.device_error() == 0
    gt2.layer.decode_rows(R - 4, 4, Wg)
    torch.cuda.synchronize()
    assert gt2.layer.device_error() & 1
    # a healthy layer still reports nothing after all of this
    ref.layer.gemv(xb, y0)
    torch.cuda.synchronize()
    assert ref.layer.device_error() == 0
    for g in (gt, ref, gt2):
        g.layer.release()

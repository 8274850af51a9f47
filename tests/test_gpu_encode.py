"""Encoder parity: the GPU exhaustive seed search and stream packing against
the oracle's encoder (Sec. 3.1 seed search, Alg. 1 emit step).

Every decision of the search (pivot rows, exponent, mantissas, winning seed) is
taken in fp64 with the same rounding steps on both sides, so the GPU fields and
errors must equal the oracle's exactly.
"""
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
sys.path.insert(0, os.path.join(ROOT, "oracle"))

import oracle as O  # noqa: E402

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _lib():
    from paper_2609_38477_gb300 import build

    build.build()
    from paper_2609_38477_gb300 import seedq as Q

    return Q


def _blocks(rng, n, S, k):
    """Random blocks, a zero block, and blocks planted exactly on the codebook."""
    w = rng.normal(0.0, 0.02, (n, 8)).astype(np.float32)
    w[0] = 0.0
    taps = O.find_taps(S)
    for i in range(1, min(n, 4)):
        seed = int(rng.integers(1, 1 << S))
        E = int(rng.integers(-8, -2))
        t = rng.integers(-8, 8, k).tolist()
        w[i] = O.reconstruct_block(S, k, taps, seed, E, t)
    if n > 6:
        # Wide exponent spread (the rounded right-hand-side path) and a block
        # with zero entries and a subnormal (the exact path).
        w[4] = np.array([3e-7, -0.05, 0.02, 1e-5, -0.03, 0.011, -2e-6, 0.04], np.float32)
        w[5] = np.array([0.0, -0.01, 0.0, 0.013, 1e-40, -0.02, 0.0, 0.008], np.float32)
    return w


def _gpu_encode(Q, S, k, w):
    n = w.shape[0]
    wd = torch.from_numpy(w).cuda()
    seed = torch.zeros(n, dtype=torch.int32, device="cuda")
    E = torch.zeros(n, dtype=torch.int8, device="cuda")
    t = torch.zeros(n * 6, dtype=torch.int8, device="cuda")
    err = torch.zeros(n, dtype=torch.float64, device="cuda")
    Q.encode_blocks(S, k, wd, n, seed, E, t, err)
    torch.cuda.synchronize()
    return (seed.cpu().numpy().view(np.uint32), E.cpu().numpy(), t.cpu().numpy().reshape(n, 6),
            err.cpu().numpy())


@pytest.mark.parametrize("S,k,n", [(8, 2, 96), (8, 3, 96), (8, 6, 48), (10, 4, 64), (10, 5, 48),
                                   (12, 3, 32), (12, 2, 32), (16, 3, 3)])
def test_encode_blocks_match_oracle(S, k, n):
    Q = _lib()
    rng = np.random.default_rng(1000 * S + k)
    w = _blocks(rng, n, S, k)
    gs, gE, gt, gerr = _gpu_encode(Q, S, k, w)
    taps = O.find_taps(S)
    for b in range(n):
        seed, E, t, err = O.encode_block(S, k, taps, w[b].astype(np.float64))
        assert (int(gs[b]), int(gE[b]), list(gt[b, :k])) == (seed, E, list(t)), f"block {b}"
        assert gerr[b] == err, f"block {b}: {gerr[b]!r} != {err!r}"
        assert not gt[b, k:].any()
    # Planted blocks are reproduced with zero error.
    assert np.all(gerr[1:min(n, 4)] == 0.0)


def test_encode_rejects_unsupported_rungs():
    Q = _lib()
    w = torch.zeros((1, 8), dtype=torch.float32, device="cuda")
    o = torch.zeros(8, dtype=torch.int32, device="cuda")
    for S, k in ((9, 3), (18, 3), (8, 1), (8, 7)):
        with pytest.raises(Q.SeedQError) as e:
            Q.encode_blocks(S, k, w, 1, o, o, o, None)
        assert e.value.status == 6


def test_encode_layer_pack_decode_round_trip():
    """A layer with several rungs: encode every block at its rung on the GPU,
    pack, bind, decode.  Fields equal the oracle's search at the oracle's rung
    map; the packed stream equals the oracle's packing of its own fields; the
    decoded weights equal the oracle's reconstruction."""
    Q = _lib()
    rng = np.random.default_rng(7)
    R, Cc = 48, 128
    a = np.exp(rng.normal(0, 1, Cc)).astype(np.float32)
    rho = np.exp(rng.normal(0, 0.5, R)).astype(np.float32)
    rungs = [(8, 2), (8, 3), (10, 3), (12, 3), (10, 5)]
    theta = [0.5, 0.8, 1.2, 2.0]
    s = O.Sched(rungs, theta, -1, 0.0)
    ot = O.Tensor(R, Cc, a, rho)
    rm = ot.rung_rows(s, 0)
    assert len(set(rm.ravel().tolist())) >= 4
    W = rng.normal(0, 0.02, (R, Cc)).astype(np.float32)

    layer = Q.Layer(R, Cc, a, rho, rungs, theta, -1, 0.0, 0, max_batch=1)
    nb = Cc // 8
    Wd = torch.from_numpy(W).cuda()
    seed = torch.zeros(R * nb, dtype=torch.int32, device="cuda")
    E = torch.zeros(R * nb, dtype=torch.int8, device="cuda")
    t = torch.zeros(R * nb * 6, dtype=torch.int8, device="cuda")
    err = torch.zeros(R * nb, dtype=torch.float64, device="cuda")
    layer.encode(Wd, seed, E, t, err)
    bits = layer.stream_bits
    nbytes = Q.stream_bytes_required(bits)
    buf = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    layer.pack_stream(seed, E, t, buf, nbytes)
    torch.cuda.synchronize()
    gs = seed.cpu().numpy().view(np.uint32).reshape(R, nb)
    gE = E.cpu().numpy().reshape(R, nb)
    gt = t.cpu().numpy().reshape(R, nb, 6)
    gerr = err.cpu().numpy().reshape(R, nb)

    perm = ot.perm
    ref_stream = np.zeros(nbytes, np.uint8)
    ref_W = np.zeros((R, Cc), np.float32)
    pos = 0
    for r in range(R):
        for c in range(nb):
            S, k = rungs[rm[r, c]]
            taps = O.find_taps(S)
            blk = W[r, perm[8 * c:8 * c + 8]].astype(np.float64)
            sd, e, tt, er = O.encode_block(S, k, taps, blk)
            assert (int(gs[r, c]), int(gE[r, c]), list(gt[r, c, :k])) == (sd, e, list(tt)), (r, c)
            assert gerr[r, c] == er, (r, c)
            O.write_bits(ref_stream, pos, S, sd)
            O.write_bits(ref_stream, pos + S, 4, e & 15)
            for j in range(k):
                O.write_bits(ref_stream, pos + S + 4 + 4 * j, 4, tt[j] & 15)
            pos += O.block_bits(S, k)
            ref_W[r, perm[8 * c:8 * c + 8]] = O.reconstruct_block(S, k, taps, sd, e, tt)
    assert pos == bits
    assert np.array_equal(buf.cpu().numpy(), ref_stream)

    layer.bind_stream(buf, bits, nbytes)
    Wout = torch.empty((R, Cc), dtype=torch.float32, device="cuda")
    layer.decode_weights(Wout)
    torch.cuda.synchronize()
    assert np.array_equal(Wout.cpu().numpy(), ref_W)
    assert layer.device_error() == 0
    layer.release()

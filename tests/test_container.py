"""Container file: the library's native reader/writer against the oracle's own.

CPU tests: both writers produce the same bytes for the same model, each reader
reads the other's file, and malformed files are rejected.  GPU test: layers
loaded from the stored golden container decode to the oracle's weights and
multiply to the oracle's outputs.
"""
import os
import struct
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
GOLDEN = os.path.join(ROOT, "tests", "golden")
sys.path.insert(0, ROOT)
sys.path.insert(0, os.path.join(ROOT, "oracle"))
sys.path.insert(0, GOLDEN)

import oracle as O  # noqa: E402
import make_container as MC  # noqa: E402

from paper_2609_38477_gb300 import build  # noqa: E402

GOLDEN_FILE = os.path.join(GOLDEN, "tiny_model.seedq")


@pytest.fixture(scope="module")
def Q():
    build.build()
    from paper_2609_38477_gb300 import seedq

    return seedq


def _same_tensor(x, y):
    assert x["name"] == y["name"] and x["rows"] == y["rows"] and x["cols"] == y["cols"]
    assert np.array_equal(x["a"], y["a"])
    assert (x["rho"] is None) == (y["rho"] is None)
    if x["rho"] is not None:
        assert np.array_equal(x["rho"], y["rho"])
    assert x["tie_count"] == y["tie_count"] and x["stream_bits"] == y["stream_bits"]
    assert np.array_equal(np.asarray(x["outlier_cols"], np.int32), np.asarray(y["outlier_cols"], np.int32))
    assert np.array_equal(np.asarray(x["outlier_vals"], np.uint16).reshape(x["rows"], -1),
                          np.asarray(y["outlier_vals"], np.uint16).reshape(y["rows"], -1))
    n = (x["stream_bits"] + 7) // 8
    assert np.array_equal(np.asarray(x["stream"])[:n], np.asarray(y["stream"])[:n])


def test_golden_matches_its_script(tmp_path):
    """The stored file is what the oracle-only script writes."""
    p = tmp_path / "again.seedq"
    O.write_container(str(p), MC.RUNGS, MC.THETA, MC.J_TIE, MC.Q_FLOOR, MC.model())
    assert p.read_bytes() == open(GOLDEN_FILE, "rb").read()


def test_library_reads_oracle_file(Q):
    ref = O.read_container(GOLDEN_FILE)
    c = Q.Container(GOLDEN_FILE)
    assert c.rungs == ref["rungs"] and c.theta == ref["theta"]
    assert c.j_tie == ref["j_tie"] and c.q == ref["q"] and c.count == len(ref["tensors"])
    for i, t in enumerate(ref["tensors"]):
        _same_tensor(c.tensor(i), t)
    c.close()


def test_library_writes_the_same_bytes(Q, tmp_path):
    p = tmp_path / "lib.seedq"
    Q.container_write(str(p), MC.RUNGS, MC.THETA, MC.J_TIE, MC.Q_FLOOR, MC.model())
    assert p.read_bytes() == open(GOLDEN_FILE, "rb").read()
    back = O.read_container(str(p))
    for t, u in zip(MC.model(), back["tensors"]):
        _same_tensor(t, u)


def test_malformed_files_are_rejected(Q, tmp_path):
    data = bytearray(open(GOLDEN_FILE, "rb").read())
    cases = {}
    flip = bytearray(data)
    flip[200] ^= 1
    cases["flipped"] = (bytes(flip), 8)
    cases["truncated"] = (bytes(data[:-20]), 8)
    cases["magic"] = (b"XEEDQ" + bytes(data[5:]), 8)
    # Other LFSR taps (hash recomputed so only the taps differ).
    body = bytearray(data[:-8])
    nrungs = struct.unpack_from("<I", body, 12)[0]
    taps_at = 16 + 8 * nrungs + 8 * (nrungs - 1) + 12
    struct.pack_into("<I", body, taps_at, 0x71)
    cases["taps"] = (bytes(body) + struct.pack("<Q", O._fnv1a(bytes(body))), 6)
    for name, (blob, status) in cases.items():
        p = tmp_path / f"{name}.seedq"
        p.write_bytes(blob)
        with pytest.raises(Q.SeedQError) as e:
            Q.Container(str(p))
        assert e.value.status == status, name
    with pytest.raises(Q.SeedQError) as e:
        Q.Container(str(tmp_path / "missing.seedq"))
    assert e.value.status == 7


@pytest.mark.gpu
def test_loaded_layers_decode_and_multiply(Q):
    torch = pytest.importorskip("torch")
    ref = O.read_container(GOLDEN_FILE)
    s = O.Sched(ref["rungs"], ref["theta"], ref["j_tie"], ref["q"])
    layers = Q.load_layers(GOLDEN_FILE, max_batch=4)
    assert [n for n, _ in layers] == [t["name"] for t in ref["tensors"]]
    for (name, L), t in zip(layers, ref["tensors"]):
        ot = O.Tensor(t["rows"], t["cols"], t["a"], t["rho"])
        Wo = ot.decode_rows(s, t["tie_count"], t["stream"], t["stream_bits"],
                            outlier_cols=t["outlier_cols"] if len(t["outlier_cols"]) else None,
                            outlier_vals=t["outlier_vals"] if len(t["outlier_cols"]) else None)
        Wg = torch.empty((t["rows"], t["cols"]), dtype=torch.float32, device="cuda")
        L.decode_weights(Wg)
        torch.cuda.synchronize()
        assert np.array_equal(Wg.cpu().numpy(), Wo), name
        rng = np.random.default_rng(3)
        xf = rng.normal(0, 1, (4, t["cols"])).astype(np.float32)
        xb = (xf.view(np.uint32) >> 16).astype(np.uint16)
        y64 = O.gemv_f64(Wo, xb)
        X = torch.from_numpy(xb.view(np.int16)).cuda()
        Y = torch.empty((4, t["rows"]), dtype=torch.float32, device="cuda")
        L.gemm_small_batch(X, 4, Y)
        torch.cuda.synchronize()
        xd = (xb.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        yabs = np.abs(Wo.astype(np.float64)) @ np.abs(xd).T
        err = np.abs(Y.cpu().numpy().astype(np.float64) - y64)
        assert np.all(err <= 1e-3 * yabs.T + 1e-30), name
        assert L.device_error() == 0
        L.release()

"""CPU checks of the C ABI library: it builds, loads, exports every symbol the
header declares, carries the stream format's LFSR taps, and rejects bad
arguments before touching a GPU."""
import ctypes as C
import os
import re

import numpy as np
import pytest

import oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def Q():
    from paper_2609_38477_gb300 import build

    build.build()
    from paper_2609_38477_gb300 import seedq

    seedq.lib()
    return seedq


def _declared_symbols():
    txt = open(os.path.join(ROOT, "include", "seedq.h")).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(seedq_[a-z_0-9]+)\s*\(", txt)))


def test_every_declared_symbol_is_exported(Q):
    names = _declared_symbols()
    assert len(names) >= 15
    L = C.CDLL(Q.LIB_PATH)
    for n in names:
        assert hasattr(L, n), n
    assert sorted(Q.SIGNATURES) == names


def test_lfsr_taps_agree_with_oracle_search(Q):
    """The library's tap table (format constant) equals the oracle's brute-force
    choice of primitive polynomials (reading R1) for every width."""
    for S in range(8, 17):
        assert Q.lfsr_taps(S) == O.find_taps(S)
    assert Q.lfsr_taps(7) == 0 and Q.lfsr_taps(17) == 0


def test_stream_bytes_required(Q):
    for bits in (1, 127, 128, 129, 10 ** 9 + 3):
        nb = Q.stream_bytes_required(bits)
        assert nb % 16 == 0 and nb >= (bits + 7) // 8 + 16


def _prepare(Q, **kw):
    base = dict(rows=4, cols=16, a=np.ones(16, np.float32), rho=None,
                rungs=[(8, 3), (16, 3)], theta=[1.0], j_tie=-1, q=0.0, tie_count=0)
    base.update(kw)
    return Q.Layer(base["rows"], base["cols"], base["a"], base["rho"], base["rungs"],
                   base["theta"], base["j_tie"], base["q"], base["tie_count"],
                   stream=0)


@pytest.mark.parametrize("kw,status", [
    (dict(cols=12), 1),                                        # C not a multiple of 8
    (dict(rows=0), 1),
    (dict(a=np.full(16, np.nan, np.float32)), 1),              # non-finite factor
    (dict(a=np.zeros(16, np.float32)), 1),                     # unit mean undefined
    (dict(rho=np.array([1, 0, 1, 1], np.float32)), 1),         # rho must be > 0
    (dict(rungs=[(9, 3), (16, 3)]), 6),                        # odd seed width
    (dict(rungs=[(8, 7), (16, 3)]), 6),                        # k outside 2..6
    (dict(rungs=[(16, 3), (8, 3)]), 3),                        # rates not increasing
    (dict(rungs=[(8, 3), (12, 3), (16, 3)], theta=[2.0, 1.0]), 3),  # theta not increasing
    (dict(j_tie=1), 3),                                        # j_tie out of range
    (dict(tie_count=-1), 3),
    (dict(cols=65544, a=np.ones(65544, np.float32)), 6),       # wider than supported
])
def test_prepare_rejects_bad_arguments_on_host(Q, kw, status):
    with pytest.raises(Q.SeedQError) as e:
        _prepare(Q, **kw)
    assert e.value.status == status


@pytest.mark.parametrize("factors,rungs,slopes,rbar,floor_f,status", [
    ([], [(8, 3), (16, 3)], [1.0], 4.0, 0.06, 1),                              # no tensors
    ([(4, 12, np.ones(12, np.float32), None)], [(8, 3), (16, 3)], [1.0], 4.0, 0.06, 1),
    ([(4, 16, np.zeros(16, np.float32), None)], [(8, 3), (16, 3)], [1.0], 4.0, 0.06, 1),
    ([(4, 16, np.ones(16, np.float32), np.array([1, 0, 1, 1], np.float32))],
     [(8, 3), (16, 3)], [1.0], 4.0, 0.06, 1),                                  # rho must be > 0
    ([(4, 16, np.ones(16, np.float32), None)], [(9, 3), (16, 3)], [1.0], 4.0, 0.06, 6),
    ([(4, 16, np.ones(16, np.float32), None)], [(16, 3), (8, 3)], [1.0], 4.0, 0.06, 3),
    ([(4, 16, np.ones(16, np.float32), None)], [(8, 3), (16, 3)], [-1.0], 4.0, 0.06, 3),
    ([(4, 16, np.ones(16, np.float32), None)], [(8, 3), (16, 3)], [1.0], 0.0, 0.06, 1),
    ([(4, 16, np.ones(16, np.float32), None)], [(8, 3), (16, 3)], [1.0], 4.0, 1.5, 1),
])
def test_allocate_rejects_bad_arguments_on_host(Q, factors, rungs, slopes, rbar, floor_f, status):
    """Alg. 1 on the device validates everything on the host before any CUDA call."""
    with pytest.raises(Q.SeedQError) as e:
        Q.allocate(factors, rungs, slopes, rbar, floor_f, stream=0)
    assert e.value.status == status


def _dims(**kw):
    d = dict(n_layers=1, d_model=64, n_heads=2, n_kv_heads=1, head_dim=32, d_ff=96, vocab=10)
    d.update(kw)
    return d


@pytest.mark.parametrize("kw", [dict(d_model=48), dict(d_ff=40), dict(n_heads=3, n_kv_heads=2),
                                dict(n_layers=0), dict(head_dim=20), dict(vocab=0)])
def test_importance_rejects_bad_shapes_on_host(Q, kw):
    """Shapes the column pass cannot tile (in-dimensions not multiples of 32,
    query heads not a multiple of the key-value heads) fail before any launch."""
    fake = 1 << 20  # 16-byte aligned, never dereferenced: validation comes first
    layer = {k: fake for k in ("attn_norm", "mlp_norm", "wq", "wk", "wv", "wo", "wgate", "wup", "wdown")}
    dims = _dims(**kw)
    out = {k: fake for k in ("a_o", "a_down", "rho_o", "rho_down")}
    with pytest.raises(Q.SeedQError) as e:
        Q.importance(dims, [layer] * max(dims["n_layers"], 1), fake, fake, out, stream=0)
    assert e.value.status == 1


def test_importance_rejects_missing_pointers_on_host(Q):
    fake = 1 << 20
    layer = {k: fake for k in ("attn_norm", "mlp_norm", "wq", "wk", "wv", "wo", "wgate", "wup", "wdown")}
    out = {k: fake for k in ("a_o", "a_down", "rho_o", "rho_down")}
    for missing in ("wv", "attn_norm"):
        bad = dict(layer)
        bad[missing] = 0
        with pytest.raises(Q.SeedQError) as e:
            Q.importance(_dims(), [bad], fake, fake, out, stream=0)
        assert e.value.status == 1
    misaligned = dict(layer, wq=fake + 2)
    with pytest.raises(Q.SeedQError) as e:
        Q.importance(_dims(), [misaligned], fake, fake, out, stream=0)
    assert e.value.status == 1
    with pytest.raises(Q.SeedQError) as e:
        Q.importance(_dims(), [layer], fake, fake, dict(out, a_o=0), stream=0)
    assert e.value.status == 1

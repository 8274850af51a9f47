"""Parity of the data-free importance, the outlier statistics and the device
allocator against the oracle (Sec. 3.2, 3.4, 3.5, App. A.1, A.5, A.8; Alg. 1).

Tolerances (float tables): every product W^2 g is rounded once in fp32 and
summed in fp32 over at most 16 rows (32 columns for the row sums) before the
fp64 sums, so each one-hop sum has relative error below ~40 u (u = 2^-24) of
its value (all terms are non-negative); the backward proxy composes two hops
per layer, and the float32 output adds u/2.  The tests use 2e-6 for the
one-hop quantities (a^(o), a^(down)) and 2e-6 (2L + 1) for rho after L layers.
The dynamic-range statistic, the activation ratio of exactly represented a
(gamma^2) and the allocator are exact, so those compare bit for bit.
"""
import json
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
sys.path.insert(0, os.path.join(ROOT, "oracle"))

import importance as I  # noqa: E402
import oracle as O  # noqa: E402
from paper_2609_38477_gb300 import workloads as W  # noqa: E402

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ONE_HOP = 2e-6


@pytest.fixture(scope="module")
def Q():
    from paper_2609_38477_gb300 import build

    build.build()
    from paper_2609_38477_gb300 import seedq

    return seedq


@pytest.fixture(scope="module")
def G():
    from paper_2609_38477_gb300 import workload_gpu

    return workload_gpu


def _f16_dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda()


def _rel(got, want):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    return np.max(np.abs(got - want) / np.maximum(np.abs(want), 1e-300))


def test_synth_fp16_matches_the_host_generator(Q):
    spec = W.MODELS["tiny"]
    key = W.weight_key(spec, 1, "up")
    n = 4099 * 8
    out = torch.empty(n, dtype=torch.int16, device="cuda")
    Q.synth_fp16(key, 0, n, W.W_SCALE_M, W.W_SCALE_E, out)
    R, C = spec.shape("up")
    host = W.synth_weight_rows(spec, 1, "up", 0, R).ravel()
    assert np.array_equal(out.cpu().numpy().view(np.uint16), host[:n])


@pytest.mark.parametrize("R,C,zeros", [(1, 32, 0.0), (65, 64, 0.0), (512, 96, 0.0), (777, 32, 0.0),
                                       (1000, 64, 0.6), (3000, 128, 0.3), (4096, 32, 0.0)])
def test_column_stats_against_oracle(Q, R, C, zeros):
    rng = np.random.default_rng(R * 7 + C)
    Wf = rng.normal(0, 0.02, (R, C)).astype(np.float32)
    Wf[rng.random((R, C)) < zeros] = 0.0
    # Spikes: a column with one huge weight, one with two, a subnormal column.
    if R > 4:
        Wf[R // 3, 0] = 60.0
        Wf[1, C - 1] = -45.0
        Wf[R // 2, C - 1] = 50.0
        Wf[:, 1] = 3e-7
        Wf[0, 1] = 0.5
    bits = Wf.astype(np.float16).view(np.uint16)
    g = rng.uniform(0.1, 3.0, R).astype(np.float32)
    dr = torch.empty(C, dtype=torch.float64, device="cuda")
    cs = torch.empty(C, dtype=torch.float64, device="cuda")
    Q.column_stats(_f16_dev(bits), R, C, dr, torch.from_numpy(g).cuda(), cs)
    torch.cuda.synchronize()
    want = I.dynamic_range(bits)
    got = dr.cpu().numpy()
    assert np.array_equal(got, np.where(want >= I.DR_MIN, want, 0.0))
    assert _rel(cs.cpu().numpy(), I.sq_cols(bits, g.astype(np.float64))) < ONE_HOP


def test_column_stats_unweighted_and_all_candidates(Q):
    """Median 0 in every column (mostly zero weights) sends every column down
    the exact-median path; the unweighted sums are plain sums of squares."""
    R, C = 333, 64
    rng = np.random.default_rng(11)
    Wf = np.zeros((R, C), np.float32)
    idx = rng.random((R, C)) < 0.3
    Wf[idx] = rng.normal(0, 1, idx.sum())
    bits = Wf.astype(np.float16).view(np.uint16)
    dr = torch.empty(C, dtype=torch.float64, device="cuda")
    cs = torch.empty(C, dtype=torch.float64, device="cuda")
    Q.column_stats(_f16_dev(bits), R, C, dr, None, cs)
    torch.cuda.synchronize()
    want = I.dynamic_range(bits)
    assert np.all(want >= I.DR_MIN)
    assert np.array_equal(dr.cpu().numpy(), want)
    assert _rel(cs.cpu().numpy(), I.sq_cols(bits, np.ones(R))) < ONE_HOP


def test_column_stats_rejects_bad_shapes(Q):
    x = torch.zeros(64 * 40, dtype=torch.int16, device="cuda")
    dr = torch.empty(64, dtype=torch.float64, device="cuda")
    for R, C in ((0, 32), (4, 40), (4, 16)):
        with pytest.raises(Q.SeedQError) as e:
            Q.column_stats(x, R, C, dr)
        assert e.value.status == 1


def _check_model(Q, G, name):
    spec = W.MODELS[name]
    m = W.SynthModel(spec)
    gm = G.synth_model_device(spec)
    # The device copy is the host model, bit for bit.
    for i, t in enumerate(gm.tensors()):
        assert np.array_equal(t.cpu().numpy().view(np.uint16), m.tensor(i)), i
    out = G.importance_buffers(spec)
    got_out = G.run_importance(gm, out)
    torch.cuda.synchronize()
    tables = I.importance_tables(m)
    L, d, f, qd = spec.n_layers, spec.d_model, spec.d_ff, spec.q_dim
    a_o = out["a_o"].cpu().numpy().reshape(L, qd)
    a_dn = out["a_down"].cpu().numpy().reshape(L, f)
    r_o = out["rho_o"].cpu().numpy().reshape(L, d)
    r_dn = out["rho_down"].cpu().numpy().reshape(L, d)
    for l in range(L):
        _, ao, ro = tables[7 * l + 3]
        _, ad, rd = tables[7 * l + 6]
        assert _rel(a_o[l], ao) < ONE_HOP, l
        assert _rel(a_dn[l], ad) < ONE_HOP, l
        tol = ONE_HOP * (2 * (L - l) + 1)
        assert _rel(r_o[l], ro) < tol, l
        assert _rel(r_dn[l], rd) < tol, l
    # Outlier statistics: exact dynamic range; exact activation ratio where a
    # is gamma^2, within one float32 step of a elsewhere.
    dr = out["dyn_range"].cpu().numpy()
    ar = out["act_ratio"].cpu().numpy()
    off = 0
    ratios = []
    for i, (tname, a, _) in enumerate(tables):
        Wt = m.tensor(i)
        C = Wt.shape[1]
        want = I.dynamic_range(Wt)
        assert np.array_equal(dr[off:off + C], np.where(want >= I.DR_MIN, want, 0.0)), tname
        r = I.activation_ratio(a)
        ratios.append(r)
        if tname.endswith((".o", ".down")):
            assert _rel(ar[off:off + C], r) < 4 * ONE_HOP, tname
            # No decision of the rule sits within the tolerance of its threshold.
            assert not np.any(np.abs(r / I.ACT_MIN - 1) < 1e-4), tname
        else:
            assert np.array_equal(ar[off:off + C], r), tname
        off += C
    assert got_out == I.model_outliers(m, tables)
    return spec, got_out


@pytest.mark.parametrize("name", ["tiny", "tiny_mha", "tiny_odd"])
def test_importance_small_models_against_oracle(Q, G, name):
    spec, got = _check_model(Q, G, name)
    names = spec.tensor_names()
    for (l, k, r, c, _) in W.super_weights(spec):
        assert (names.index(f"l{l}.{k}"), c) in got


@pytest.mark.parametrize("name", ["llama2_7b", "llama3_8b"])
def test_importance_full_shape_sampled(Q, G, name):
    """Full Llama-shaped checkpoints in the launch configuration of the
    benchmark (Llama-3-8B: 4 query heads per value head); outputs checked on
    samples the oracle computes one by one."""
    spec = W.MODELS[name]
    gm = G.synth_model_device(spec)
    out = G.importance_buffers(spec)
    got = G.run_importance(gm, out)
    torch.cuda.synchronize()
    L, d, f, qd = spec.n_layers, spec.d_model, spec.d_ff, spec.q_dim
    a_o = out["a_o"].cpu().numpy().reshape(L, qd)
    a_dn = out["a_down"].cpu().numpy().reshape(L, f)
    r_dn = out["rho_down"].cpu().numpy().reshape(L, d)
    rng = np.random.default_rng(5)
    for l in (0, 1, L - 1):
        a_attn = I.a_from_gain(W.synth_gain(spec, l, "attn"))
        a_mlp = I.a_from_gain(W.synth_gain(spec, l, "mlp"))
        for i in rng.integers(0, qd, 6):
            h, o = divmod(int(i), spec.head_dim)
            row = (h // (spec.n_heads // spec.n_kv_heads)) * spec.head_dim + o
            Wv = W.synth_weight_rows(spec, l, "v", row, 1)
            assert _rel(a_o[l, i], I.sq_rows(Wv, a_attn)[0]) < ONE_HOP
        for c in rng.integers(0, f, 6):
            g2 = I.sq_rows(W.synth_weight_rows(spec, l, "gate", int(c), 1), a_mlp)
            u = I.sq_rows(W.synth_weight_rows(spec, l, "up", int(c), 1), a_mlp)
            assert _rel(a_dn[l, c], I.silu_sq_moment(g2)[0] * u[0]) < ONE_HOP
    # rho of the last down projection: the head's column sums of squares
    # (checked on the smaller head; the 128k-row one takes minutes on the host).
    if spec.vocab <= 64000:
        head = np.zeros(d)
        R = spec.vocab
        for r0 in range(0, R, 4000):
            head += I.sq_cols(W.synth_weight_rows(spec, None, "lm_head", r0, min(4000, R - r0)),
                              np.ones(min(4000, R - r0)))
        assert _rel(r_dn[L - 1], I.unit_mean(head)) < 2 * ONE_HOP
    # Planted super weights: exact statistic and selected.
    names = spec.tensor_names()
    dr = out["dyn_range"].cpu().numpy()
    offs = np.cumsum([0] + [spec.shape(n.split(".")[-1] if n != "lm_head" else "lm_head")[1]
                            for n in names])
    for (l, k, r, c, _) in W.super_weights(spec):
        t = names.index(f"l{l}.{k}")
        Wt = W.synth_weight_rows(spec, l, k, 0, spec.shape(k)[0])
        want = I.dynamic_range(Wt[:, [c]])[0]
        assert want >= I.DR_MIN and dr[offs[t] + c] == want
        assert (t, c) in got
    assert np.all(np.isfinite(a_o)) and np.all(a_o > 0)
    assert np.all(np.isfinite(r_dn)) and np.all(r_dn > 0)


# ---------------------------------------------------------------- allocator

def _factors(w):
    out = []
    for i, t in enumerate(w.tensors):
        a, rho = W.importance(w, i)
        out.append((t.R, t.C, a, rho))
    return out


@pytest.mark.parametrize("name", ["c0", "c1", "c2", "c3", "c4", "c4_3"])
def test_allocator_reproduces_stored_schedules(Q, name):
    """The stored schedules were written by the oracle's allocator; the device
    allocator reproduces every field exactly."""
    d = json.load(open(os.path.join(ROOT, "tests", "golden", f"schedule_{name}.json")))
    w = W.WORKLOADS[name]
    theta, jt, q, T, bits = Q.allocate(_factors(w), [tuple(r) for r in d["rungs"]], d["slopes"],
                                       d["rbar"], d["floor_f"])
    assert list(theta) == d["theta"]
    assert jt == d["j_tie"] and q == d["q"]
    assert [int(x) for x in T] == d["tie_count"]
    assert [int(x) for x in bits] == d["stream_bits"]


@pytest.mark.parametrize("trial", range(6))
def test_allocator_matches_oracle_random(Q, trial):
    rng = np.random.default_rng(100 + trial)
    rungs, _, slopes = O.hull_rungs(W.DAMAGE_TABLES["llama2_7b"](), 4.0)
    fs = []
    for t in range(1 + trial % 3):
        R, Cc = int(rng.integers(1, 90)), 8 * int(rng.integers(1, 40))
        a = np.exp(rng.normal(0, 1, Cc)).astype(np.float32)
        a[rng.integers(0, Cc, 3)] = a[0]  # ties in a
        rho = np.exp(rng.normal(0, 0.5, R)).astype(np.float32) if (trial + t) % 2 else None
        fs.append((R, Cc, a, rho))
    rbar = 3.7 + 0.1 * trial
    floor_f = [0.0, 0.06, 0.3][trial % 3]
    ts = [O.Tensor(R, Cc, a, rho) for R, Cc, a, rho in fs]
    try:
        s, T, bits = O.allocate(ts, rungs, slopes, rbar, floor_f)
    except RuntimeError:
        with pytest.raises(Q.SeedQError) as e:
            Q.allocate(fs, rungs, slopes, rbar, floor_f)
        assert e.value.status == 3
        return
    got = Q.allocate(fs, rungs, slopes, rbar, floor_f)
    assert list(got[0]) == list(s.theta) and got[1] == s.j_tie and got[2] == s.q
    assert list(got[3]) == list(T) and list(got[4]) == list(bits)


def test_allocator_errors(Q):
    rungs, _, slopes = O.hull_rungs(W.DAMAGE_TABLES["llama2_7b"](), 4.0)
    fs = [(16, 64, np.ones(64, np.float32), None)]
    with pytest.raises(Q.SeedQError) as e:  # below the lowest rung's rate
        Q.allocate(fs, rungs, slopes, 1.0, 0.06)
    assert e.value.status == 3
    theta, jt, q, T, bits = Q.allocate(fs, rungs, slopes, 10.0, 0.06)  # above the top rung
    L = [O.block_bits(S, k) for S, k in rungs]
    assert jt == -1 and list(T) == [0] and int(bits[0]) == 16 * 8 * L[-1]
    with pytest.raises(Q.SeedQError) as e:
        Q.allocate([(16, 60, np.ones(60, np.float32), None)], rungs, slopes, 4.0, 0.06)
    assert e.value.status == 1

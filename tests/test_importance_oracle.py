"""Pins of the importance / outlier oracle (Sec. 3.2, 3.5, App. A.1, A.8)
against facts that do not come from the oracle itself: an adaptive quadrature
of the same integral, second moments estimated by sampling the random vectors
the propagation describes, a hand-derived closed form of the backward proxy on
diagonal networks, numpy's median, and hand-built ranking cases."""
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
sys.path.insert(0, os.path.join(ROOT, "oracle"))

import importance as I  # noqa: E402
from paper_2609_38477_gb300 import workloads as W  # noqa: E402


def f16bits(x):
    return np.asarray(x, np.float32).astype(np.float16).view(np.uint16)


# ----------------------------------------------------------- E[silu(g)^2]

@pytest.mark.parametrize("var", [1e-4, 0.01, 0.3, 1.0, 4.0])
def test_silu_moment_against_adaptive_quadrature(var):
    integrate = pytest.importorskip("scipy.integrate")
    s = np.sqrt(var)
    dens = lambda g: (g / (1 + np.exp(-g))) ** 2 * np.exp(-g * g / (2 * var)) / np.sqrt(2 * np.pi * var)
    ref, _ = integrate.quad(dens, -40 * s, 40 * s, limit=400, epsabs=0, epsrel=1e-13)
    assert I.silu_sq_moment(var) == pytest.approx(ref, rel=1e-8)


def test_silu_moment_limits():
    # silu(x) = x/2 + O(x^2) near 0, so E ~ var/4 for small var; for large var
    # silu(x)^2 ~ x^2 on x > 0 and ~0 on x < 0, so E ~ var/2.
    assert I.silu_sq_moment(1e-8) / 1e-8 == pytest.approx(0.25, rel=1e-6)
    assert 0.45 < I.silu_sq_moment(100.0) / 100.0 < 0.55
    assert I.silu_sq_moment(0.0) == 0.0


# -------------------------------------------------- Eq. prop by sampling

def _sampled_second_moment(M, var, n=200_000, seed=0):
    rng = np.random.default_rng(seed)
    X = rng.normal(0, 1, (n, var.size)) * np.sqrt(var)
    return ((X @ M.T) ** 2).mean(axis=0)


def test_sq_rows_is_the_forward_second_moment():
    rng = np.random.default_rng(1)
    Wb = f16bits(rng.normal(0, 0.3, (12, 20)))
    a = rng.uniform(0.2, 3.0, 20)
    emp = _sampled_second_moment(I.f16(Wb), a)
    assert np.allclose(I.sq_rows(Wb, a), emp, rtol=0.03)


def test_sq_cols_is_the_backward_second_moment():
    rng = np.random.default_rng(2)
    Wb = f16bits(rng.normal(0, 0.3, (20, 12)))
    g = rng.uniform(0.2, 3.0, 20)
    emp = _sampled_second_moment(I.f16(Wb).T, g)
    assert np.allclose(I.sq_cols(Wb, g), emp, rtol=0.03)


def test_a_o_follows_the_value_path_with_shared_heads():
    """One attended position per head: query head h outputs the value vector of
    key-value head h * n_kv / n_heads, so a^(o) is the second moment of that."""
    rng = np.random.default_rng(3)
    n_heads, n_kv, hd, d = 4, 2, 3, 10
    Wb = f16bits(rng.normal(0, 0.4, (n_kv * hd, d)))
    a = rng.uniform(0.5, 2.0, d)
    X = rng.normal(0, 1, (200_000, d)) * np.sqrt(a)
    V = X @ I.f16(Wb).T
    O = np.concatenate([V[:, (h * n_kv // n_heads) * hd:(h * n_kv // n_heads + 1) * hd]
                        for h in range(n_heads)], axis=1)
    assert np.allclose(I.a_o(Wb, a, n_heads, n_kv), (O ** 2).mean(axis=0), rtol=0.03)


def test_a_down_factorises_for_independent_branches():
    """Gate and up reading disjoint channels makes g_c and u_c independent, so
    E[(silu(g_c) u_c)^2] = E[silu(g_c)^2] E[u_c^2] holds exactly."""
    rng = np.random.default_rng(4)
    d, f = 12, 5
    Wg = np.zeros((f, d)); Wu = np.zeros((f, d))
    Wg[:, : d // 2] = rng.normal(0, 0.5, (f, d // 2))
    Wu[:, d // 2:] = rng.normal(0, 0.5, (f, d // 2))
    Wgb, Wub = f16bits(Wg), f16bits(Wu)
    a = rng.uniform(0.5, 2.0, d)
    X = rng.normal(0, 1, (400_000, d)) * np.sqrt(a)
    G = X @ I.f16(Wgb).T
    U = X @ I.f16(Wub).T
    emp = ((G / (1 + np.exp(-G)) * U) ** 2).mean(axis=0)
    assert np.allclose(I.a_down(Wgb, Wub, a), emp, rtol=0.03)


# --------------------------------------- backward proxy: closed form

class _Spec:
    def __init__(self, L, d, n_heads, n_kv, hd, f, V):
        self.n_layers, self.d_model, self.n_heads, self.n_kv_heads = L, d, n_heads, n_kv
        self.head_dim, self.d_ff, self.vocab = hd, f, V


class _DiagModel:
    """Every matrix diagonal (or a 0/1 selection), so the proxy has a closed form."""

    def __init__(self, spec, diag, lm):
        self.spec, self.diag, self.lm = spec, diag, lm

    def weight(self, l, kind):
        return self.diag[(l, kind)]

    def lm_head(self):
        return self.lm


def test_rho_proxy_closed_form_two_diagonal_layers():
    d = 6
    spec = _Spec(2, d, 2, 2, 3, d, d)
    rng = np.random.default_rng(5)
    vals = {}
    diag = {}
    for l in range(2):
        for k in ("o", "v", "gate", "up", "down"):
            v = rng.choice([0.25, 0.5, 1.0, 2.0, 3.0], d)
            vals[(l, k)] = v
            diag[(l, k)] = f16bits(np.diag(v))
    s_lm = rng.choice([0.5, 1.0, 2.0], d)
    out = I.rho_proxy(_DiagModel(spec, diag, f16bits(np.diag(s_lm))))
    # Hand derivation: the head gives s_lm^2; each layer, last first: rho_down
    # is the stream scale, the MLP adds (s_gate^2 + s_up^2) s_down^2 of it,
    # rho_o is the new scale, attention adds s_v^2 s_o^2 of that.
    G = s_lm ** 2
    exp = {}
    for l in (1, 0):
        v = lambda k: vals[(l, k)] ** 2
        rd = G.copy()
        G = G * (1 + (v("gate") + v("up")) * v("down"))
        ro = G.copy()
        G = G * (1 + v("v") * v("o"))
        exp[l] = (ro, rd)
    for l in (0, 1):
        assert np.allclose(out[l][0], exp[l][0], rtol=1e-14)
        assert np.allclose(out[l][1], exp[l][1], rtol=1e-14)


def test_rho_proxy_sums_query_heads_sharing_a_value_head():
    n_heads, n_kv, hd = 4, 2, 2
    d = n_heads * hd
    spec = _Spec(1, d, n_heads, n_kv, hd, d, d)
    eye = f16bits(np.eye(d))
    zero = f16bits(np.zeros((d, d)))
    Wv = np.zeros((n_kv * hd, d))
    Wv[np.arange(n_kv * hd), np.arange(n_kv * hd)] = 1.0  # value channel j reads stream channel j
    diag = {(0, "o"): eye, (0, "v"): f16bits(Wv), (0, "gate"): zero, (0, "up"): zero,
            (0, "down"): zero}
    s_lm = np.arange(1, d + 1, dtype=np.float64) / 4
    (ro, rd), = I.rho_proxy(_DiagModel(spec, diag, f16bits(np.diag(s_lm))))
    G = s_lm ** 2
    assert np.array_equal(rd, G) and np.array_equal(ro, G)
    # Value channel (j, i) collects the query heads j*2 and j*2+1 at offset i.
    heads = G.reshape(n_heads, hd)
    gv = np.stack([heads[2 * j] + heads[2 * j + 1] for j in range(n_kv)]).ravel()
    # Nothing after this layer reads the stream, so check through a second call
    # with one more (identity) layer in front: its rho is the stream scale.
    spec2 = _Spec(2, d, n_heads, n_kv, hd, d, d)
    diag2 = dict(diag)
    for k in ("o", "v", "gate", "up", "down"):
        diag2[(1, k)] = diag[(0, k)]
        diag2[(0, k)] = zero
    diag2[(0, "v")] = f16bits(np.zeros((n_kv * hd, d)))
    out = I.rho_proxy(_DiagModel(spec2, diag2, f16bits(np.diag(s_lm))))
    after = G.copy()
    after[: n_kv * hd] += gv
    assert np.array_equal(out[0][1], after)


def test_stored_rho_is_the_proxy_at_unit_mean():
    m = W.SynthModel(W.MODELS["tiny"])
    raw = I.rho_proxy(m)
    tables = I.importance_tables(m)
    for l, (ro, rd) in enumerate(raw):
        for got, want in ((tables[7 * l + 3][2], ro), (tables[7 * l + 6][2], rd)):
            assert got.dtype == np.float32
            assert np.allclose(got, want / want.mean(), rtol=1e-6)
            assert abs(float(np.mean(got.astype(np.float64))) - 1.0) < 1e-6


@pytest.mark.parametrize("name", ["tiny", "tiny_mha", "tiny_odd"])
def test_importance_tables_wiring(name):
    """Each tensor's entry carries the factors of its own inputs: q, k, v read
    the attention norm's gain, gate and up the MLP norm's, the head the final
    norm's (Eq. gamma, squared gains decoded here from the FP16 bits without
    numpy); o takes the second moment of W_v's outputs repeated over the query
    heads and down the gate/up propagation of the MLP gain (Eq. prop, the
    formulas pinned above by sampling); only o and down carry rho."""
    import struct

    m = W.SynthModel(W.MODELS[name])
    s = m.spec
    tables = I.importance_tables(m)
    assert len(tables) == 7 * s.n_layers + 1

    def sq_gain(bits):
        vals = struct.unpack("<%de" % len(bits), np.asarray(bits, np.uint16).tobytes())
        return np.array([v * v for v in vals], np.float64)

    for l in range(s.n_layers):
        ga, gm = sq_gain(m.gain(l, "attn")), sq_gain(m.gain(l, "mlp"))
        names = [t[0] for t in tables[7 * l: 7 * l + 7]]
        assert names == [f"l{l}.{k}" for k in I.KINDS]
        for j in (0, 1, 2):
            assert np.array_equal(tables[7 * l + j][1], ga.astype(np.float32)), (l, j)
        for j in (4, 5):
            assert np.array_equal(tables[7 * l + j][1], gm.astype(np.float32)), (l, j)
        Wv = I.f16(m.weight(l, "v"))
        vo = (Wv * Wv) @ ga
        hd = s.head_dim
        rep = s.n_heads // s.n_kv_heads
        ao = np.concatenate([vo[(h // rep) * hd:(h // rep + 1) * hd] for h in range(s.n_heads)])
        assert np.allclose(tables[7 * l + 3][1], ao, rtol=1e-6)
        Wg, Wu = I.f16(m.weight(l, "gate")), I.f16(m.weight(l, "up"))
        ad = I.silu_sq_moment((Wg * Wg) @ gm) * ((Wu * Wu) @ gm)
        assert np.allclose(tables[7 * l + 6][1], ad, rtol=1e-6)
        for j in (0, 1, 2, 4, 5):
            assert tables[7 * l + j][2] is None
        assert tables[7 * l + 3][2] is not None and tables[7 * l + 6][2] is not None
    name, a_head, rho_head = tables[-1]
    assert name == "lm_head" and rho_head is None
    assert np.array_equal(a_head, sq_gain(m.gain(None, "final")).astype(np.float32))


# ------------------------------------------------------- outlier rules

@pytest.mark.parametrize("R", [7, 8])
def test_column_median_matches_numpy(R):
    rng = np.random.default_rng(6 + R)
    Wb = f16bits(rng.normal(0, 1, (R, 9)))
    mx, med = I.column_max_median(Wb)
    A = np.abs(I.f16(Wb))
    assert np.array_equal(med, np.median(A, axis=0))
    assert np.array_equal(mx, A.max(axis=0))
    assert np.array_equal(I.dynamic_range(Wb), A.max(axis=0) / (np.median(A, axis=0) + 2.0 ** -24))


def test_merge_ranks_by_better_position_then_tensor_then_column():
    big = 5e3
    dr = [np.array([0.0, big + 2, 0.0]), np.array([big, 0.0, big + 1])]
    ratio = [np.array([150.0, 0.0, 0.0]), np.array([0.0, 400.0, 150.0])]
    # dynamic-range list: (0,1) (1,2) (1,0); activation list: (1,1) (0,0) (1,2)
    got = I.select_outliers(dr, ratio, n_keep=10)
    assert got == [(0, 1), (1, 1), (0, 0), (1, 2), (1, 0)]
    assert I.select_outliers(dr, ratio) == got[:4]


def test_thresholds_are_inclusive_and_lists_capped_at_32():
    dr = [np.full(40, I.DR_MIN), np.array([I.DR_MIN * (1 - 1e-12)])]
    ratio = [np.zeros(40), np.zeros(1)]
    got = I.select_outliers(dr, ratio, n_keep=100)
    # All 40 columns qualify (>=) and tie; the first 32 by column are kept.
    assert got == [(0, c) for c in range(32)]


def test_activation_mean_is_the_correctly_rounded_sum():
    from fractions import Fraction

    a = np.array([2.0 ** 53, 1.0, 1.0, 1.0], np.float32)
    # Exact sum 2^53 + 3 lies halfway between two doubles and rounds to even,
    # 2^53 + 4; summing in column order would give 2^53.
    exact = sum(Fraction(float(x)) for x in a)
    assert float(exact) == 2.0 ** 53 + 4
    assert I.activation_ratio(a)[1] == 1.0 / ((2.0 ** 53 + 4) / 4)
    rng = np.random.default_rng(9)
    b = np.exp(rng.normal(0, 6, 1000)).astype(np.float32)
    mean = float(sum(Fraction(float(x)) for x in b)) / b.size
    assert np.array_equal(I.activation_ratio(b), b.astype(np.float64) / mean)


def test_tiny_model_recovers_planted_super_weights_and_massive_channel():
    m = W.SynthModel(W.MODELS["tiny"])
    spec = m.spec
    names = spec.tensor_names()
    got = I.model_outliers(m)
    down = names.index("l1.down")
    for (l, k, r, c, _) in W.super_weights(spec):
        assert (names.index(f"l{l}.{k}"), c) in got
    mc = int(W.massive_channels(spec)[0])
    assert any(c == mc and names[t].startswith("l1.") for t, c in got if t != down)

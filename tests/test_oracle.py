"""Pins of the CPU oracle against what the paper and mathematics fix.

Each test checks the oracle against something other than itself: values the
paper prints, hand-worked examples, closed forms, textbook algorithms (GF(2)
primitivity, brute-force hulls and allocations) or a library routine.
"""
import itertools
import json
import os

import numpy as np
import pytest

import oracle as O
from paper_2609_38477_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _table_grids():
    rows = []
    for line in open(os.path.join(GOLDEN, "table_grids.txt")):
        if line.startswith("#") or not line.strip():
            continue
        S, k, rate, e2, e3 = line.split()
        rows.append((int(S), int(k), float(rate), e2, e3))
    return rows


# ------------------------------------------------------------------ Eq. rate

def test_rate_matches_table_grids():
    """Eq. rate with m = e = 4 reproduces every rate entry of the rung-grid table (App. B.3)."""
    for S, k, rate, _, _ in _table_grids():
        assert O.block_bits(S, k) / 8.0 == rate


def test_seedlm_point_is_32_bits():
    """Sec. 3.1: SeedLM's 4-bit point is (16,3) with m = e = 4."""
    assert O.block_bits(16, 3) == 32


# --------------------------------------------------------------------- LFSR

def _gf2_mulmod(a, b, p, deg):
    r = 0
    while b:
        if b & 1:
            r ^= a
        b >>= 1
        a <<= 1
        if (a >> deg) & 1:
            a ^= p
    return r


def _gf2_powmod(base, e, p, deg):
    r, b = 1, base
    while e:
        if e & 1:
            r = _gf2_mulmod(r, b, p, deg)
        b = _gf2_mulmod(b, b, p, deg)
        e >>= 1
    return r


def _prime_factors(n):
    out, d = [], 2
    while d * d <= n:
        while n % d == 0:
            if d not in out:
                out.append(d)
            n //= d
        d += 1
    if n > 1:
        out.append(n)
    return out


@pytest.mark.parametrize("S", range(8, 17))
def test_taps_primitive_by_gf2_order(S):
    """Maximal length (Sec. 3.1) <=> the characteristic polynomial is primitive:
    x has multiplicative order 2^S - 1 modulo p(x) (textbook test in GF(2)[x])."""
    taps = O.find_taps(S)
    p = (1 << S) | taps
    n = (1 << S) - 1
    assert _gf2_powmod(2, n, p, S) == 1
    for q in _prime_factors(n):
        assert _gf2_powmod(2, n // q, p, S) != 1


@pytest.mark.parametrize("S", [8, 11, 16])
def test_sequence_period(S):
    """Sec. 3.1 searches every nonzero seed, 2^S - 1 of them: the output bit sequence repeats with
    period exactly 2^S - 1 and no smaller divisor."""
    taps = O.find_taps(S)
    n = (1 << S) - 1
    o = O.lfsr_bits(S, taps, 0x5A5A & n or 1, 2 * n + S)
    assert np.array_equal(o[:n + S], o[n:2 * n + S])
    for q in _prime_factors(n):
        d = n // q
        assert not np.array_equal(o[:n], o[d:d + n])


def test_taps_minimal_largest_tap():
    """Reading R1: no primitive polynomial has a smaller largest tap below S.
    Checked by the GF(2) order test over every candidate with a smaller tap."""
    for S in range(8, 17):
        m = max(i for i in range(S) if (O.find_taps(S) >> i) & 1)
        n = (1 << S) - 1
        for mm in range(1, m):
            for mid in range(1 << max(mm - 1, 0)):
                taps = 1 | (1 << mm) | (mid << 1)
                p = (1 << S) | taps
                prim = _gf2_powmod(2, n, p, S) == 1 and all(
                    _gf2_powmod(2, n // q, p, S) != 1 for q in _prime_factors(n))
                assert not prim, (S, hex(taps))


def _fixture(name):
    out = {}
    for line in open(os.path.join(GOLDEN, name)):
        if line.startswith("#") or not line.strip():
            continue
        key, *vals = line.split()
        out[key] = vals
    return out


def test_hand_worked_s8_sequence():
    fx = _fixture("lfsr_s8_seed1.txt")
    taps = O.find_taps(8)
    assert taps == 0b11101  # x^8 + x^4 + x^3 + x^2 + 1
    bits = [int(v) for v in fx["bits"]]
    assert list(O.lfsr_bits(8, taps, 1, len(bits))) == bits
    states = [int(v) for v in fx["states"]]
    o = O.lfsr_bits(8, taps, 1, 40)
    got = [int(sum(int(o[n + i]) << i for i in range(8))) for n in range(len(states))]
    assert got == states
    w = O.reconstruct_block(8, 3, taps, 1, 0, [1, 0, 0])
    assert [float(v) for v in w] == [float(v) for v in fx["weights"]]


def test_window_identity():
    """x_{n+1} = (x_n >> 1) | (o_{n+S} << (S-1)) for the window states."""
    for S in (9, 14, 16):
        taps = O.find_taps(S)
        o = O.lfsr_bits(S, taps, 12345 % ((1 << S) - 1) + 1, 80)
        x = [sum(int(o[n + i]) << i for i in range(S)) for n in range(60)]
        for n in range(59):
            assert x[n + 1] == (x[n] >> 1) | (int(o[n + S]) << (S - 1))


# -------------------------------------------------------------- Eq. codec

def _states(S, taps, seed, count):
    o = O.lfsr_bits(S, taps, seed, S + count)
    return [sum(int(o[n + i]) << i for i in range(S)) for n in range(count)]


def test_codec_matches_matrix_form():
    """Eq. codec w = U(s) t_hat with U in [-1,1]^{8 x k} filled row-major from
    consecutive states and t_hat = t 2^E, checked against numpy's matmul."""
    rng = np.random.default_rng(3)
    for S in (8, 10, 12, 14, 16):
        taps = O.find_taps(S)
        for k in (2, 3, 4, 5, 6):
            seed = int(rng.integers(1, 1 << S))
            t = [int(v) for v in rng.integers(-8, 8, k)]
            E = int(rng.integers(-8, 8))
            x = np.array(_states(S, taps, seed, 8 * k), np.float64).reshape(8, k)
            U = (x - 2 ** (S - 1)) / 2 ** (S - 1)
            assert U.min() >= -1 and U.max() <= 1
            ref = U @ (np.array(t, np.float64) * 2.0 ** E)
            got = O.reconstruct_block(S, k, taps, seed, E, t)
            assert np.array_equal(got.astype(np.float64), ref)


def test_exactness_invariant():
    """|I_i| < 2^21 and E - S + 1 in [-23, 0]: every reconstructed weight is an
    exact fp32 value, so bit-exact parity is well posed."""
    rng = np.random.default_rng(4)
    for S in (8, 16):
        taps = O.find_taps(S)
        for k in (2, 6):
            for _ in range(50):
                seed = int(rng.integers(1, 1 << S))
                t = [-8] * k if _ % 2 else [int(v) for v in rng.integers(-8, 8, k)]
                E = int(rng.integers(-8, 8))
                x = np.array(_states(S, taps, seed, 8 * k), np.float64).reshape(8, k)
                exact = ((x - 2 ** (S - 1)) @ np.array(t, np.float64)) * 2.0 ** (E - S + 1)
                assert np.array_equal(exact.astype(np.float32).astype(np.float64), exact)


def test_seed_zero_is_all_minus_one():
    """Reading R12: seed 0 gives the all-zero sequence, U = -1 everywhere, so
    w_i = -2^E sum_j t_j (closed form)."""
    for S, k in ((8, 3), (16, 6)):
        t = [3, -2, 7, 1, -8, 5][:k]
        w = O.reconstruct_block(S, k, O.find_taps(S), 0, -2, t)
        assert np.all(w == np.float32(-(2.0 ** -2) * sum(t)))


def test_bit_io_round_trip():
    rng = np.random.default_rng(5)
    buf = np.zeros(64, np.uint8)
    vals = []
    pos = 0
    for _ in range(40):
        n = int(rng.integers(1, 17))
        v = int(rng.integers(0, 1 << n))
        O.write_bits(buf, pos, n, v)
        vals.append((pos, n, v))
        pos += n
    for p, n, v in vals:
        assert O.read_bits(buf, p, n) == v
    # LSB-first little-endian layout: bit p lives in byte p >> 3 at bit p & 7.
    buf2 = np.zeros(4, np.uint8)
    O.write_bits(buf2, 3, 6, 0b101101)
    assert int(buf2[0]) == (0b01101 << 3) and int(buf2[1]) == 0b1


# ------------------------------------------------------------- splitmix64

def test_splitmix64_known_answer_and_second_implementation():
    """splitmix64's first output from state 0 is 0xE220A8397B1DCDAF (published
    reference value); the C oracle and the numpy input generator, written
    separately from the published definition, agree."""
    assert O.splitmix64_at(0, 0) == 0xE220A8397B1DCDAF
    for key in (0, 1, 0xDEADBEEF12345678):
        for i in (0, 1, 2, 1000, 2 ** 40):
            assert O.splitmix64_at(key, i) == W.splitmix64_at(key, i)
    idx = np.arange(100, dtype=np.uint64)
    assert all(int(a) == O.splitmix64_at(77, int(i)) for i, a in zip(idx, W.splitmix64_at(77, idx)))


def test_synthetic_field_ranges():
    """Workload recipe: seeds uniform over nonzero states, t uniform int4,
    E uniform in [-8, -3]."""
    Es, ts = set(), set()
    for b in range(3000):
        for S, k in ((8, 2), (16, 6)):
            seed, E, t = O.synth_fields(1234, b, S, k)
            assert 1 <= seed <= (1 << S) - 1
            Es.add(E)
            ts.update(t)
    assert Es == set(range(-8, -2))
    assert ts == set(range(-8, 8))


# ------------------------------------------------------------------- hull

def _hull_brute(points):
    """Lower-hull membership by definition: point i is kept iff it has the
    lowest e at its rate and no segment between a point left of it and a point
    right of it passes on or below it; rising tails dropped."""
    best = {}
    for i, (S, k, e) in enumerate(points):
        r = O.block_bits(S, k)
        if r not in best or e < points[best[r]][2]:
            best[r] = i
    cand = sorted(best.values(), key=lambda i: O.block_bits(*points[i][:2]))
    keep = []
    for i in cand:
        xi, yi = O.block_bits(*points[i][:2]) / 8, points[i][2]
        ok = True
        for a in cand:
            for b in cand:
                xa, ya = O.block_bits(*points[a][:2]) / 8, points[a][2]
                xb, yb = O.block_bits(*points[b][:2]) / 8, points[b][2]
                if xa < xi < xb:
                    yl = ya + (yb - ya) * (xi - xa) / (xb - xa)
                    if yl <= yi + 1e-15:
                        ok = False
        if ok:
            keep.append(i)
    while len(keep) >= 2 and points[keep[-1]][2] >= points[keep[-2]][2]:
        keep.pop()
    return keep


def test_hull_llama2_7b_worked_example():
    """Lower convex hull of the Llama-2-7B column of the rung-grid table: eight
    rungs with decreasing slopes (Sec. 3.4; App. B.3 reports hulls of four to
    eight rungs)."""
    d = W.DAMAGE_LLAMA2_7B
    rungs, es, slopes = O.hull_rungs(d, 4.0)
    assert rungs == [(8, 3), (10, 3), (12, 3), (14, 3), (16, 3), (14, 4), (16, 5), (16, 6)]
    assert np.allclose(slopes, [5.1576, 1.4412, 0.4268, 0.2052, 0.0912, 0.041333333, 0.0134])
    assert all(a > b for a, b in zip(slopes, slopes[1:]))
    pts = [(S, k, e) for (S, k), e in sorted(d.items())]
    assert O.hull(pts) == _hull_brute(pts)


def test_hull_llama3_8b_worked_example():
    d = W.DAMAGE_LLAMA3_8B
    rungs, _, slopes = O.hull_rungs(d, 4.0)
    assert rungs == [(10, 3), (12, 3), (14, 3), (16, 3), (14, 4), (16, 5)]
    assert all(a > b for a, b in zip(slopes, slopes[1:]))


def test_hull_random_brute_force():
    rng = np.random.default_rng(6)
    grid = [(S, k) for S in range(8, 17, 2) for k in range(2, 7)]
    for _ in range(200):
        sel = rng.choice(len(grid), size=8, replace=False)
        pts = [(grid[i][0], grid[i][1], float(rng.uniform(0.01, 3.0))) for i in sel]
        assert O.hull(pts) == _hull_brute(pts)


def test_band_filter_synthetic_hull():
    """App. A.5 band: rungs within 1.0 below and 1.5 above the target rate.  The
    synthetic sub-4-bit hull (reading R11) loses (16,5) and (16,6) at 3.0."""
    full = O.hull([(S, k, e) for (S, k), e in sorted(W.damage_synthetic_k2().items())])
    assert len(full) == 9
    rungs, _, _ = O.hull_rungs(W.damage_synthetic_k2(), 3.0)
    assert rungs == [(8, 2), (10, 2), (12, 2), (14, 2), (16, 2), (16, 3), (14, 4)]


# ---------------------------------------------------------------- schedule

def test_perm_and_unit_mean_factors():
    """Sec. 3.3: channels sorted ascending by a (stable); abar and rho have unit
    mean over the tensor (Eq. imp and its normalization)."""
    rng = np.random.default_rng(7)
    a = rng.choice([0.5, 1.0, 2.0, 3.0], size=64).astype(np.float32)  # many ties
    rho = rng.uniform(0.5, 2, size=5).astype(np.float32)
    t = O.Tensor(5, 64, a, rho)
    assert np.array_equal(t.perm, np.argsort(a, kind="stable"))
    ab = a[t.perm].astype(np.float64).reshape(8, 8).mean(axis=1)
    assert np.allclose(t.abar, ab / ab.mean(), rtol=1e-14)
    r64 = rho.astype(np.float64)
    assert np.allclose(t.rho, r64 / r64.mean(), rtol=1e-14)
    assert abs(t.abar.mean() - 1) < 1e-14 and abs(t.rho.mean() - 1) < 1e-14


def test_ladder_floor_and_tie_hand_case():
    """Eq. ladder, the floor and the tie pass of Alg. 2 on a hand-built case:
    2 rows x 3 blocks, block means 1, 2, 3 (unit mean 0.5, 1, 1.5), rho = 1."""
    a = np.repeat(np.array([1.0, 2.0, 3.0], np.float32), 8)
    t = O.Tensor(2, 24, a)
    assert np.allclose(t.abar, [0.5, 1.0, 1.5])
    # thresholds: 0.75 (rung 0 -> 1), 1.0 (1 -> 2); ties at theta[1] = 1.0
    s = O.Sched([(8, 3), (12, 3), (16, 3)], [0.75, 1.0], 1, 0.0)
    assert t.rung_rows(s, 0).tolist() == [[0, 2, 2], [0, 2, 2]]
    # T = 1: only the first tied block in row-major order (row 0, block 1) drops.
    assert t.rung_rows(s, 1).tolist() == [[0, 1, 2], [0, 2, 2]]
    assert t.rung_rows(s, 2).tolist() == [[0, 1, 2], [0, 1, 2]]
    assert t.rung_rows(s, 1, r0=1, nrows=1).tolist() == [[0, 2, 2]]
    # floor q = 0.8 lifts block 0 (0.5) to 0.8 >= 0.75: rung 1.
    s2 = O.Sched([(8, 3), (12, 3), (16, 3)], [0.75, 1.0], -1, 0.8)
    assert t.rung_rows(s2, 0).tolist() == [[1, 2, 2], [1, 2, 2]]
    assert t.tied_blocks(s) == 2


def _load_schedule(name):
    d = json.load(open(os.path.join(GOLDEN, f"schedule_{name}.json")))
    return d, O.Sched([tuple(r) for r in d["rungs"]], d["theta"], d["j_tie"], d["q"])


@pytest.mark.parametrize("name", ["c0", "c1", "c2"])
def test_stored_schedule_budget_and_recount(name):
    """App. A.5 / A.7: the payload rate is held at rbar, short of it by less
    than one block's rate step; the stored per-tensor bit counts equal a
    block-by-block recount of the decoder's rung map."""
    d, s = _load_schedule(name)
    w = W.WORKLOADS[name]
    assert d["a_rho_checksum"] == W.a_rho_checksum(w)
    nblocks = sum(t.R * t.C // 8 for t in w.tensors)
    total = sum(d["stream_bits"])
    steps = [O.block_bits(*b) - O.block_bits(*a) for a, b in zip(d["rungs"], d["rungs"][1:])]
    assert 0 <= w.rbar * 8 * nblocks - total < max(steps)
    for i, t in enumerate(w.tensors[:3] if name != "c0" else w.tensors):
        tt = O.Tensor(t.R, t.C, *W.importance(w, i))
        rm = tt.rung_rows(s, d["tie_count"][i])
        L = np.array([O.block_bits(S, k) for S, k in d["rungs"]])
        assert int(L[rm].sum()) == d["stream_bits"][i]
        # Sec. 3.3: sorted channels make the rung non-decreasing along a row.
        assert np.all(np.diff(rm.astype(np.int32), axis=1) >= 0)
        # Only in-hull rungs, and tie demotions never exceed the tied group.
        assert d["tie_count"][i] <= tt.tied_blocks(s)


def _objective(imp, es, rungs, assign):
    return sum(imp[b] * es[j] for b, j in enumerate(assign))


def test_allocation_optimal_brute_force():
    """App. A.5 (Everett): the allocation minimizes sum imp_b e(g_b) over all
    allocations whose total rate does not exceed its own; brute force over
    every rung assignment of tiny tensors."""
    rng = np.random.default_rng(8)
    rungs, es, slopes = O.hull_rungs(W.DAMAGE_LLAMA2_7B, 4.0)
    rungs, es, slopes = rungs[2:6], es[2:6], slopes[2:5]
    L = [O.block_bits(S, k) for S, k in rungs]
    for trial in range(6):
        nb = 7
        a = np.exp(rng.normal(0, 1, 8 * nb)).astype(np.float32)
        t = O.Tensor(1, 8 * nb, a)
        s, T, bits = O.allocate([t], rungs, slopes, 3.8 + 0.05 * trial, 0.0)
        rm = t.rung_rows(s, int(T[0]))[0]
        imp = [t.imp(s, 0, c) for c in range(nb)]
        total = sum(L[j] for j in rm)
        assert total == int(bits[0])
        obj = _objective(imp, es, rungs, rm)
        best = min(_objective(imp, es, rungs, asg)
                   for asg in itertools.product(range(len(rungs)), repeat=nb)
                   if sum(L[j] for j in asg) <= total)
        assert obj <= best * (1 + 1e-9)


def test_schedule_independent_of_payload():
    """Sec. 3.6: no rung depends on a decoded weight.  Two different payloads
    parse into identical block boundaries: decoding the second stream with the
    first's schedule reproduces the second tensor exactly."""
    w = W.WORKLOADS["c0"]
    d, s = _load_schedule("c0")
    t = O.Tensor(w.tensors[0].R, w.tensors[0].C, *W.importance(w, 0))
    T = d["tie_count"][0]
    for key in (11, 22):
        stream, bits = t.synth_pack(s, T, key)
        assert bits == d["stream_bits"][0]
        Wd = t.decode_rows(s, T, stream, bits, 0, 16)
        assert np.array_equal(Wd, t.synth_rows(s, T, key, 0, 16))


def test_seed_bit_flip_footprint():
    """Sec. 4.3 / App. A.7: a corrupted seed affects only its own block; the
    footprint N_flip (Eq. security_metrics) is at most B = 8 weights, all in
    one block of 8 permuted channels of one row."""
    w = W.WORKLOADS["c0"]
    d, s = _load_schedule("c0")
    t = O.Tensor(w.tensors[0].R, w.tensors[0].C, *W.importance(w, 0))
    T = d["tie_count"][0]
    stream, bits = t.synth_pack(s, T, 5)
    rows = 4
    W0 = t.decode_rows(s, T, stream, bits, 0, rows)
    rm = t.rung_rows(s, T, 0, rows)
    L = np.array([O.block_bits(S, k) for S, k in d["rungs"]])
    off = int(L[rm[1, :]][:37].sum() + L[rm[0]].sum())  # block 37 of row 1
    bad = stream.copy()
    bad[(off + 2) >> 3] ^= np.uint8(1 << ((off + 2) & 7))  # a seed bit
    W1 = t.decode_rows(s, T, bad, bits, 0, rows)
    diff = np.argwhere(W0 != W1)
    assert 1 <= len(diff) <= 8
    assert set(diff[:, 0]) == {1}
    assert set(diff[:, 1]) <= set(t.perm[8 * 37:8 * 38].tolist())
    dW = (W1 - W0).astype(np.float64)
    eta = np.linalg.norm(dW) / np.linalg.norm(W0.astype(np.float64))
    assert 0 < eta < 1


def test_table_fault_changes_whole_tensor_parse():
    """App. A.7: a fault in the tables changes how the whole tensor is parsed."""
    w = W.WORKLOADS["c0"]
    d, s = _load_schedule("c0")
    t = O.Tensor(w.tensors[0].R, w.tensors[0].C, *W.importance(w, 0))
    T = d["tie_count"][0]
    th = list(d["theta"])
    th[4] = th[4] * 0.5
    s_bad = O.Sched([tuple(r) for r in d["rungs"]], th, d["j_tie"], d["q"])
    a, b = t.rung_rows(s, T), t.rung_rows(s_bad, T)
    assert (a != b).mean() > 0.01


# ------------------------------------------------------------- decoder

def test_outlier_overwrite():
    """Sec. 3.5 / App. A.6: outlier columns are stored in FP16 and overwrite the
    codec's reconstruction at the decoder."""
    w = W.WORKLOADS["c0"]
    d, s = _load_schedule("c0")
    t = O.Tensor(w.tensors[0].R, w.tensors[0].C, *W.importance(w, 0))
    T = d["tie_count"][0]
    cols, vals = W.outlier_case(w, 0, 4)
    stream, bits = t.synth_pack(s, T, 9)
    W0 = t.decode_rows(s, T, stream, bits, 0, 8)
    W1 = t.decode_rows(s, T, stream, bits, 0, 8, cols, vals)
    ref = vals[:8].view(np.float16).astype(np.float32)
    assert np.array_equal(W1[:, cols], ref)
    keep = np.setdiff1d(np.arange(t.C), cols)
    assert np.array_equal(W1[:, keep], W0[:, keep])


def test_gemv_f64_against_numpy():
    rng = np.random.default_rng(9)
    Wm = rng.normal(size=(37, 96)).astype(np.float32)
    x = W.to_bf16_bits(rng.normal(size=(3, 96)).astype(np.float32))
    y = O.gemv_f64(Wm, x)
    ref = W.bf16_bits_to_f32(x).astype(np.float64) @ Wm.astype(np.float64).T
    assert np.allclose(y, ref, rtol=1e-13, atol=1e-12)


def test_decode_rows_offset_consistency():
    """Decoding a row range from its own bit offset equals the same rows of a
    whole-tensor decode (left-to-right parse, Alg. 2)."""
    w = W.WORKLOADS["c0"]
    d, s = _load_schedule("c0")
    t = O.Tensor(w.tensors[0].R, w.tensors[0].C, *W.importance(w, 0))
    T = d["tie_count"][0]
    stream, bits = t.synth_pack(s, T, 3)
    full = t.decode_rows(s, T, stream, bits)
    part = t.decode_rows(s, T, stream, bits, 500, 7)
    assert np.array_equal(full[500:507], part)
    with pytest.raises(ValueError):
        t.decode_rows(s, T, stream, bits - 1)


def test_threaded_baseline_matches_plain():
    w = W.WORKLOADS["c0"]
    d, s = _load_schedule("c0")
    t = O.Tensor(w.tensors[0].R, w.tensors[0].C, *W.importance(w, 0))
    T = d["tie_count"][0]
    stream, bits = t.synth_pack(s, T, 3)
    x = W.x_bf16(w, 0, 2)
    y, n = t.decode_gemv_threads(s, T, stream, bits, x, 3)
    assert n == 3
    assert np.array_equal(y, O.gemv_f64(t.decode_rows(s, T, stream, bits), x))


# --------------------------------------------------------- tiny encoder

def test_encoder_recovers_planted_blocks():
    """Sec. 3.1 seed search: a block that is exactly U(s0) t0 2^E0 is found
    with zero quantized error."""
    for S, k in ((8, 3), (10, 2), (12, 4)):
        taps = O.find_taps(S)
        s0, E0, t0 = 77 % ((1 << S) - 1), -4, [3, -5, 7, 1][:k]
        w = O.reconstruct_block(S, k, taps, s0, E0, t0).astype(np.float64)
        seed, E, t, err = O.encode_block(S, k, taps, w)
        assert err == 0.0
        assert np.array_equal(O.reconstruct_block(S, k, taps, seed, E, t).astype(np.float64), w)


def test_encoder_beats_other_seeds_lstsq():
    """For random blocks, no other seed gives a smaller quantized error than the
    chosen one; each competitor is fitted here with numpy's lstsq and the same
    exponent rule, an implementation independent of the oracle's solver."""
    rng = np.random.default_rng(10)
    S, k = 8, 3
    taps = O.find_taps(S)
    for _ in range(6):
        w = rng.normal(0, 0.02, 8)
        seed, E, t, err = O.encode_block(S, k, taps, w)
        for s2 in rng.choice(np.arange(1, 1 << S), 40, replace=False):
            x = np.array(_states(S, taps, int(s2), 8 * k), np.float64).reshape(8, k)
            U = (x - 2 ** (S - 1)) / 2 ** (S - 1)
            ts = np.linalg.lstsq(U, w, rcond=None)[0]
            for E2 in range(-8, 8):
                m = np.rint(ts / 2.0 ** E2)
                if m.min() >= -8 and m.max() <= 7:
                    break
            m = np.clip(np.rint(ts / 2.0 ** E2), -8, 7)
            e2 = float(((w - U @ m * 2.0 ** E2) ** 2).sum())
            assert err <= e2 + 1e-15


def test_round_trip_64x64_mixed_rungs():
    """Encode a 64x64 matrix with the oracle's seed search at the rungs the
    schedule assigns (four rungs, the last block column of every row at S = 16),
    pack, decode: the decoder reproduces the encoder's reconstruction bit for bit
    (Sec. 3.1 seed search, Alg. 2 decode)."""
    rng = np.random.default_rng(11)
    R = Cc = 64
    a = np.exp(rng.normal(0, 1, Cc)).astype(np.float32)
    t = O.Tensor(R, Cc, a)
    ab = t.abar
    assert ab[7] > ab[6]
    rungs = [(8, 3), (10, 3), (12, 3), (16, 3)]
    # thresholds below the top block mean, the last one between the two largest
    th = [float(ab[2]), float(ab[5]), float((ab[6] + ab[7]) / 2)]
    s = O.Sched(rungs, th, -1, 0.0)
    rm = t.rung_rows(s, 0)
    assert set(rm.ravel().tolist()) == {0, 1, 2, 3}
    assert np.all(rm[:, 7] == 3) and np.all(rm[:, :7] < 3)
    Wt = rng.normal(0, 0.02, (R, Cc))
    stream = np.zeros(64 * 8 * 6 + 64, np.uint8)
    ref = np.zeros((R, Cc), np.float32)
    errs = np.zeros((R, Cc // 8))
    pos = 0
    for r in range(R):
        for c in range(Cc // 8):
            S, k = rungs[rm[r, c]]
            blk = Wt[r, t.perm[8 * c:8 * c + 8]]
            seed, E, tt, err = O.encode_block(S, k, O.find_taps(S), blk)
            O.write_bits(stream, pos, S, seed)
            O.write_bits(stream, pos + S, 4, E & 15)
            for j in range(k):
                O.write_bits(stream, pos + S + 4 + 4 * j, 4, tt[j] & 15)
            pos += O.block_bits(S, k)
            rec = O.reconstruct_block(S, k, O.find_taps(S), seed, E, tt)
            ref[r, t.perm[8 * c:8 * c + 8]] = rec
            errs[r, c] = err
            assert abs(float(((blk - rec.astype(np.float64)) ** 2).sum()) - err) <= 1e-15
    assert pos == t.row_bit_offset(s, 0, R)
    dec = t.decode_rows(s, 0, stream, pos)
    assert np.array_equal(dec, ref)
    # A wider seed space fits at least as well on average (more seeds searched).
    assert errs[:, 7].mean() < errs[:, 0].mean()


# ------------------------------------------- checker helpers of the GPU tests
#
# or_synth_gemv_threads (the fp64 y reference of the large parity tests),
# or_synth_pack_rows (the reference of the device stream bits) and
# or_decode_gemv_threads, pinned to a whole-tensor left-to-right parse
# (Alg. 2 with the tie counter running from row 0) on a tensor whose tied group
# spans every row and is only partly demoted, so a row range starting inside
# the demoted part needs the right carry-in.

def _tie_case():
    rng = np.random.default_rng(21)
    R, Cc = 64, 256
    a = np.exp(rng.normal(0, 0.7, Cc)).astype(np.float32)
    t = O.Tensor(R, Cc, a)
    ab = t.abar
    assert len(set(ab.tolist())) == Cc // 8
    cstar = 20
    # thresholds: one between block means, one exactly at block column cstar's
    # mean, whose tied group (column cstar of every row, rho = 1) is demoted
    # for its first T members only
    s = O.Sched([(8, 3), (12, 3), (16, 3)], [float(ab[10]), float(ab[cstar])], 1, 0.0)
    T = 20
    assert t.tied_blocks(s) == R
    full_rm = t.rung_rows(s, T)
    assert np.all(full_rm[:T, cstar] == 1) and np.all(full_rm[T:, cstar] == 2)
    key = 0x5EED
    stream, bits = t.synth_pack(s, T, key)
    full = t.decode_rows(s, T, stream, bits)
    L = np.array([O.block_bits(S, k) for S, k in s.rungs], np.int64)
    off = np.concatenate([[0], np.cumsum(L[full_rm].sum(axis=1))])
    assert off[-1] == bits
    return t, s, T, key, stream, bits, full, off


def _exact_y(Wm, x, nb):
    import math
    xf = W.bf16_bits_to_f32(x).astype(np.float64).reshape(nb, -1)
    Wd = Wm.astype(np.float64)
    y = np.array([[math.fsum(Wd[r] * xf[b]) for r in range(Wd.shape[0])] for b in range(nb)])
    ya = np.abs(xf) @ np.abs(Wd).T
    return y, ya


@pytest.mark.parametrize("nb", [1, 3, 16])
@pytest.mark.parametrize("r0,n", [(0, 64), (15, 10), (20, 9), (37, 27)])
def test_synth_gemv_threads_pinned(nb, r0, n):
    t, s, T, key, stream, bits, full, off = _tie_case()
    rng = np.random.default_rng(nb * 100 + r0)
    x = W.to_bf16_bits(rng.normal(0, 1, nb * t.C).astype(np.float32)).reshape(nb, t.C)
    y, ya = t.synth_gemv(s, T, key, x, r0, n, nthreads=3)
    ry, rya = _exact_y(full[r0:r0 + n], x, nb)
    assert y.shape == (nb, n)
    assert np.all(np.abs(y - ry) <= 1e-13 * rya + 1e-300)
    assert np.allclose(ya, rya, rtol=1e-13, atol=0)
    # the rows themselves, generated from the same carry-in
    assert np.array_equal(t.synth_rows(s, T, key, r0, n), full[r0:r0 + n])


@pytest.mark.parametrize("r0,n", [(0, 5), (15, 10), (19, 2), (20, 44)])
def test_synth_pack_rows_is_a_slice(r0, n):
    t, s, T, key, stream, bits, full, off = _tie_case()
    part, pbits = t.synth_pack_rows(s, T, key, r0, n, int(off[r0 + n] - off[r0]))
    assert pbits == off[r0 + n] - off[r0]
    allbits = np.unpackbits(stream, bitorder="little")[off[r0]:off[r0 + n]]
    assert np.array_equal(np.unpackbits(part, bitorder="little")[:pbits], allbits)


@pytest.mark.parametrize("r0,n", [(15, 10), (33, 31)])
def test_decode_gemv_threads_row_range(r0, n):
    t, s, T, key, stream, bits, full, off = _tie_case()
    x = W.x_bf16(W.WORKLOADS["c0"], 0, 2)[:, :t.C].copy()
    y, used = t.decode_gemv_threads(s, T, stream, bits, x, 4, r0, n)
    ry, rya = _exact_y(full[r0:r0 + n], x, 2)
    assert np.all(np.abs(y[:, r0:r0 + n] - ry) <= 1e-13 * rya + 1e-300)

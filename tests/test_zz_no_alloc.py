"""The allocation-free row pass (seedq_row_plan_static) against seedq_layer_prepare.

Callers that cannot allocate device memory when they need a plan (a fixed
budget reserved up front, an allocator-less runtime) use the static-scratch
entry point; its breakpoints and row offsets must equal those the allocating
prepare path builds, call after call, since every call shares one scratch array.
"""
import json
import os

import numpy as np
import pytest

from paper_2609_38477_gb300 import workloads as W

torch = pytest.importorskip("torch")
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")

pytestmark = pytest.mark.gpu


def _seq_sum(v: np.ndarray) -> float:
    """Left-to-right fp64 sum (the fixed order of App. A.7)."""
    return float(np.cumsum(np.asarray(v, np.float64))[-1])


def _factors(a, rho, perm, R):
    nb = a.size // 8
    ap = a[perm].astype(np.float64).reshape(nb, 8)
    s = ap[:, 0].copy()
    for i in range(1, 8):
        s = s + ap[:, i]
    abar = s / 8.0
    abar = abar / (_seq_sum(abar) / nb)
    if rho is None:
        r = np.ones(R, np.float64)
    else:
        r64 = rho.astype(np.float64)
        r = r64 / (_seq_sum(r64) / R)
    return abar, r


def _rung_map(brk, R, J, nb):
    c = np.arange(nb)
    rm = np.zeros((R, nb), np.uint8)
    for j in range(J - 1):
        rm += (brk[:, j:j + 1] <= c[None, :]).astype(np.uint8)
    return rm


@pytest.mark.parametrize("name,i", [("c1", 0), ("c2", 6)])
def test_static_row_plan_matches_prepare(name, i):
    from paper_2609_38477_gb300 import build

    build.build()
    from paper_2609_38477_gb300 import seedq as Q

    d = json.load(open(os.path.join(GOLDEN, f"schedule_{name}.json")))
    w = W.WORKLOADS[name]
    t = w.tensors[i]
    a, rho = W.importance(w, i)
    rungs = [tuple(r) for r in d["rungs"]]
    J, T = len(rungs), d["tie_count"][i]
    layer = Q.Layer(t.R, t.C, a, rho, rungs, d["theta"], d["j_tie"], d["q"], T, max_batch=1)
    ref_rm = layer.rung_map()
    ref_off = layer.row_offsets()
    abar, r = _factors(a, rho, layer.perm(), t.R)
    abar_d = torch.from_numpy(abar).cuda()
    rho_d = torch.from_numpy(r).cuda()
    brk = torch.empty((t.R, J - 1), dtype=torch.int32, device="cuda")
    off = torch.empty(t.R + 1, dtype=torch.int64, device="cuda")
    summ = torch.empty(2, dtype=torch.int64, device="cuda")
    for call in range(2):
        brk.fill_(-7)
        off.fill_(-7)
        Q.row_plan_static(abar_d, rho_d, t.R, t.C // 8, rungs, d["theta"], d["j_tie"], d["q"], T,
                          brk, off, summ)
        torch.cuda.synchronize()
        got_rm = _rung_map(brk.cpu().numpy(), t.R, J, t.C // 8)
        assert np.array_equal(got_rm, ref_rm), f"call {call}"
        assert np.array_equal(off.cpu().numpy().view(np.uint64), ref_off), f"call {call}"
        s = summ.cpu().numpy()
        assert int(s[1]) == layer.stream_bits == d["stream_bits"][i]
        assert T <= int(s[0])
    layer.release()


def test_static_row_plan_rejects_oversize():
    from paper_2609_38477_gb300 import build

    build.build()
    from paper_2609_38477_gb300 import seedq as Q

    big = Q.STATIC_PLAN_MAX_ROWS + 1
    with pytest.raises(Q.SeedQError) as e:
        Q.row_plan_static(1, 1, big, 512, [(8, 3), (16, 3)], [1.0], -1, 0.0, 0, 1, 1, 1)
    assert e.value.status == 6


@pytest.mark.parametrize("name,i", [("c0", 0), ("c2", 3)])
def test_static_row_plan_matches_oracle(name, i):
    """The allocation-free row pass against the CPU oracle's schedule (Alg. 2:
    rung map with the tie pass, row bit offsets), fed the oracle's own factors."""
    import oracle as O
    from paper_2609_38477_gb300 import build

    build.build()
    from paper_2609_38477_gb300 import seedq as Q

    d = json.load(open(os.path.join(GOLDEN, f"schedule_{name}.json")))
    w = W.WORKLOADS[name]
    t = w.tensors[i]
    a, rho = W.importance(w, i)
    rungs = [tuple(r) for r in d["rungs"]]
    s = O.Sched(rungs, d["theta"], d["j_tie"], d["q"])
    ot = O.Tensor(t.R, t.C, a, rho)
    J, T, nb = len(rungs), d["tie_count"][i], t.C // 8
    want_rm = ot.rung_rows(s, T)
    L = np.array([O.block_bits(S, k) for S, k in rungs], np.uint64)
    want_off = np.concatenate([[0], np.cumsum(L[want_rm].sum(axis=1, dtype=np.uint64))]).astype(np.uint64)
    assert int(want_off[-1]) == d["stream_bits"][i]
    abar_d = torch.from_numpy(ot.abar).cuda()
    rho_d = torch.from_numpy(ot.rho).cuda()
    brk = torch.empty((t.R, J - 1), dtype=torch.int32, device="cuda")
    off = torch.empty(t.R + 1, dtype=torch.int64, device="cuda")
    summ = torch.empty(2, dtype=torch.int64, device="cuda")
    for call in range(2):
        brk.fill_(-7)
        off.fill_(-7)
        Q.row_plan_static(abar_d, rho_d, t.R, nb, rungs, d["theta"], d["j_tie"], d["q"], T, brk, off, summ)
        torch.cuda.synchronize()
        assert np.array_equal(_rung_map(brk.cpu().numpy(), t.R, J, nb), want_rm), f"call {call}"
        assert np.array_equal(off.cpu().numpy().view(np.uint64), want_off), f"call {call}"
        assert int(summ.cpu().numpy()[0]) == ot.tied_blocks(s)


def test_static_row_plan_single_rung():
    """One rung: no breakpoints (brk may be NULL), no ties; every row holds nb
    blocks of S + 4k + 4 bits (Eq. rate), so row r starts at r * nb * L."""
    from paper_2609_38477_gb300 import build

    build.build()
    from paper_2609_38477_gb300 import seedq as Q

    R, nb, S, k = 777, 96, 12, 3
    abar_d = torch.ones(nb, dtype=torch.float64, device="cuda")
    rho_d = torch.ones(R, dtype=torch.float64, device="cuda")
    off = torch.empty(R + 1, dtype=torch.int64, device="cuda")
    summ = torch.empty(2, dtype=torch.int64, device="cuda")
    for call in range(2):
        off.fill_(-7)
        Q.row_plan_static(abar_d, rho_d, R, nb, [(S, k)], [], -1, 0.0, 0, None, off, summ)
        torch.cuda.synchronize()
        L = S + 4 * k + 4
        assert np.array_equal(off.cpu().numpy(), np.arange(R + 1, dtype=np.int64) * nb * L), f"call {call}"
        assert summ.cpu().numpy().tolist() == [0, R * nb * L]

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

"""Write the decoder schedule tables of every synthetic workload.

The schedule (hull rungs, thresholds theta_j = lambda / s_j, the tied
threshold, the floor q and the per-tensor tie counts T_t) is what the paper's
global table carries (Sec. 3.6, Alg. 1 output).  It is produced here by the
oracle's encoder-side allocator only, from the seeded importance factors of
``paper_2609_38477_gb300.workloads`` and the damage tables printed in the
paper; nothing here touches the CUDA library.

Usage: python tests/golden/make_schedules.py [workload ...]
"""
from __future__ import annotations

import json
import os
import sys
import time

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)
sys.path.insert(0, os.path.join(ROOT, "oracle"))

import oracle as O  # noqa: E402
from paper_2609_38477_gb300 import workloads as W  # noqa: E402

FLOOR_F = 0.06  # Sec. 3.3: f chosen once on Llama-2-7B and fixed for every model


def make(name: str) -> dict:
    w = W.WORKLOADS[name]
    rungs, es, slopes = O.hull_rungs(W.DAMAGE_TABLES[w.damage](), w.rbar)
    tensors = [O.Tensor(t.R, t.C, *W.importance(w, i)) for i, t in enumerate(w.tensors)]
    sched, T, bits = O.allocate(tensors, rungs, slopes, w.rbar, FLOOR_F)
    nblocks = sum(t.R * t.C // 8 for t in w.tensors)
    return {
        "workload": name,
        "description": w.description,
        "rbar": w.rbar,
        "floor_f": FLOOR_F,
        "damage_table": w.damage,
        "rungs": [list(r) for r in rungs],
        "hull_damage": es,
        "slopes": slopes,
        "theta": [float(x) for x in sched.theta],
        "j_tie": sched.j_tie,
        "q": sched.q,
        "tie_count": [int(x) for x in T],
        "stream_bits": [int(x) for x in bits],
        "mean_bits_per_weight": float(sum(int(x) for x in bits) / (8 * nblocks)),
        "a_rho_checksum": W.a_rho_checksum(w),
    }


def main(names):
    for name in names:
        t0 = time.time()
        d = make(name)
        path = os.path.join(HERE, f"schedule_{name}.json")
        with open(path, "w") as f:
            json.dump(d, f, indent=1)
        print(f"{name}: J={len(d['rungs'])} j_tie={d['j_tie']} "
              f"mean={d['mean_bits_per_weight']:.9f} bpw ({time.time() - t0:.1f}s) -> {path}")


if __name__ == "__main__":
    main(sys.argv[1:] or list(W.WORKLOADS))

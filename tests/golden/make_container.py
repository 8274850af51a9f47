"""Write tests/golden/tiny_model.seedq with the oracle only.

A two-tensor model in the container layout: the Sec. 3.6 table (four rungs,
thresholds, floor) and, per tensor, shape, importance factors, tie count,
FP16 outlier columns and the synthetic payload stream the oracle packs
(seeded counter-based fields, as the workload recipe draws them).

Usage: python tests/golden/make_container.py
"""
from __future__ import annotations

import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, os.path.join(ROOT, "oracle"))

import oracle as O  # noqa: E402

RUNGS = [(8, 3), (10, 3), (12, 3), (14, 4)]
THETA = [0.7, 1.1, 1.6]
J_TIE = -1
Q_FLOOR = 0.0


def model():
    rng = np.random.default_rng(20260)
    s = O.Sched(RUNGS, THETA, J_TIE, Q_FLOOR)
    tensors = []
    for name, R, Cc, with_rho, n_out, key in (("t0", 48, 64, True, 2, 0x1234),
                                              ("t1", 32, 128, False, 0, 0x5678)):
        a = np.exp(rng.normal(0, 1, Cc)).astype(np.float32)
        rho = np.exp(rng.normal(0, 0.5, R)).astype(np.float32) if with_rho else None
        ot = O.Tensor(R, Cc, a, rho)
        stream, bits = ot.synth_pack(s, 0, key)
        cols = np.sort(rng.choice(Cc, n_out, replace=False)).astype(np.int32)
        vals = (rng.normal(0, 4, (R, n_out)).astype(np.float16)).view(np.uint16)
        tensors.append({"name": name, "rows": R, "cols": Cc, "a": a, "rho": rho, "tie_count": 0,
                        "outlier_cols": cols, "outlier_vals": vals, "stream": stream,
                        "stream_bits": bits, "key": key})
    return tensors


def main():
    path = os.path.join(HERE, "tiny_model.seedq")
    O.write_container(path, RUNGS, THETA, J_TIE, Q_FLOOR, model())
    print(path, os.path.getsize(path), "bytes")


if __name__ == "__main__":
    main()

"""Writes tests/golden/oracle_tiny.json: the fp64 oracle's outputs on one tiny
seeded unit, a regression fixture that keeps the oracle from drifting.

The paper prints no worked numeric example of the compression path, so no
fixture here carries the paper's own numbers; this one is produced only from
the oracle (and the seeded input generator).  Run from the repository root:
    python tests/golden/make_golden.py
"""
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import grkv_inputs as gi  # noqa: E402
import oracle as O  # noqa: E402

WL = gi.Workload("golden_tiny", 1, 2, 96, 16, 4, 24, 5, 1e-2, "f32", "lowrank", 12345)


def params():
    return O.Params(group=WL.group, n=WL.n, d=WL.d, window=WL.window, budget=WL.budget,
                    pool_kernel=WL.pool_kernel, n_sink=4, beta=0.1, lambda_v=WL.lambda_v)


def compute():
    q, k, v = gi.unit_arrays(WL, 0)
    out = O.compress_unit(q, k, v, params())
    # the key step (converged CG) on the same unit
    import dataclasses
    key = O.compress_unit(q, k, v, dataclasses.replace(params(), update_k=True, lambda_k=0.05,
                                                       cg_iters=2000, cg_tol=1e-13))
    return {
        "workload": WL.__dict__,
        "idx": out["idx"].tolist(),
        "fixed": out["fixed"].astype(int).tolist(),
        "scores": out["scores"].tolist(),
        "y": out["y"].tolist(),
        "v_out": out["v_out"].tolist(),
        "k_out_key_step": key["k_out"].tolist(),
    }


if __name__ == "__main__":
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "oracle_tiny.json")
    with open(path, "w") as f:
        json.dump(compute(), f, indent=0)
    print("wrote", path)

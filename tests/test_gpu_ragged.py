"""GPU parity of per-unit budgets (grkv_compress_ragged): every unit against
the oracle's compression with its own budget (Sec. 4.2 of the paper pairs
GRKV with layer- and head-wise budget allocations), and equal budgets give
exactly grkv_compress's results."""
import numpy as np
import pytest
import torch

import grkv_inputs as gi
import oracle as O
from paper_2605_31105_gb300 import binding as b
from tests import gpu_cases as G

pytestmark = pytest.mark.gpu


def _ragged(c, p, budgets):
    dt = torch.bfloat16 if c.wl.dtype == "bf16" else torch.float32
    rows = int(sum(budgets))
    ko = torch.empty((rows, 128), dtype=dt, device="cuda")
    vo = torch.empty_like(ko)
    idx = torch.full((rows,), -1, dtype=torch.int32, device="cuda")
    ws = torch.full((b.grkv_compress_ragged_workspace_size(p, budgets),), 0xFF,
                    dtype=torch.uint8, device="cuda")
    b.grkv_compress_ragged(p, budgets, c.dq, c.dk, c.dv, ko, vo, idx, ws)
    assert b.grkv_status(ws) == b.GRKV_OK
    off = np.concatenate([[0], np.cumsum(budgets)])
    idx, ko, vo = idx.cpu().numpy(), G.to_host(ko), G.to_host(vo)
    return [(idx[off[u]:off[u + 1]], ko[off[u]:off[u + 1]], vo[off[u]:off[u + 1]])
            for u in range(c.U)]


@pytest.mark.parametrize("wl,budgets", [
    (gi.workload(1), [512, 512, 256, 256, 384, 1024, 512, 128]),
    (gi.workload(1).replace(dtype="f32", units=4, n=2048), [256, 100, 100, 33]),
], ids=["c1_bf16", "c1_f32_n2048"])
def test_ragged_budgets_match_oracle(grkv_lib, wl, budgets):
    c = G.Case(wl)
    p = G.lib_params(wl, c.U)
    out = _ragged(c, p, budgets)
    scores, _, _ = G.run_score(c, p)   # budget-independent
    for u, (iu, ku, vu) in enumerate(out):
        op = G.oracle_params(wl, budget=budgets[u])
        ora = O.compress_unit(c.q[u], c.k[u], c.v[u], op)
        G.check_unit_end_to_end(wl.name + "_ragged", u, c.q[u], c.k[u], c.v[u], op, ora, iu,
                                scores[u], ku, vu, wl.dtype)


def test_equal_budgets_are_grkv_compress(grkv_lib):
    """With one budget for every unit the ragged entry point is grkv_compress
    bit for bit (deterministic mode: same kernels, same order)."""
    wl = gi.workload(2).replace(units=3, n=8192, budget=1024)
    c = G.Case(wl)
    p = G.lib_params(wl, c.U)
    p.flags = b.GRKV_DETERMINISTIC
    idx, ko, vo = G.run_compress(c, p)
    out = _ragged(c, p, [wl.budget] * c.U)
    for u, (iu, ku, vu) in enumerate(out):
        np.testing.assert_array_equal(iu, idx[u])
        np.testing.assert_array_equal(ku, ko[u])
        np.testing.assert_array_equal(vu, vo[u])

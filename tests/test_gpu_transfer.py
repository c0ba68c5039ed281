"""GPU parity of the decode-side transfer check (grkv_transfer_check, App. G
of the paper) against the fp64 oracle, through the C ABI.

The check composes the scoring path's attention outputs, so its tolerances
follow from the bound on those outputs (gpu_cases): with delta the Frobenius
norm of the elementwise bound on a GPU output Y = A V,
  |e_gpu - e_ora| <= 2 sqrt(e_ora) (delta_full + delta_cache) + (delta_full + delta_cache)^2
for each squared error e, the same with e = ||Y||^2 for the norms, and a
cosine off by at most 2 (||ds_w|| / ||s_w|| + ||ds_h|| / ||s_h||), ||ds|| <=
delta / sqrt(rows) for a mean over rows.  The failure flag is an integer
decision: it is compared where both of its error differences exceed their
bounds (elsewhere either answer is consistent with the arithmetic).
"""
import math

import numpy as np
import pytest
import torch

import grkv_inputs as gi
import oracle as O
from paper_2605_31105_gb300 import binding as b
from tests import gpu_cases as G

pytestmark = pytest.mark.gpu

RAGGED = gi.Workload("ragged_g3_w5_n1000", 3, 3, 1000, 128, 5, 77, 5, 1e-2, "f32", "lowrank", 777)
CASES = {
    "c1_llama_layer_bf16_held32": (gi.workload(1), 32),
    "ragged_f32_held7": (RAGGED, 7),
    "c2_recipe_n8192_held32": (gi.workload(2).replace(units=3, n=8192, budget=1024), 32),
}


def _y_bound(q, kc, vc, op, window_rule, tc):
    """Frobenius norm of the elementwise bound on the GPU's Y = A V of the
    queries q over the cache (kc, vc) (see gpu_cases)."""
    q = np.asarray(q, np.float64)
    g, h = q.shape[0], q.shape[1]
    sub = O.Params(group=g, n=kc.shape[0], d=op.d, window=h, budget=kc.shape[0],
                   causal=bool(window_rule and op.causal))
    A, _, _ = O.softmax_rows(O.window_logits(q, kc, sub))
    tol = G.score_rel_tol(q, kc, sub) + kc.shape[0] * G.U + (2.0 ** -8 if tc else 0.0)
    lim = tol * (A @ np.abs(np.asarray(vc, np.float64))) + 1e-7
    return float(np.linalg.norm(lim)), h * g


@pytest.mark.parametrize("name", list(CASES))
def test_transfer_check_matches_oracle(grkv_lib, name):
    wl, held = CASES[name]
    c = G.Case(wl)
    p = G.lib_params(wl, c.U)
    idx, ko, vo = G.run_compress(c, p)
    qh = np.stack([gi.heldout_queries(wl, u, held) for u in c.units])
    dqh = G.to_device(qh, wl.dtype)
    dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    dko = torch.from_numpy(ko).to(dt).cuda()
    dvo = torch.from_numpy(vo).to(dt).cuda()
    didx = torch.from_numpy(idx).cuda()
    rep = torch.full((c.U, 8), float("nan"), dtype=torch.float32, device="cuda")
    ws = torch.full((b.grkv_transfer_workspace_size(p, held),), 0xFF, dtype=torch.uint8,
                    device="cuda")
    b.grkv_transfer_check(p, held, c.dq, dqh, c.dk, c.dv, didx, dko, dvo, rep, ws)
    assert b.grkv_status(ws) == b.GRKV_OK
    rep = rep.cpu().numpy().astype(np.float64)
    op = G.oracle_params(wl)
    tc = G.uses_tensor_cores(p)
    oras = []
    for i in range(c.U):
        K, V = c.k[i].astype(np.float64), c.v[i].astype(np.float64)
        K0, V0 = K[idx[i]], V[idx[i]]
        Ko, Vo = ko[i].astype(np.float64), vo[i].astype(np.float64)
        o = O.transfer_check(c.q[i], qh[i], K, V, idx[i], Ko, Vo, op)
        oras.append(o)
        dwf, mw = _y_bound(c.q[i], K, V, op, True, tc)
        dhf, mh = _y_bound(qh[i], K, V, op, False, tc)
        bounds = {}
        for nm, kc, vc in (("base", K0, V0), ("comp", Ko, Vo)):
            dw, _ = _y_bound(c.q[i], kc, vc, op, True, tc)
            dh, _ = _y_bound(qh[i], kc, vc, op, False, tc)
            bounds["e_win_" + nm] = dwf + dw
            bounds["e_held_" + nm] = dhf + dh
        got = dict(zip(["e_win_base", "e_win_comp", "e_held_base", "e_held_comp", "y_win2",
                        "y_held2", "cos", "fail"], rep[i]))
        for key, dl in list(bounds.items()) + [("y_win2", dwf), ("y_held2", dhf)]:
            ref = o[key]
            lim = 2 * math.sqrt(ref) * dl + dl * dl + 1e-6 * ref + 1e-12
            assert abs(got[key] - ref) <= lim, f"unit {i} {key}: {got[key]:.6e} vs {ref:.6e} (bound {lim:.2e})"
        yw = O.cache_output(c.q[i], K, V, op, True)
        yh = O.cache_output(qh[i], K, V, op, False)
        cos_lim = 2 * (dwf / math.sqrt(mw) / np.linalg.norm(yw.mean(0)) +
                       dhf / math.sqrt(mh) / np.linalg.norm(yh.mean(0))) + 1e-6
        assert abs(got["cos"] - o["cos"]) <= cos_lim, (i, got["cos"], o["cos"], cos_lim)
        decided = (abs(o["e_win_comp"] - o["e_win_base"]) >
                   4 * math.sqrt(max(o["e_win_base"], o["e_win_comp"])) *
                   (bounds["e_win_base"] + bounds["e_win_comp"]) and
                   abs(o["e_held_comp"] - o["e_held_base"]) >
                   4 * math.sqrt(max(o["e_held_base"], o["e_held_comp"])) *
                   (bounds["e_held_base"] + bounds["e_held_comp"]))
        if decided:
            assert bool(got["fail"]) == o["fail"], f"unit {i}: failure flag"
    # the value step lowers the window error on every unit (Eq. 6 at lambda > 0)
    assert all(o["e_win_comp"] < o["e_win_base"] for o in oras)


def test_transfer_check_full_budget_has_no_error(grkv_lib):
    """B = n and lambda = inf: the compressed and eviction-only caches are the
    full cache.  With GRKV_DETERMINISTIC the attention outputs of identical
    caches are bit-identical, so every error is exactly zero and no unit
    fails (a tie is not a failure)."""
    wl = gi.workload(1).replace(units=2, n=1024, budget=1024)
    c = G.Case(wl)
    p = G.lib_params(wl, c.U, lambda_v=math.inf)
    idx, ko, vo = G.run_compress(c, p)
    held = 16
    qh = np.stack([gi.heldout_queries(wl, u, held) for u in c.units])
    rep = torch.empty((c.U, 8), dtype=torch.float32, device="cuda")
    p.flags = b.GRKV_DETERMINISTIC
    ws = torch.empty((b.grkv_transfer_workspace_size(p, held),), dtype=torch.uint8, device="cuda")
    dko = torch.from_numpy(ko).to(torch.bfloat16).cuda()
    dvo = torch.from_numpy(vo).to(torch.bfloat16).cuda()
    b.grkv_transfer_check(p, held, c.dq, G.to_device(qh, wl.dtype), c.dk, c.dv,
                          torch.from_numpy(idx).cuda(), dko, dvo, rep, ws)
    assert b.grkv_status(ws) == b.GRKV_OK
    r = rep.cpu().numpy()
    assert (r[:, :4] == 0).all(), r
    assert (r[:, 7] == 0).all()
    assert (r[:, 4:6] > 0).all() and (np.abs(r[:, 6]) <= 1.0 + 1e-6).all()

"""GPU parity: every stage of the CUDA path against the fp64 oracle, through
the C ABI, element by element on the same seeded inputs.

Stage tests feed both sides identical inputs (the oracle's fp32 scores, its
fp32 target and its retained set), so integer results must match bit for bit
and merged values within the method's bar; the end-to-end test checks the
retained set up to score ties within the derived score tolerance.
"""
import math

import numpy as np
import pytest

import grkv_inputs as gi
import oracle as O
from paper_2605_31105_gb300 import binding as b
from tests import gpu_cases as G

pytestmark = pytest.mark.gpu

RAGGED = gi.Workload("ragged_g3_w5_n1000", 3, 3, 1000, 128, 5, 77, 5, 1e-2, "bf16", "lowrank", 777)
M256 = gi.Workload("m256_spans_n8192", 2, 4, 8192, 128, 64, 512, 7, 1e-1, "bf16", "spans", 888)
# 128 < m < 256: the second 128-row block of the tensor-core merge is partly padding
M160 = gi.Workload("m160_lowrank_n3000", 2, 4, 3000, 128, 40, 300, 7, 1e-1, "bf16", "lowrank", 161)
M200 = gi.Workload("m200_spans_n2500", 2, 5, 2500, 128, 40, 333, 7, 1e-1, "bf16", "spans", 202)

CASES = {
    "c0_full": (gi.workload(0), {}),
    "c1_full": (gi.workload(1), {}),
    "ragged_causal": (RAGGED, {}),
    "ragged_noncausal_avgpool": (RAGGED, dict(causal=False, pool_type="avg")),
    "ragged_f32": (RAGGED.replace(dtype="f32"), {}),
    "m256_spans": (M256, {}),
    "m160_ragged": (M160, {}),
    "m200_noncausal": (M200, dict(causal=False)),
    "c2_recipe_n8192": (gi.workload(2).replace(units=3, n=8192, budget=1024), {}),
    "g1_w1": (RAGGED.replace(group=1, window=1, budget=40, seed=5), dict(n_sink=0, beta=0.0)),
}


class Prepared:
    def __init__(self, wl, over):
        self.wl = wl
        self.over = over
        self.case = G.Case(wl)
        self.op = G.oracle_params(wl, **over)
        self.p = G.lib_params(wl, self.case.U, **over)
        self.ora = [O.compress_unit(self.case.q[i], self.case.k[i], self.case.v[i], self.op)
                    for i in range(self.case.U)]
        self.tol = [G.score_rel_tol(self.case.q[i], self.case.k[i], self.op)
                    for i in range(self.case.U)]


@pytest.fixture(scope="module", params=list(CASES))
def prep(request, grkv_lib):
    wl, over = CASES[request.param]
    return Prepared(wl, over)


PATHS = {"default": 0, "one_read": b.GRKV_ONE_READ_SCORE, "portable": b.GRKV_FORCE_SIMT}


@pytest.mark.parametrize("path", list(PATHS))
def test_score_stage(prep, path):
    c, op = prep.case, prep.op
    p = G.lib_params(prep.wl, c.U, **prep.over)
    p.flags = PATHS[path]
    scores, y, rs = G.run_score(c, p)
    for i, ora in enumerate(prep.ora):
        lb = G.logit_bound(c.q[i], c.k[i], op)
        np.testing.assert_allclose(rs[i, :, 0], ora["row_max"], rtol=0, atol=lb + 1e-6)
        G.assert_scores(rs[i, :, 1], ora["row_sum"], prep.tol[i] + op.n * G.U, "row_sum")
        G.assert_scores(scores[i], ora["scores"], prep.tol[i])
        s_abs = ora["attn"] @ np.abs(c.v[i].astype(np.float64))
        lim = (prep.tol[i] + op.n * G.U + G.y_tol_extra(p)) * s_abs + 1e-7
        err = np.abs(y[i] - ora["y"])
        assert (err <= lim).all(), f"y: worst excess {(err - lim).max():.3e}"


def test_select_stage_bit_exact(prep):
    scores32 = np.stack([o["scores32"] for o in prep.ora])
    idx = G.run_select(prep.p, scores32)
    for i, ora in enumerate(prep.ora):
        np.testing.assert_array_equal(idx[i], ora["idx"])


def oracle_row_stats(prep):
    """[U][m][2] fp32 (M_r, L_r) of the full window attention, as grkv_score writes them."""
    return np.stack([np.stack([o["row_max"], o["row_sum"]], -1) for o in prep.ora]).astype(np.float32)


@pytest.mark.parametrize("stats", [False, True], ids=["two_pass", "row_stats"])
@pytest.mark.parametrize("path", ["default", "portable"])
def test_merge_stage(prep, path, stats):
    c, op = prep.case, prep.op
    scores32 = np.stack([o["scores32"] for o in prep.ora])
    y32 = np.stack([o["y"].astype(np.float32) for o in prep.ora])
    idx = np.stack([o["idx"] for o in prep.ora])
    p = G.lib_params(prep.wl, c.U, **prep.over)
    p.flags = PATHS[path]
    ko, vo = G.run_merge(c, p, scores32, y32, idx,
                         row_stats=oracle_row_stats(prep) if stats else None)
    for i in range(c.U):
        ref = O.merge_unit(c.q[i], c.k[i], c.v[i], scores32[i], y32[i], idx[i], op)
        np.testing.assert_array_equal(ko[i], c.k[i][idx[i]])            # K_out = K0
        fixed = ref["fixed"]
        np.testing.assert_array_equal(vo[i][fixed], c.v[i][idx[i]][fixed])  # F rows as V0
        G.assert_values(vo[i], ref["v_out"], c.wl.dtype)


def test_merge_row_stats_far_below_full_max_takes_two_passes(grkv_lib):
    """A key that dominates one window row is left out of the retained set, so
    the retained maximum of that row lies far (more than 64 in log2 units)
    below the full-cache maximum given in row_stats: the one-pass Gram would
    lose that row, and the unit must be recomputed with two passes."""
    wl = gi.workload(1).replace(units=2, n=2048, budget=256, seed=99)
    c = G.Case(wl)
    op = G.oracle_params(wl)
    row, jstar = 5, 300
    qr = c.q[0].reshape(op.m, op.d)[row].astype(np.float64)
    spike = gi.bf16_value(gi.bf16_bits(qr * (3000.0 / float(qr @ qr))))
    c.k[0][jstar] = spike
    c.dk = G.to_device(c.k, wl.dtype)
    ora = [O.compress_unit(c.q[i], c.k[i], c.v[i], op) for i in range(c.U)]
    idx = np.stack([o["idx"] for o in ora])
    P = wl.n - wl.window
    if jstar in idx[0]:
        keep = [j for j in idx[0][: op.budget - op.window] if j != jstar]
        extra = next(j for j in range(op.n_sink, P) if j not in set(idx[0]) and j != jstar)
        idx[0][: op.budget - op.window] = np.sort(np.array(keep + [extra]))
    assert jstar not in idx[0]
    lg = O.window_logits(c.q[0], c.k[0], op)
    gap = (lg[row].max() - lg[row][idx[0]].max()) / math.log(2.0)
    assert gap > 64.0, gap
    scores32 = np.stack([o["scores32"] for o in ora])
    y32 = np.stack([o["y"].astype(np.float32) for o in ora])
    rs = np.stack([np.stack([o["row_max"], o["row_sum"]], -1) for o in ora]).astype(np.float32)
    p = G.lib_params(wl, c.U)
    ko, vo = G.run_merge(c, p, scores32, y32, idx, row_stats=rs)
    for i in range(c.U):
        ref = O.merge_unit(c.q[i], c.k[i], c.v[i], scores32[i], y32[i], idx[i], op)
        np.testing.assert_array_equal(ko[i], c.k[i][idx[i]])
        G.assert_values(vo[i], ref["v_out"], wl.dtype)


def test_compress_end_to_end(prep):
    """grkv_compress on every unit: each unit's retained set, K_out and V_out
    against the oracle (check_unit_end_to_end: no unit is skipped)."""
    c, op = prep.case, prep.op
    idx, ko, vo = G.run_compress(c, prep.p)
    scores, _, _ = G.run_score(c, prep.p)
    for i, ora in enumerate(prep.ora):
        G.check_unit_end_to_end(prep.wl.name, i, c.q[i], c.k[i], c.v[i], op, ora, idx[i],
                                scores[i], ko[i], vo[i], c.wl.dtype)


# ------------------------------------------------------------- edge cases --
EDGE = gi.Workload("edge_n600", 2, 2, 600, 128, 8, 64, 7, 1e-2, "bf16", "lowrank", 4242)


@pytest.mark.parametrize("over", [
    dict(budget=8),                       # B = w: only the window is kept
    dict(budget=600),                     # B = n: nothing evicted, zero update
    dict(pool_kernel=1),
    dict(lambda_v=math.inf),              # values unchanged
    dict(lambda_v=1e6),
    dict(lambda_v=1e-5),
    dict(n_sink=0, beta=0.0),
    dict(beta=0.5, n_sink=64),
], ids=lambda d: ",".join(f"{k}={v}" for k, v in d.items()))
def test_edge_cases(grkv_lib, over):
    wl = EDGE.replace(budget=over.get("budget", EDGE.budget))
    over = {k: v for k, v in over.items() if k != "budget"}
    c = G.Case(wl)
    op = G.oracle_params(wl, **over)
    p = G.lib_params(wl, c.U, **over)
    idx, ko, vo = G.run_compress(c, p)
    for i in range(c.U):
        ora = O.compress_unit(c.q[i], c.k[i], c.v[i], op)
        assert G.idx_tie_check(idx[i], ora, op, G.score_rel_tol(c.q[i], c.k[i], op)) == 0
        G.assert_values(vo[i], ora["v_out"], wl.dtype)
        if wl.budget == wl.n:
            G.assert_values(vo[i], c.v[i].astype(np.float64), wl.dtype, "B = n leaves V")
        if math.isinf(op.lambda_v):
            np.testing.assert_array_equal(vo[i], c.v[i][idx[i]])


def test_select_ties_take_smaller_positions(grkv_lib):
    wl = EDGE
    p = G.lib_params(wl, 2)
    op = G.oracle_params(wl)
    P = wl.n - wl.window
    flat = np.full((2, P), 0.25, np.float32)             # every score tied
    steps = np.repeat(np.arange(P // 8, dtype=np.float32), 8)[:P][None].repeat(2, 0)
    steps = np.concatenate([steps, np.zeros((2, P - steps.shape[1]), np.float32)], 1)
    for s in (flat, steps):
        idx = G.run_select(p, s)
        for i in range(2):
            np.testing.assert_array_equal(idx[i], O.select(O.pool(s[i], op), op))


@pytest.mark.parametrize("n", [32768, 32800, 40032])
@pytest.mark.parametrize("pool", ["max", "avg"])
def test_select_long_prefixes(grkv_lib, n, pool):
    """n - w = 32736 and 32768 take the shared-memory selection kernel, 40000
    the global-memory one; coarse score levels make many ties at the cut."""
    wl = gi.Workload(f"select_n{n}", 2, 4, n, 128, 32, 2048, 7, 1e-2, "bf16", "lowrank", 4242)
    p = G.lib_params(wl, 2, pool_type=pool)
    op = G.oracle_params(wl, pool_type=pool)
    rng = np.random.default_rng(n)
    s = rng.integers(0, 64, size=(2, n - 32)).astype(np.float32) / 64.0
    idx = G.run_select(p, s)
    for i in range(2):
        np.testing.assert_array_equal(idx[i], O.select(O.pool(s[i], op), op))


@pytest.mark.parametrize("path", ["default", "portable"])
def test_merge_reports_out_of_range_idx(grkv_lib, path):
    """An idx entry outside [0, n) is reported as GRKV_ERR_INVALID_ARG in the
    device status and read as position 0 (no out-of-bounds access)."""
    wl = gi.workload(1).replace(units=2, n=2048, budget=256, seed=7)
    c = G.Case(wl)
    op = G.oracle_params(wl)
    ora = [O.compress_unit(c.q[i], c.k[i], c.v[i], op) for i in range(c.U)]
    idx = np.stack([o["idx"] for o in ora]).astype(np.int32)
    idx[0][10] = wl.n + 5
    idx[1][3] = -1
    scores32 = np.stack([o["scores32"] for o in ora])
    y32 = np.stack([o["y"].astype(np.float32) for o in ora])
    p = G.lib_params(wl, c.U)
    p.flags = PATHS[path]
    G.run_merge(c, p, scores32, y32, idx, expect_status=b.GRKV_ERR_INVALID_ARG)


def test_zero_units_is_a_no_op(grkv_lib):
    import torch
    p = b.params(0, 4, 1024, 32, 128)
    ws = torch.empty(1024, dtype=torch.uint8, device="cuda")
    z = torch.empty(16, dtype=torch.bfloat16, device="cuda")
    zi = torch.empty(16, dtype=torch.int32, device="cuda")
    assert b.grkv_compress(p, z, z, z, z, z, zi, ws) == b.GRKV_OK
    assert b.grkv_status(ws) == b.GRKV_OK


def test_singular_dual_system_reports_numeric_status(grkv_lib):
    """lambda = 0 with every retained token fixed: X_G = 0, the dual matrix is
    0 and its first Cholesky pivot is exactly 0; the device reports
    GRKV_ERR_NUMERIC through the status word and the context stays usable."""
    wl = EDGE.replace(budget=EDGE.window)
    c = G.Case(wl)
    p = G.lib_params(wl, c.U, lambda_v=0.0)
    op = G.oracle_params(wl, lambda_v=0.0)
    ora = [O.compress_unit(c.q[i], c.k[i], c.v[i], G.oracle_params(wl)) for i in range(c.U)]
    scores32 = np.stack([o["scores32"] for o in ora])
    y32 = np.stack([o["y"].astype(np.float32) for o in ora])
    idx = np.stack([o["idx"] for o in ora])
    G.run_merge(c, p, scores32, y32, idx, expect_status=b.GRKV_ERR_NUMERIC)
    # the next call on the same context is unaffected
    p2 = G.lib_params(wl, c.U)
    _, vo = G.run_merge(c, p2, scores32, y32, idx)
    assert op.lambda_v == 0.0 and np.isfinite(vo).all()


def _compress_sampled(wl, check_units, flags=0):
    """grkv_compress over every unit of `wl` at full size, in the launch
    configuration the bench times, then grkv_score with the same flags on the
    same inputs; the sampled units against the oracle, each one compared."""
    import torch
    U = wl.units
    q = np.empty((U, wl.group, wl.window, wl.d), np.uint16)
    k = np.empty((U, wl.n, wl.d), np.uint16)
    v = np.empty_like(k)
    gi.fill_units(wl, q, k, v)
    as_dev = lambda x: torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).cuda()
    dq, dk, dv = as_dev(q), as_dev(k), as_dev(v)
    del q, k, v
    p = G.lib_params(wl, U)
    p.flags = flags
    ko = torch.empty((U, wl.budget, wl.d), dtype=torch.bfloat16, device="cuda")
    vo = torch.empty_like(ko)
    idx = torch.empty((U, wl.budget), dtype=torch.int32, device="cuda")
    ws = G.workspace(p)
    b.grkv_compress(p, dq, dk, dv, ko, vo, idx, ws)
    assert b.grkv_status(ws) == b.GRKV_OK
    sel = torch.tensor(list(check_units), dtype=torch.long, device="cuda")
    idx, ko, vo = idx[sel].cpu().numpy(), G.to_host(ko[sel]), G.to_host(vo[sel])
    scores = torch.empty((U, wl.n - wl.window), dtype=torch.float32, device="cuda")
    y = torch.empty((U, wl.m, wl.d), dtype=torch.float32, device="cuda")
    rs = torch.empty((U, wl.m, 2), dtype=torch.float32, device="cuda")
    b.grkv_score(p, dq, dk, dv, scores, y, rs, ws)
    assert b.grkv_status(ws) == b.GRKV_OK
    scores = G.to_host(scores[sel])
    del dq, dk, dv
    torch.cuda.empty_cache()
    op = G.oracle_params(wl)
    for i, u in enumerate(check_units):
        qu, ku, vu = gi.unit_arrays(wl, u)
        ora = O.compress_unit(qu, ku, vu, op)
        G.check_unit_end_to_end(wl.name, u, qu, ku, vu, op, ora, idx[i], scores[i], ko[i],
                                vo[i], wl.dtype)


def test_full_size_c2_sampled_units(grkv_lib):
    """The 32-layer, 32K-token workload (256 units) at full size; eight units
    spread over the layers against the oracle."""
    _compress_sampled(gi.workload(2), (0, 37, 74, 111, 148, 185, 222, 255))


def test_full_size_c2_one_read_scoring(grkv_lib):
    """The one-read scoring path (GRKV_ONE_READ_SCORE: groups of CTAs, K re-read
    from L2) at the full 256-unit size, where every CTA runs many phases."""
    _compress_sampled(gi.workload(2), (0, 131, 255), flags=b.GRKV_ONE_READ_SCORE)


def test_full_size_c3_mistral_128k_sampled_units(grkv_lib):
    """The Mistral-shaped 128K-token workload (256 units, m = 256) at full
    size in its own launch configuration; the first and last KV heads of
    layers 0 and 31 against the oracle."""
    _compress_sampled(gi.workload(3), (0, 7, 248, 255))


@pytest.mark.parametrize("wl", list(gi.sweep_points()), ids=lambda w: f"n{w.n}_b{w.budget}")
def test_full_size_c4_sweep_point(grkv_lib, wl):
    """Every (n, B) point of the batch-4 sweep at full size (32 units): the
    first, a middle and the last unit against the oracle."""
    _compress_sampled(wl, (0, 13, 31))


# --------------------------------------------------------------- key step --
EDGE_KEY = gi.Workload("edge_n600", 2, 2, 600, 128, 8, 64, 7, 1e-2, "bf16", "lowrank", 4242)
# B = 300 with m = 128: the CG products of a unit are split over 4 CTAs with
# 80, 80, 80 and 60 retained columns (a ragged last share)
SPLIT_KEY = gi.Workload("split_b300", 2, 4, 3000, 128, 32, 300, 7, 1e-2, "bf16", "lowrank", 4343)
KEY_CASES = {
    # workload, path flags, lambda_k (1e-2 Llama default, 1e-1 Mistral default)
    "c0_f32_portable": (gi.workload(0), 0, 1e-2),
    "c1_bf16_default": (gi.workload(1).replace(units=2), 0, 1e-1),
    "c1_bf16_portable": (gi.workload(1).replace(units=2), b.GRKV_FORCE_SIMT, 1e-1),
    "edge_bf16_default": (EDGE_KEY, 0, 1e-2),
    "split_ragged_bf16": (SPLIT_KEY, 0, 1e-2),
}


@pytest.mark.parametrize("name", list(KEY_CASES))
def test_key_step(grkv_lib, name):
    """GRKV_UPDATE_K: the key step of Algorithm 1 at t = 0 (App. D.2) run to a
    relative CG residual of 1e-6 in fp32 on the GPU, against the converged
    linearised ridge solution (fp64 CG to 1e-12) of the oracle, on the
    oracle's retained set.  K_out is held to the method's bar; the update
    K_out - K0 to 2e-3 of its norm plus the rounding of K_out to its dtype.
    V_out and the fixed rows of K_out are those of the value step alone."""
    wl, flags, lam = KEY_CASES[name]
    c = G.Case(wl)
    op = G.oracle_params(wl, update_k=True, lambda_k=lam, cg_iters=4000, cg_tol=1e-12)
    ora = [O.compress_unit(c.q[i], c.k[i], c.v[i], op) for i in range(c.U)]
    idx = np.stack([o["idx"] for o in ora]).astype(np.int32)
    scores32 = np.stack([o["scores32"] for o in ora])
    y32 = np.stack([o["y"].astype(np.float32) for o in ora])
    p = G.lib_params(wl, c.U)
    p.flags = flags
    ko0, vo0 = G.run_merge(c, p, scores32, y32, idx)
    p.flags = flags | b.GRKV_UPDATE_K
    p.lambda_k = lam
    p.cg_iters = 4000
    p.cg_tol = 1e-6
    ko, vo = G.run_merge(c, p, scores32, y32, idx)
    np.testing.assert_array_equal(vo, vo0)
    rnd = 2.0 ** -8 if wl.dtype == "bf16" else 2.0 ** -23
    for i, o in enumerate(ora):
        K0 = c.k[i][idx[i]].astype(np.float64)
        fixed = o["fixed"]
        np.testing.assert_array_equal(ko[i][fixed], ko0[i][fixed])
        G.assert_values(ko[i], o["k_out"], wl.dtype, what="k_out")
        d_ora = o["k_out"] - K0
        d_gpu = ko[i].astype(np.float64) - K0
        assert np.abs(d_ora).max() > 0
        err = np.linalg.norm(d_gpu - d_ora)
        lim = 2e-3 * np.linalg.norm(d_ora) + rnd * np.linalg.norm(o["k_out"])
        assert err <= lim, f"unit {i}: key update error {err:.3e} > {lim:.3e}"


@pytest.mark.parametrize("name,steps", [("c0_f32_portable", 2), ("c0_f32_portable", 3),
                                        ("c1_bf16_default", 2), ("edge_bf16_default", 3)])
def test_alternation_steps(grkv_lib, name, steps):
    """S > 1 (Algorithm 1's outer loop): step t re-runs the value step from V0
    with X at the current keys K^(t), then the key step linearised at K^(t),
    against the oracle's alternation (fp64, CG to 1e-12) run for the same S
    with the stop test off.  K_out and V_out are held to the method's bar;
    fixed rows keep K0 and V0 bit for bit."""
    wl, flags, lam = KEY_CASES[name]
    c = G.Case(wl)
    op = G.oracle_params(wl, update_k=True, lambda_k=lam, cg_iters=4000, cg_tol=1e-12)
    ora = [O.compress_unit(c.q[i], c.k[i], c.v[i], G.oracle_params(wl)) for i in range(c.U)]
    idx = np.stack([o["idx"] for o in ora]).astype(np.int32)
    scores32 = np.stack([o["scores32"] for o in ora])
    y32 = np.stack([o["y"].astype(np.float32) for o in ora])
    p = G.lib_params(wl, c.U)
    p.flags = flags | b.GRKV_UPDATE_K
    p.lambda_k = lam
    p.cg_iters = 4000
    p.cg_tol = 1e-6
    p.steps = steps
    p.step_tol = 0.0
    ko, vo = G.run_merge(c, p, scores32, y32, idx)
    for i, o in enumerate(ora):
        alt = O.alternate(c.q[i], c.k[i], c.v[i], scores32[i], o["y"], idx[i], op, steps, stop=0.0)
        assert len(alt["deltas"]) == steps
        fixed = alt["fixed"]
        np.testing.assert_array_equal(ko[i][fixed], c.k[i][idx[i]][fixed])
        np.testing.assert_array_equal(vo[i][fixed], c.v[i][idx[i]][fixed])
        G.assert_values(ko[i], alt["k_out"], wl.dtype, what=f"k_out (S = {steps})")
        G.assert_values(vo[i], alt["v_out"], wl.dtype, what=f"v_out (S = {steps})")


def test_key_step_zero_iterations_and_large_lambda(grkv_lib):
    wl = gi.workload(1).replace(units=1)
    c = G.Case(wl)
    op = G.oracle_params(wl)
    o = O.compress_unit(c.q[0], c.k[0], c.v[0], op)
    args = (o["scores32"][None], o["y"].astype(np.float32)[None], o["idx"][None].astype(np.int32))
    p = G.lib_params(wl, 1)
    ko0, _ = G.run_merge(c, p, *args)
    p.flags = b.GRKV_UPDATE_K
    p.cg_iters = 0                      # alpha = 0: K_out = K0 exactly
    ko, _ = G.run_merge(c, p, *args)
    np.testing.assert_array_equal(ko, ko0)
    p.cg_iters = 64
    p.lambda_k = 1e7                    # the ridge keeps K0 (update far below a bf16 ulp)
    ko, _ = G.run_merge(c, p, *args)
    np.testing.assert_array_equal(ko, ko0)


def test_key_step_through_compress(grkv_lib):
    """grkv_compress with GRKV_UPDATE_K runs the key step on its own selection
    and target: K_out differs from K0 on free slots only."""
    wl = EDGE_KEY
    c = G.Case(wl)
    p = G.lib_params(wl, c.U)
    idx0, ko0, vo0 = G.run_compress(c, p)
    p.flags = b.GRKV_UPDATE_K
    idx, ko, vo = G.run_compress(c, p)
    np.testing.assert_array_equal(idx, idx0)
    np.testing.assert_array_equal(vo, vo0)
    for i in range(c.U):
        np.testing.assert_array_equal(ko0[i], c.k[i][idx0[i]])
        assert (ko[i] != ko0[i]).any()


# ---------------------------------------------------------- deterministic --
@pytest.mark.parametrize("wl", [gi.workload(1), gi.workload(2).replace(units=3, n=8192, budget=1024),
                                M256], ids=["c1", "c2_recipe_n8192", "m256_spans"])
def test_deterministic_mode_is_bitwise_reproducible(grkv_lib, wl):
    """GRKV_DETERMINISTIC: two calls give bit-identical Y, scores, row
    statistics and compressed caches, and the results still match the oracle."""
    c = G.Case(wl)
    p = G.lib_params(wl, c.U)
    p.flags = b.GRKV_DETERMINISTIC
    s1, y1, r1 = G.run_score(c, p)
    s2, y2, r2 = G.run_score(c, p)
    np.testing.assert_array_equal(y1, y2)
    np.testing.assert_array_equal(s1, s2)
    np.testing.assert_array_equal(r1, r2)
    i1, k1, v1 = G.run_compress(c, p)
    i2, k2, v2 = G.run_compress(c, p)
    np.testing.assert_array_equal(i1, i2)
    np.testing.assert_array_equal(k1, k2)
    np.testing.assert_array_equal(v1, v2)
    op = G.oracle_params(wl)
    for i in range(c.U):
        ora = O.compress_unit(c.q[i], c.k[i], c.v[i], op)
        tol = G.score_rel_tol(c.q[i], c.k[i], op)
        s_abs = ora["attn"] @ np.abs(c.v[i].astype(np.float64))
        lim = (tol + op.n * G.U + G.y_tol_extra(p)) * s_abs + 1e-7
        assert (np.abs(y1[i] - ora["y"]) <= lim).all()
        G.check_unit_end_to_end(wl.name + "_deterministic", i, c.q[i], c.k[i], c.v[i], op, ora,
                                i1[i], s1[i], k1[i], v1[i], wl.dtype)


# ------------------------------------------------------ bounded-wait exit --
@pytest.mark.parametrize("path", ["default", "one_read"])
def test_bounded_wait_timeout_exits_cleanly(grkv_lib, path):
    """GRKV_TEST_TIMEOUT makes the scoring kernel's first CTA withhold one
    arrive with a ~2 ms wait budget: its waits expire, every role of the CTA
    (and of the CTAs that wait for its statistics) gives up, the kernel frees
    its tensor memory and returns, and the status word reads
    GRKV_ERR_TIMEOUT.  The next calls on the same context run normally (they
    allocate tensor memory on every SM again) and match the oracle."""
    import torch
    wl = gi.workload(1)
    c = G.Case(wl)
    p = G.lib_params(wl, c.U)
    p.flags = b.GRKV_TEST_TIMEOUT | PATHS[path]
    m, P = wl.m, wl.n - wl.window
    scores = torch.empty((c.U, P), dtype=torch.float32, device="cuda")
    y = torch.empty((c.U, m, 128), dtype=torch.float32, device="cuda")
    rs = torch.empty((c.U, m, 2), dtype=torch.float32, device="cuda")
    ws = G.workspace(p)
    b.grkv_score(p, c.dq, c.dk, c.dv, scores, y, rs, ws)
    assert b.grkv_status(ws) == b.GRKV_ERR_TIMEOUT
    torch.cuda.synchronize()
    op = G.oracle_params(wl)
    for flags in (b.GRKV_ONE_READ_SCORE, 0):
        p.flags = flags
        s2, _, _ = G.run_score(c, p)
        for i in range(c.U):
            ora = O.compress_unit(c.q[i], c.k[i], c.v[i], op)
            G.assert_scores(s2[i], ora["scores"], G.score_rel_tol(c.q[i], c.k[i], op))


# ---------------------------------------------------------- GRKV_CHECKS --
def test_checks_flag_reports_bad_arguments(grkv_lib):
    """GRKV_CHECKS: valid calls report GRKV_OK; an idx that is not ascending or
    lacks the window in its last w slots reports GRKV_ERR_BOUNDS; a non-finite
    key reports GRKV_ERR_INVALID_ARG (device-side checks, status word)."""
    import torch
    wl = gi.workload(1).replace(units=2, n=2048, budget=256, seed=7)
    c = G.Case(wl)
    op = G.oracle_params(wl)
    ora = [O.compress_unit(c.q[i], c.k[i], c.v[i], op) for i in range(c.U)]
    idx = np.stack([o["idx"] for o in ora]).astype(np.int32)
    scores32 = np.stack([o["scores32"] for o in ora])
    y32 = np.stack([o["y"].astype(np.float32) for o in ora])
    p = G.lib_params(wl, c.U)
    p.flags = b.GRKV_CHECKS
    G.run_compress(c, p)
    _, vo = G.run_merge(c, p, scores32, y32, idx)
    for i in range(c.U):
        G.assert_values(vo[i], ora[i]["v_out"], wl.dtype)
    swapped = idx.copy()
    swapped[0][[10, 11]] = swapped[0][[11, 10]]
    G.run_merge(c, p, scores32, y32, swapped, expect_status=b.GRKV_ERR_BOUNDS)
    no_window = idx.copy()
    no_window[1][-1] = wl.n - wl.window - 1
    G.run_merge(c, p, scores32, y32, no_window, expect_status=b.GRKV_ERR_BOUNDS)
    c.dk[1, 17, 5] = float("nan")
    ko = torch.empty((c.U, wl.budget, 128), dtype=torch.bfloat16, device="cuda")
    vo2 = torch.empty_like(ko)
    idx_out = torch.empty((c.U, wl.budget), dtype=torch.int32, device="cuda")
    ws = G.workspace(p)
    b.grkv_compress(p, c.dq, c.dk, c.dv, ko, vo2, idx_out, ws)
    assert b.grkv_status(ws) == b.GRKV_ERR_INVALID_ARG

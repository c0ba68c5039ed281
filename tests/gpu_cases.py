"""Helpers of the GPU parity tests: seeded cases, C-ABI calls, tolerances.

Tolerances follow from the arithmetic of the CUDA path (fp32 accumulation of
exact bf16 or fp32 products, fp32 exponentials):
  * a logit l = s * sum_t q_t k_t accumulated in fp32 over d terms is off by
    at most s * gamma_d * sum_t |q_t k_t|, gamma_d = d u / (1 - d u), u = 2^-24;
  * a probability exp(l - M) / L then has relative error <= 2 * that bound
    (its own logit and the row log-normaliser) plus a few ulps of exp/divide;
  * a prefix score is a sum of m such probabilities: add m u.
The merged values are held to the bar of the method's statement: for every
retained row, max |gpu - oracle| / ||oracle row||_2 <= 1e-4 (fp32 inputs) or
2e-2 (bf16 inputs).
"""
from __future__ import annotations

import math

import numpy as np
import torch

import grkv_inputs as gi
import oracle as O
from paper_2605_31105_gb300 import binding as b

U = 2.0 ** -24
V_TOL = {"f32": 1e-4, "bf16": 2e-2}


def oracle_params(wl: gi.Workload, **over) -> O.Params:
    kw = dict(group=wl.group, n=wl.n, d=wl.d, window=wl.window, budget=wl.budget,
              pool_kernel=wl.pool_kernel, lambda_v=wl.lambda_v)
    kw.update(over)
    return O.Params(**kw)


def uses_tensor_cores(p) -> bool:
    """The library scores on the tensor cores for bf16 with m <= 256."""
    return (p.dtype == b.GRKV_BF16 and p.group * p.window <= 256
            and not (p.flags & b.GRKV_FORCE_SIMT))


def y_tol_extra(p) -> float:
    """The tensor-core path rounds P to bf16 before Y = P V: relative 2^-9
    per term, counted as 2^-8."""
    return 2.0 ** -8 if uses_tensor_cores(p) else 0.0


def lib_params(wl: gi.Workload, units: int, **over) -> b.grkv_params:
    p = b.params(units, wl.group, wl.n, wl.window, wl.budget, pool_kernel=wl.pool_kernel,
                 lambda_v=wl.lambda_v, dtype=wl.dtype)
    for key, val in over.items():
        if key == "pool_type":
            val = {"max": b.GRKV_POOL_MAX, "avg": b.GRKV_POOL_AVG}[val]
        if key == "causal":
            val = int(val)
        setattr(p, key, val)
    return p


def to_device(x: np.ndarray, dtype: str) -> torch.Tensor:
    if dtype == "bf16":
        return torch.from_numpy(gi.bf16_bits(x).view(np.int16)).view(torch.bfloat16).cuda()
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).cuda()


def to_host(t: torch.Tensor) -> np.ndarray:
    return t.float().cpu().numpy()


class Case:
    """Seeded inputs of some units of a workload, on the host and the device."""

    def __init__(self, wl: gi.Workload, units=None):
        self.wl = wl
        self.units = list(range(wl.units)) if units is None else list(units)
        arrs = [gi.unit_arrays(wl, u) for u in self.units]
        self.q = np.stack([a[0] for a in arrs])
        self.k = np.stack([a[1] for a in arrs])
        self.v = np.stack([a[2] for a in arrs])
        self.dq = to_device(self.q, wl.dtype)
        self.dk = to_device(self.k, wl.dtype)
        self.dv = to_device(self.v, wl.dtype)

    @property
    def U(self):
        return len(self.units)


def workspace(p) -> torch.Tensor:
    """A workspace filled with a NaN byte pattern, so a kernel that reads a
    workspace byte it did not write first cannot pass by luck."""
    return torch.full((max(256, b.grkv_workspace_size(p)),), 0xFF, dtype=torch.uint8,
                      device="cuda")


def run_score(c: Case, p):
    m, P = p.group * p.window, p.n - p.window
    scores = torch.empty((c.U, P), dtype=torch.float32, device="cuda")
    y = torch.empty((c.U, m, 128), dtype=torch.float32, device="cuda")
    rs = torch.empty((c.U, m, 2), dtype=torch.float32, device="cuda")
    ws = workspace(p)
    b.grkv_score(p, c.dq, c.dk, c.dv, scores, y, rs, ws)
    assert b.grkv_status(ws) == b.GRKV_OK
    return to_host(scores), to_host(y), to_host(rs)


def run_select(p, scores: np.ndarray):
    d_scores = torch.from_numpy(np.ascontiguousarray(scores, dtype=np.float32)).cuda()
    idx = torch.empty((scores.shape[0], p.budget), dtype=torch.int32, device="cuda")
    ws = workspace(p)
    b.grkv_select(p, d_scores, idx, ws)
    assert b.grkv_status(ws) == b.GRKV_OK
    return idx.cpu().numpy()


def _out_dtype(c: Case):
    return torch.bfloat16 if c.wl.dtype == "bf16" else torch.float32


def run_merge(c: Case, p, scores, y, idx, expect_status=b.GRKV_OK, row_stats=None):
    ko = torch.empty((c.U, p.budget, 128), dtype=_out_dtype(c), device="cuda")
    vo = torch.empty_like(ko)
    ws = workspace(p)
    rs = None
    if row_stats is not None:
        rs = torch.from_numpy(np.ascontiguousarray(row_stats, np.float32)).cuda()
    b.grkv_merge(p, c.dq, c.dk, c.dv,
                 torch.from_numpy(np.ascontiguousarray(scores, np.float32)).cuda(),
                 torch.from_numpy(np.ascontiguousarray(y, np.float32)).cuda(),
                 torch.from_numpy(np.ascontiguousarray(idx, np.int32)).cuda(), ko, vo, ws,
                 row_stats=rs)
    assert b.grkv_status(ws) == expect_status
    return to_host(ko), to_host(vo)


def run_compress(c: Case, p):
    ko = torch.empty((c.U, p.budget, 128), dtype=_out_dtype(c), device="cuda")
    vo = torch.empty_like(ko)
    idx = torch.empty((c.U, p.budget), dtype=torch.int32, device="cuda")
    ws = workspace(p)
    b.grkv_compress(p, c.dq, c.dk, c.dv, ko, vo, idx, ws)
    assert b.grkv_status(ws) == b.GRKV_OK
    return idx.cpu().numpy(), to_host(ko), to_host(vo)


# ----------------------------------------------------------------- bounds --
def logit_bound(q, k, op: O.Params) -> float:
    """s * gamma_d * max_{r,j} sum_t |q_rt k_jt|: worst fp32 error of a logit."""
    Q = np.abs(q.reshape(op.m, op.d)).astype(np.float64)
    K = np.abs(k).astype(np.float64)
    gam = op.d * U / (1 - op.d * U)
    return O.effective_scale(op) * gam * float((Q @ K.T).max())


def score_rel_tol(q, k, op: O.Params) -> float:
    return 2.0 * logit_bound(q, k, op) + (op.m + 8) * U + 1e-6


def assert_scores(gpu, ora, tol_rel, what="scores"):
    err = np.abs(gpu.astype(np.float64) - ora)
    lim = tol_rel * np.abs(ora) + 1e-30
    bad = err > lim
    assert not bad.any(), (f"{what}: {bad.sum()} of {bad.size} beyond tolerance; worst rel "
                           f"{(err / np.maximum(np.abs(ora), 1e-30)).max():.3e} vs {tol_rel:.3e}")


def assert_values(gpu, ora, dtype: str, what="v_out"):
    """max_j ||gpu_j - ora_j||_inf / ||ora_j||_2 within the method's bar."""
    den = np.maximum(np.linalg.norm(ora, axis=-1), 1e-30)
    rel = np.abs(gpu.astype(np.float64) - ora).max(axis=-1) / den
    assert rel.max() <= V_TOL[dtype], f"{what}: max row-relative error {rel.max():.3e}"
    return float(rel.max())


def idx_tie_check(gpu_idx, ora, op: O.Params, tol_rel: float):
    """Retained sets must agree except where the oracle's pooled scores sit
    within the score tolerance of the cut: returns the number of such swaps."""
    return tie_stats(gpu_idx, ora, op, tol_rel)["swaps"]


def tie_stats(gpu_idx, ora, op: O.Params, tol_rel: float) -> dict:
    """Positions where the GPU's retained set differs from the oracle's.

    Each differing position must be a prefix position whose oracle pooled
    score lies within 2 * tol_rel (the derived bound on the GPU's score error,
    counted for both scores of a swapped pair) of the cut, the (B - w)-th
    largest pooled score.  Returns the number of swapped pairs and the largest
    relative gap |pooled_j - cut| / cut among them, so that swaps beyond the
    1e-6 tie width can be reported."""
    g, o = set(gpu_idx.tolist()), set(ora["idx"].tolist())
    diff = sorted(g ^ o)
    out = {"swaps": len(diff) // 2, "max_gap": 0.0, "bound": 2 * tol_rel}
    if not diff:
        return out
    pooled = ora["pooled"].astype(np.float64)
    kk = op.budget - op.window
    cut = np.sort(pooled)[::-1][kk - 1]
    for j in diff:
        assert j < op.n - op.window, f"window position {j} differs"
        gap = abs(pooled[j] - cut) / cut
        assert gap <= 2 * tol_rel, \
            f"idx differs at {j}: pooled {pooled[j]:.9e} vs cut {cut:.9e} (gap {gap:.2e})"
        out["max_gap"] = max(out["max_gap"], gap)
    return out


# Records of every end-to-end unit check in this session (workload, unit,
# swaps, largest gap, fixed-set agreement, value error), printed by the test
# session's terminal summary.
SWAP_LOG: list = []


def check_unit_end_to_end(name: str, u: int, q, k, v, op: O.Params, ora: dict, gpu_idx,
                          gpu_scores, k_out, v_out, dtype: str) -> dict:
    """One unit of a grkv_compress run against the oracle, with no unit skipped.

    1. The GPU's prefix scores (grkv_score with the same flags, on the same
       inputs) lie within the derived tolerance of the oracle's.
    2. The GPU's retained set is exactly the oracle's selection on the GPU's
       own fp32 scores: selection is exact, so any difference from the
       oracle's retained set comes from score rounding alone.
    3. Differences from the oracle's retained set sit within the derived
       bound of the cut (tie_stats); their count and largest gap are logged.
    4. K_out = K[idx] bit for bit, and V_out is within the method's bar of
       the oracle's merge (Algorithm 1 value step, fp64, its own target Y)
       re-run on the GPU's retained set, with the fixed set decided on the
       GPU's fp32 scores (both sides decide integers in fp32)."""
    tol = score_rel_tol(q, k, op)
    assert_scores(gpu_scores, ora["scores"], tol, f"{name} unit {u} scores")
    np.testing.assert_array_equal(gpu_idx, O.select(O.pool(gpu_scores, op), op),
                                  err_msg=f"{name} unit {u}: selection on the GPU's scores")
    ts = tie_stats(gpu_idx, ora, op, tol)
    np.testing.assert_array_equal(k_out, k[gpu_idx])
    ref = O.merge_unit(q, k, v, gpu_scores, ora["y"], gpu_idx, op)
    fixed_same = bool(np.array_equal(ref["fixed"], O.fixed_set(gpu_idx, ora["scores32"], op)))
    err = assert_values(v_out, ref["v_out"], dtype, f"{name} unit {u} v_out")
    rec = {"workload": name, "unit": u, "swaps": ts["swaps"], "max_gap": ts["max_gap"],
           "bound": ts["bound"], "fixed_same": fixed_same, "v_err": err}
    SWAP_LOG.append(rec)
    return rec

"""Plain fp64 CPU oracle of GRKV's prefill-time KV compression path.

TEST INFRASTRUCTURE ONLY.  This package is the parity reference for the CUDA
library.  Only the test suite, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` may import it; the library never does, and it
shares no code with the library.  Every function is a direct, slow
restatement of the definition it cites (GRKV, arXiv 2605.31105), computed in
float64 from the exact input values.  Library primitives (matmul, Cholesky,
triangular solve, sort) serve as single steps; nothing is blocked, fused or
reordered beyond what the definition states.

Notation (one unit = one layer x KV head):
    q  [g][w][d]  window queries of the g query heads that share the KV head;
                  stacked row r = h*w + a, query position p_a = n - w + a
    k, v [n][d]   full key / value cache
    m = g*w       stacked window rows
    B             budget, window included

Readings where the paper is silent (each is a parameter here):
    * causal=True: window query a sees keys j <= n - w + a (its prefill
      attention); causal=False is the literal softmax over all n keys.
    * the per-key score is the sum over all m stacked rows of the window
      attention probabilities (sum and mean rank identically).
    * pooling runs over the n - w prefix scores only; max pool ignores
      out-of-range cells, avg pool zero-pads with divisor k.
    * selection keeps the B - w best pooled prefix scores, ties to the smaller
      index, then appends the window; idx is ascending.
    * decisions that turn floats into indices (pooling, selection, fixed
      set) are taken on fp32 scores, the precision the CUDA path stores them
      in; everything else stays fp64.
    * fixed set F = retained sinks (j < n_sink) U window U the floor(beta*B)
      retained prefix non-sink tokens with the largest unpooled score.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np
import scipy.linalg

__all__ = [
    "Params", "effective_scale", "window_logits", "softmax_rows", "window_attention",
    "target", "column_scores", "pool", "select", "fixed_set", "retained_attention",
    "value_step_dual", "value_step_primal", "key_jvp", "key_vjp", "key_step_dual",
    "alternate", "merge_unit", "compress_unit", "cache_output", "transfer_check", "l_common",
]

f64 = np.float64


@dataclasses.dataclass(frozen=True)
class Params:
    group: int
    n: int
    d: int
    window: int
    budget: int
    pool_kernel: int = 7
    pool_type: str = "max"        # "max" | "avg"
    n_sink: int = 4
    beta: float = 0.10
    lambda_v: float = 1e-2
    scale: float = 0.0            # 0 -> fp32(1/sqrt(d))
    causal: bool = True
    update_k: bool = False        # also run the key step (App. D.2)
    lambda_k: float = 1e-2
    cg_iters: int = 512           # most conjugate-gradient iterations of the key step
    cg_tol: float = 1e-4          # ... stopping once ||r|| <= cg_tol ||e||

    @property
    def m(self) -> int:
        return self.group * self.window


def effective_scale(p: Params) -> float:
    """Logit scale 1/sqrt(d) (Sec. 3.1), as the fp32 value the library uses."""
    s = p.scale if p.scale != 0.0 else 1.0 / math.sqrt(p.d)
    return float(np.float32(s))


def _mask(p: Params, cols: np.ndarray) -> np.ndarray:
    """True where stacked row r may attend to key position cols[j]."""
    m, w, n = p.m, p.window, p.n
    if not p.causal:
        return np.ones((m, cols.size), dtype=bool)
    a = np.arange(m) % w                       # window slot of row r
    last_visible = n - w + a                   # query position of row r
    return cols[None, :] <= last_visible[:, None]


def window_logits(q, k, p: Params, cols=None) -> np.ndarray:
    """l_rj = s * q_r . k_j for the stacked window rows (Eq. 4, inside the
    softmax); masked entries are -inf.  `cols` are the key positions of the
    rows of k (default 0..n-1)."""
    Q = np.asarray(q, dtype=f64).reshape(p.m, p.d)
    K = np.asarray(k, dtype=f64)
    cols = np.arange(K.shape[0]) if cols is None else np.asarray(cols)
    lg = effective_scale(p) * (Q @ K.T)
    lg[~_mask(p, cols)] = -np.inf
    return lg


def softmax_rows(lg: np.ndarray):
    """Row softmax with its max M_r and normaliser L_r = sum_j exp(l_rj - M_r)."""
    M = lg.max(axis=1)
    E = np.exp(lg - M[:, None])
    L = E.sum(axis=1)
    return E / L[:, None], M, L


def window_attention(q, k, p: Params):
    """A_win^full = softmax(Q_win K_full^T / sqrt(d)) (Eq. 4); returns (A, M, L)."""
    return softmax_rows(window_logits(q, k, p))


def target(A: np.ndarray, v) -> np.ndarray:
    """Y = A_win^full V_full, the regression target (Sec. 3.4, Algorithm 1)."""
    return A @ np.asarray(v, dtype=f64)


def column_scores(A: np.ndarray, p: Params) -> np.ndarray:
    """SnapKV-style per-key score (Sec. 1-2: window attention aggregated per
    key): c_j = sum_r A_rj for the prefix keys j < n - w."""
    return A[:, : p.n - p.window].sum(axis=0)


def pool(c32: np.ndarray, p: Params) -> np.ndarray:
    """1-D pooling of the fp32 prefix scores with an odd kernel k (SnapKV's
    span pooling).  Max: max over in-range neighbours |t - j| <= k//2.  Avg:
    left-to-right fp64 sum of the in-range neighbours (zero padding), / k,
    rounded to fp32."""
    c = np.asarray(c32, dtype=np.float32)
    P, h = c.size, p.pool_kernel // 2
    if p.pool_type == "max":
        out = c.copy()
        for t in range(1, min(h, P - 1) + 1):
            out[:-t] = np.maximum(out[:-t], c[t:])     # neighbour j + t
            out[t:] = np.maximum(out[t:], c[:-t])      # neighbour j - t
        return out
    acc = np.zeros(P, dtype=f64)
    for t in range(-h, h + 1):                 # left to right over the window
        sh = np.zeros(P, dtype=f64)
        if t < 0 and -t < P:
            sh[-t:] = c[: P + t]
        elif t >= 0 and t < P:
            sh[: P - t] = c[t:]
        acc += sh
    return (acc / f64(p.pool_kernel)).astype(np.float32)


def select(pooled32: np.ndarray, p: Params) -> np.ndarray:
    """Retained set: the B - w largest pooled prefix scores (ties: smaller
    index first), sorted ascending, followed by the window n-w..n-1."""
    P, kk = p.n - p.window, p.budget - p.window
    j = np.arange(P)
    order = np.lexsort((j, -np.asarray(pooled32, dtype=f64)))
    keep = np.sort(order[:kk])
    return np.concatenate([keep, np.arange(P, p.n)]).astype(np.int32)


def fixed_set(idx: np.ndarray, c32: np.ndarray, p: Params) -> np.ndarray:
    """Fixed tokens F (Sec. 3.4 'fixed tokens', App. D.3): retained sinks,
    the window, and the floor(beta * B) retained prefix non-sink tokens with
    the highest unpooled score (ties: smaller index).  Returns a bool mask over
    the B retained slots."""
    idx = np.asarray(idx)
    P = p.n - p.window
    fixed = (idx < p.n_sink) | (idx >= P)
    cand = np.nonzero(~fixed)[0]
    n_fix = min(int(math.floor(f64(np.float32(p.beta)) * p.budget)), cand.size)
    if n_fix > 0:
        cj = np.asarray(c32, dtype=np.float32)[idx[cand]].astype(f64)
        order = np.lexsort((idx[cand], -cj))
        fixed[cand[order[:n_fix]]] = True
    return fixed


def retained_attention(q, k, idx, p: Params):
    """X = softmax(Q_win K_Ret^T / sqrt(d)) over the retained keys only
    (Algorithm 1, value step; Sec. 3.4), same causal rule as the target."""
    K0 = np.asarray(k, dtype=f64)[idx]
    X, _, _ = softmax_rows(window_logits(q, K0, p, cols=np.asarray(idx)))
    return X


def value_step_dual(X, Y, V0, free, lam: float):
    """Value step in dual (Woodbury) form (Sec. 3.4 'Dual solution', App. D.1,
    with the fixed-token restriction of App. D.3):
        R_V = Y - X_F V0_F - X_G V0_G
        Z   = (X_G X_G^T + lambda I_m)^-1 R_V       (Cholesky solve)
        V*_G = V0_G + X_G^T Z,  V*_F = V0_F."""
    X = np.asarray(X, dtype=f64)
    V0 = np.asarray(V0, dtype=f64)
    free = np.asarray(free, dtype=bool)
    XG = X[:, free]
    R = np.asarray(Y, dtype=f64) - X[:, ~free] @ V0[~free] - XG @ V0[free]
    N = XG @ XG.T + lam * np.eye(X.shape[0])
    Z = scipy.linalg.cho_solve(scipy.linalg.cho_factor(N, lower=True), R)
    out = V0.copy()
    out[free] = V0[free] + XG.T @ Z
    return out


def value_step_primal(X, Y, V0, free, lam: float):
    """Value step in primal form, Eq. 7 restricted to the free tokens (App. D.3):
        V*_G = (X_G^T X_G + lambda I)^-1 (X_G^T Y_G + lambda V0_G),
        Y_G  = Y - X_F V0_F,   V*_F = V0_F."""
    X = np.asarray(X, dtype=f64)
    V0 = np.asarray(V0, dtype=f64)
    free = np.asarray(free, dtype=bool)
    XG = X[:, free]
    YG = np.asarray(Y, dtype=f64) - X[:, ~free] @ V0[~free]
    M = XG.T @ XG + lam * np.eye(XG.shape[1])
    out = V0.copy()
    out[free] = np.linalg.solve(M, XG.T @ YG + lam * V0[free])
    return out


def key_jvp(X, Q, V, dK, s: float):
    """Directional derivative of f(K) = softmax(s Q K^T) V at the K whose
    (masked) retained attention is X, in direction dK (App. D.2, the
    Jacobian-vector product J[dK]):
        dS = s Q dK^T,  dA = X o (dS - rowsum(X o dS)),  df = dA V.
    Masked entries have X = 0 and contribute nothing."""
    X = np.asarray(X, dtype=f64)
    dS = s * (np.asarray(Q, dtype=f64) @ np.asarray(dK, dtype=f64).T)
    dA = X * (dS - (X * dS).sum(axis=1, keepdims=True))
    return dA @ np.asarray(V, dtype=f64)


def key_vjp(X, Q, V, W, s: float):
    """Adjoint of `key_jvp` (App. D.2, the vector-Jacobian product J^T[W]):
        dA = W V^T,  dS = X o (dA - rowsum(X o dA)),  dK = s dS^T Q."""
    X = np.asarray(X, dtype=f64)
    dA = np.asarray(W, dtype=f64) @ np.asarray(V, dtype=f64).T
    dS = X * (dA - (X * dA).sum(axis=1, keepdims=True))
    return s * (dS.T @ np.asarray(Q, dtype=f64))


def key_step_dual(X, Q, K0, V, Y, free, lam: float, s: float, iters: int, tol: float = 0.0,
                  K=None):
    """Key step of Algorithm 1 in its linearised dual form (Sec. 3.4 'Key
    step', App. D.2), linearised at the current keys K (default K0, the
    t = 0 case, where G = 0) whose retained attention is X:
        E = Y - f(K) = Y - X V,  e = vec(E),  g = vec(G),  G = K - K0
        alpha = (J_G J_G^T + lambda_k I)^-1 (e + J_G g)  (conjugate gradients)
        K*_G = K0_G + unvec(J_G^T alpha),  K*_F = K0_F
    J_G is the Jacobian of f at K with respect to the free rows only; the operator
    alpha -> J_G (J_G^T alpha) + lambda alpha is applied matrix-free (JVP of
    the VJP), as the paper does.  CG starts from alpha = 0 and runs at most
    `iters` iterations, stopping once ||r_t|| <= tol ||e|| or the search
    direction vanishes; returns K* and the residual norms ||r_t|| of every
    iteration."""
    X = np.asarray(X, dtype=f64)
    V = np.asarray(V, dtype=f64)
    K0 = np.asarray(K0, dtype=f64)
    free = np.asarray(free, dtype=bool)

    def jt(W):
        dK = key_vjp(X, Q, V, W, s)
        dK[~free] = 0.0
        return dK

    def op(a):
        return key_jvp(X, Q, V, jt(a), s) + lam * a

    E = np.asarray(Y, dtype=f64) - X @ V
    if K is not None:
        G = np.asarray(K, dtype=f64) - K0
        G[~free] = 0.0
        E = E + key_jvp(X, Q, V, G, s)
    alpha = np.zeros_like(E)
    r = E.copy()
    pdir = r.copy()
    rs = float((r * r).sum())
    hist = [math.sqrt(rs)]
    stop = (tol * hist[0]) ** 2
    for _ in range(iters):
        if rs == 0.0 or rs <= stop:
            break
        Ap = op(pdir)
        pAp = float((pdir * Ap).sum())
        if not pAp > 0.0:       # the direction has vanished: converged
            break
        a = rs / pAp
        alpha += a * pdir
        r -= a * Ap
        rs_new = float((r * r).sum())
        hist.append(math.sqrt(rs_new))
        pdir = r + (rs_new / rs) * pdir
        rs = rs_new
    K = K0.copy()
    K[free] = K0[free] + jt(alpha)[free]
    return K, hist


def alternate(q, k, v, c32, y, idx, p: Params, steps: int, stop: float = 1e-9):
    """Algorithm 1 with S = `steps` alternating value / key steps (NEXT rows:
    multi-step alternation), each linearised at the current keys:
        X = softmax over the retained keys K^(t)
        V^(t+1) = value step from V0 with that X (fixed rows keep V0)
        K^(t+1) = key step at K^(t) against V^(t+1), G = K^(t) - K0
    stopping once max(||K^(t+1) - K^(t)||_inf, ||V^(t+1) - V^(t)||_inf) <= stop.
    Returns K, V, the fixed mask and the (delta_K, delta_V) of every step."""
    idx = np.asarray(idx)
    K0 = np.asarray(k, dtype=f64)[idx]
    V0 = np.asarray(v, dtype=f64)[idx]
    fixed = fixed_set(idx, c32, p)
    Q = np.asarray(q, dtype=f64).reshape(p.m, p.d)
    s = effective_scale(p)
    lam_v, lam_k = f64(np.float32(p.lambda_v)), f64(np.float32(p.lambda_k))
    K, V = K0.copy(), V0.copy()
    deltas = []
    for _ in range(steps):
        X, _, _ = softmax_rows(window_logits(q, K, p, cols=idx))
        Vn = value_step_dual(X, y, V0, ~fixed, lam_v)
        Kn, _ = key_step_dual(X, Q, K0, Vn, y, ~fixed, lam_k, s, p.cg_iters, p.cg_tol, K=K)
        deltas.append((float(np.abs(Kn - K).max()), float(np.abs(Vn - V).max())))
        K, V = Kn, Vn
        if max(deltas[-1]) <= stop:
            break
    return {"k_out": K, "v_out": V, "fixed": fixed, "deltas": deltas}


def merge_unit(q, k, v, c32, y, idx, p: Params, mode: str = "dual"):
    """Algorithm 1 at S = 1: gather, fixed set, retained attention, value
    step, then (p.update_k) the key step against the merged values; without
    it K_out = K_Ret^0.  Inputs are the fp32 prefix scores c32 and the target
    y (as the library's grkv_merge receives them) and the retained idx."""
    idx = np.asarray(idx)
    K0 = np.asarray(k, dtype=f64)[idx]
    V0 = np.asarray(v, dtype=f64)[idx]
    fixed = fixed_set(idx, c32, p)
    X = retained_attention(q, k, idx, p)
    if math.isinf(p.lambda_v):
        V = V0.copy()
    else:
        step = value_step_dual if mode == "dual" else value_step_primal
        V = step(X, y, V0, ~fixed, f64(np.float32(p.lambda_v)))
    out = {"k_out": K0, "v_out": V, "fixed": fixed, "x": X}
    if p.update_k:
        Q = np.asarray(q, dtype=f64).reshape(p.m, p.d)
        K, hist = key_step_dual(X, Q, K0, V, y, ~fixed, f64(np.float32(p.lambda_k)),
                                effective_scale(p), p.cg_iters, p.cg_tol)
        out["k_out"] = K
        out["cg_residuals"] = hist
    return out


def compress_unit(q, k, v, p: Params, mode: str = "dual", idx=None):
    """The whole path for one unit: window attention stats, target Y, prefix
    scores, pooling, top-(B-w) selection plus window, then `merge_unit`.
    `idx` overrides the selection (test hook)."""
    A, M, L = window_attention(q, k, p)
    Y = target(A, v)
    c = column_scores(A, p)
    c32 = c.astype(np.float32)
    pooled = pool(c32, p)
    if idx is None:
        idx = select(pooled, p)
    out = merge_unit(q, k, v, c32, Y, idx, p, mode=mode)
    out.update({"attn": A, "row_max": M, "row_sum": L, "y": Y, "scores": c,
                "scores32": c32, "pooled": pooled, "idx": np.asarray(idx, dtype=np.int32)})
    return out


# --------------------------------------------------- decode-side transfer check
def cache_output(q, kc, vc, p: Params, window_rule: bool):
    """Y = A V of the stacked queries q [g][h][d] over a cache of c rows
    (kc, vc [c][d]): the attention output the paper's diagnostics compare
    (App. G, "Y = AV").  window_rule: the queries are the surrogate window
    (h = p.window) and row a sees slots j <= c - w + a, the window occupying
    the cache's last w slots (the retained-cache rule of Algorithm 1 under
    the causal reading); otherwise every query sees every slot (decoding
    queries come after the whole prompt)."""
    q = np.asarray(q, dtype=f64)
    g, h = q.shape[0], q.shape[1]
    kc = np.asarray(kc, dtype=f64)
    sub = dataclasses.replace(p, group=g, window=h, n=kc.shape[0], budget=kc.shape[0],
                              causal=bool(window_rule and p.causal))
    A, _, _ = softmax_rows(window_logits(q, kc, sub))
    return A @ np.asarray(vc, dtype=f64)


def transfer_check(q_win, q_held, k, v, idx, k_out, v_out, p: Params) -> dict:
    """Decode-side transfer check of one unit (App. G: the normalised
    discrepancy of the loss-performance diagnostic and the held-out-query
    stress test), comparing the compressed cache (k_out, v_out) with the
    eviction-only cache (K0, V0) = (K[idx], V[idx]) against the full cache:
        e_win(c)  = ||Y_win_full - Y_win(c)||_F^2    (surrogate window queries)
        e_held(c) = ||Y_held_full - Y_held(c)||_F^2  (held-out queries)
    A failure is a unit whose compressed cache lowers the window error but
    raises the held-out error relative to the eviction-only cache.  cos is
    the cosine between the mean window output and the mean held-out output
    over the full cache (the surrogate-actual similarity of Sec. 3.2)."""
    idx = np.asarray(idx)
    K0 = np.asarray(k, dtype=f64)[idx]
    V0 = np.asarray(v, dtype=f64)[idx]
    yw = cache_output(q_win, k, v, p, True)
    yh = cache_output(q_held, k, v, p, False)
    out = {"y_win2": float((yw ** 2).sum()), "y_held2": float((yh ** 2).sum())}
    for name, kc, vc in (("base", K0, V0), ("comp", k_out, v_out)):
        out["e_win_" + name] = float(((yw - cache_output(q_win, kc, vc, p, True)) ** 2).sum())
        out["e_held_" + name] = float(((yh - cache_output(q_held, kc, vc, p, False)) ** 2).sum())
    sw, sh = yw.mean(axis=0), yh.mean(axis=0)
    out["cos"] = float(sw @ sh / max(np.linalg.norm(sw) * np.linalg.norm(sh), 1e-300))
    out["fail"] = bool(out["e_win_comp"] < out["e_win_base"] and
                       out["e_held_comp"] > out["e_held_base"])
    return out


def l_common(reports, which: str = "comp", queries: str = "held") -> float:
    """L_common = sum over units of ||Y_full - Y_c||_F^2 / sum of ||Y_full||_F^2
    (App. G, normalised discrepancy), for cache `which` ("comp" or "base")
    and the held-out or window queries."""
    num = sum(r[f"e_{queries}_{which}"] for r in reports)
    den = sum(r["y_held2" if queries == "held" else "y_win2"] for r in reports)
    return num / den

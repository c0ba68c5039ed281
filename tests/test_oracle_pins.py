"""Pins of the fp64 oracle against what the paper and mathematics fix.

Each test checks one oracle function against something other than itself:
a library routine (scaled_dot_product_attention, max_pool1d, lstsq, sympy),
brute force on tiny inputs, a closed form, or an invariant of the ridge
problem (Eq. 6 / Eq. 7 and the dual form of App. D.1).
"""
import itertools
import math

import numpy as np
import pytest
import torch

import oracle as O

torch.set_default_dtype(torch.float64)


def _rand_unit(rng, g, w, n, d, peaked=True):
    k = rng.standard_normal((n, d))
    v = rng.standard_normal((n, d))
    if peaked:
        q = 1.5 * k[rng.integers(0, n, size=(g, w))] + 0.3 * rng.standard_normal((g, w, d))
    else:
        q = rng.standard_normal((g, w, d))
    return q, k, v


def _sdpa(q, k, vals, p, causal):
    """torch SDPA per query head over the shared KV head.  The causal window
    rule is the bottom-right aligned causal mask (query i of L sees keys
    j <= S - L + i), built with tril(diagonal=S-L)."""
    out = []
    for h in range(p.group):
        Q = torch.from_numpy(np.ascontiguousarray(q[h]))[None, None]
        K = torch.from_numpy(np.ascontiguousarray(k))[None, None]
        V = torch.from_numpy(np.ascontiguousarray(vals))[None, None]
        L, S = Q.shape[2], K.shape[2]
        mask = None
        if causal:
            mask = torch.ones(L, S, dtype=torch.bool).tril(diagonal=S - L)
        out.append(torch.nn.functional.scaled_dot_product_attention(
            Q, K, V, attn_mask=mask, scale=O.effective_scale(p))[0, 0].numpy())
    return np.concatenate(out, axis=0)


@pytest.mark.parametrize("causal", [True, False])
@pytest.mark.parametrize("g,w,n,d", [(1, 4, 11, 8), (3, 5, 23, 16), (2, 1, 9, 4)])
def test_window_attention_matches_sdpa(causal, g, w, n, d):
    rng = np.random.default_rng(1 + g * 100 + w * 10 + n)
    q, k, v = _rand_unit(rng, g, w, n, d)
    p = O.Params(group=g, n=n, d=d, window=w, budget=w, causal=causal)
    A, M, L = O.window_attention(q, k, p)
    # attention weights: SDPA with V = I_n returns A itself
    np.testing.assert_allclose(A, _sdpa(q, k, np.eye(n), p, causal), rtol=0, atol=1e-13)
    # target Y = A V (Algorithm 1)
    np.testing.assert_allclose(O.target(A, v), _sdpa(q, k, v, p, causal), rtol=0, atol=1e-12)
    # row stats: M + log L is the row log-sum-exp
    lg = torch.from_numpy(O.window_logits(q, k, p))
    np.testing.assert_allclose(M + np.log(L), torch.logsumexp(lg, dim=1).numpy(), rtol=1e-14)


def test_causal_rule_is_standard_causal_when_window_is_whole_sequence():
    rng = np.random.default_rng(7)
    n, d = 12, 8
    q, k, v = _rand_unit(rng, 1, n, n, d)
    p = O.Params(group=1, n=n, d=d, window=n, budget=n, causal=True)
    A, _, _ = O.window_attention(q, k, p)
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q)[None], torch.from_numpy(k)[None, None].expand(1, 1, n, d),
        torch.eye(n)[None, None], is_causal=True, scale=O.effective_scale(p))[0, 0].numpy()
    np.testing.assert_allclose(A, ref, atol=1e-13)


def test_default_scale_is_fp32_inverse_sqrt_d():
    p = O.Params(group=1, n=4, d=128, window=1, budget=1)
    assert O.effective_scale(p) == float(np.float32(1 / math.sqrt(128)))
    assert O.effective_scale(p.__class__(group=1, n=4, d=128, window=1, budget=1, scale=0.5)) == 0.5


def test_softmax_closed_form():
    # d = 1, scale 1, q = 1, k_j = ln(j + 1): weights (1, 2, 3, 4) / 10
    p = O.Params(group=1, n=4, d=1, window=1, budget=1, scale=1.0, causal=False)
    k = np.log(np.arange(1, 5, dtype=np.float64))[:, None]
    A, M, L = O.window_attention(np.ones((1, 1, 1)), k, p)
    np.testing.assert_allclose(A[0], [0.1, 0.2, 0.3, 0.4], rtol=1e-15)
    assert M[0] == pytest.approx(math.log(4)) and L[0] == pytest.approx(10 / 4)
    v = np.array([[1.0], [2.0], [3.0], [4.0]])
    assert O.target(A, v)[0, 0] == pytest.approx(3.0, rel=1e-15)   # (1+4+9+16)/10
    # scores cover the prefix n - w = 3 keys only
    np.testing.assert_allclose(O.column_scores(A, p), [0.1, 0.2, 0.3], rtol=1e-15)


@pytest.mark.parametrize("causal", [True, False])
def test_column_scores_are_sdpa_column_sums(causal):
    rng = np.random.default_rng(3)
    g, w, n, d = 2, 4, 30, 8
    q, k, v = _rand_unit(rng, g, w, n, d)
    p = O.Params(group=g, n=n, d=d, window=w, budget=w, causal=causal)
    A, _, _ = O.window_attention(q, k, p)
    ref = _sdpa(q, k, np.eye(n), p, causal).sum(axis=0)[: n - w]
    np.testing.assert_allclose(O.column_scores(A, p), ref, atol=1e-13)
    # each of the m rows is a probability vector
    np.testing.assert_allclose(A.sum(axis=1), np.ones(g * w), atol=1e-14)


@pytest.mark.parametrize("kernel", [1, 3, 7, 9])
@pytest.mark.parametrize("P", [1, 2, 5, 40])
def test_pool_matches_torch(kernel, P):
    rng = np.random.default_rng(kernel * 31 + P)
    c = rng.random(P).astype(np.float32)
    p = O.Params(group=1, n=P + 2, d=4, window=2, budget=2, pool_kernel=kernel)
    t = torch.from_numpy(c.astype(np.float64))[None, None]
    mx = torch.nn.functional.max_pool1d(t, kernel, stride=1, padding=kernel // 2)[0, 0].numpy()
    np.testing.assert_array_equal(O.pool(c, p), mx.astype(np.float32))
    av = torch.nn.functional.avg_pool1d(t, kernel, stride=1, padding=kernel // 2,
                                        count_include_pad=True)[0, 0].numpy()
    pa = O.Params(group=1, n=P + 2, d=4, window=2, budget=2, pool_kernel=kernel, pool_type="avg")
    np.testing.assert_allclose(O.pool(c, pa), av.astype(np.float32), rtol=2e-7)


def _brute_select(pooled, p):
    """Enumerate every (B-w)-subset of the prefix; keep the one with the
    largest exact score sum, ties to the lexicographically smallest indices."""
    P, kk = p.n - p.window, p.budget - p.window
    best = None
    for sub in itertools.combinations(range(P), kk):
        key = (sum(float(pooled[j]) for j in sub), tuple(-j for j in sub))
        if best is None or key > best[0]:
            best = (key, sub)
    return np.array(list(best[1]) + list(range(P, p.n)), dtype=np.int32)


@pytest.mark.parametrize("seed", range(6))
def test_select_brute_force(seed):
    rng = np.random.default_rng(seed)
    P, w = 12, 2
    kk = int(rng.integers(0, P + 1))
    p = O.Params(group=1, n=P + w, d=4, window=w, budget=kk + w)
    # integer-valued scores: exact sums, frequent ties
    pooled = rng.integers(0, 5, size=P).astype(np.float32)
    np.testing.assert_array_equal(O.select(pooled, p), _brute_select(pooled, p))
    pooled = (0.5 + 0.5 * rng.random(P)).astype(np.float32)   # distinct values
    np.testing.assert_array_equal(O.select(pooled, p), _brute_select(pooled, p))


def test_select_all_ties_and_full_budget():
    p = O.Params(group=1, n=20, d=4, window=3, budget=8)
    np.testing.assert_array_equal(O.select(np.ones(17, np.float32), p),
                                  np.r_[np.arange(5), np.arange(17, 20)])
    pf = O.Params(group=1, n=20, d=4, window=3, budget=20)
    np.testing.assert_array_equal(O.select(np.random.rand(17).astype(np.float32), pf), np.arange(20))
    pw = O.Params(group=1, n=20, d=4, window=3, budget=3)
    np.testing.assert_array_equal(O.select(np.random.rand(17).astype(np.float32), pw), [17, 18, 19])


def test_fixed_set_by_hand():
    # n = 20, w = 3, n_sink = 2, B = 10, beta = 0.25 -> floor(2.5) = 2 extra
    p = O.Params(group=1, n=20, d=4, window=3, budget=10, n_sink=2, beta=0.25)
    idx = np.array([0, 2, 5, 6, 9, 12, 16, 17, 18, 19])
    c = np.zeros(17, np.float32)
    c[[2, 5, 6, 9, 12, 16]] = [0.3, 0.9, 0.1, 0.9, 0.5, 0.05]
    c[0] = 5.0     # the sink is fixed anyway, its score does not use a slot
    fixed = O.fixed_set(idx, c, p)
    # sink 0 (token 2 is not a sink), window 17..19, and the two best of
    # {2, 5, 6, 9, 12, 16}: 5 and 9
    np.testing.assert_array_equal(np.nonzero(fixed)[0], [0, 2, 4, 7, 8, 9])
    c[9] = 0.9 - 1e-3
    c[12] = 0.9
    fixed = O.fixed_set(idx, c, p)     # 5 and 12 at 0.9 beat 9
    np.testing.assert_array_equal(idx[fixed], [0, 5, 12, 17, 18, 19])
    c[2] = c[5]                         # three-way tie: smaller indices 2, 5 win
    np.testing.assert_array_equal(idx[O.fixed_set(idx, c, p)], [0, 2, 5, 17, 18, 19])


def test_retained_attention_is_renormalised_full_attention():
    rng = np.random.default_rng(11)
    g, w, n, d = 2, 3, 25, 8
    q, k, v = _rand_unit(rng, g, w, n, d)
    p = O.Params(group=g, n=n, d=d, window=w, budget=9)
    A, _, _ = O.window_attention(q, k, p)
    idx = np.r_[np.sort(rng.choice(n - w, 6, replace=False)), np.arange(n - w, n)]
    X = O.retained_attention(q, k, idx, p)
    sub = A[:, idx]
    np.testing.assert_allclose(X, sub / sub.sum(axis=1, keepdims=True), atol=1e-14)


def _ridge_case(rng, m=4, c=9, d=5, nfix=2):
    logits = 2.0 * rng.standard_normal((m, c))
    X = np.exp(logits - logits.max(1, keepdims=True))
    X /= X.sum(1, keepdims=True)
    Y = rng.standard_normal((m, d))
    V0 = rng.standard_normal((c, d))
    free = np.ones(c, bool)
    free[rng.choice(c, nfix, replace=False)] = False
    return X, Y, V0, free


@pytest.mark.parametrize("lam", [1e-3, 1e-2, 1e-1, 1.0])
def test_dual_equals_primal(lam):
    X, Y, V0, free = _ridge_case(np.random.default_rng(int(lam * 1000) + 5), m=6, c=15)
    a = O.value_step_dual(X, Y, V0, free, lam)
    b = O.value_step_primal(X, Y, V0, free, lam)
    np.testing.assert_allclose(a, b, rtol=0, atol=1e-10 * np.abs(b).max())


def test_value_step_is_lstsq_of_augmented_system():
    rng = np.random.default_rng(21)
    X, Y, V0, free = _ridge_case(rng, m=5, c=12, d=3)
    lam = 0.03
    V = O.value_step_dual(X, Y, V0, free, lam)
    XG, XF = X[:, free], X[:, ~free]
    R = Y - XF @ V0[~free] - XG @ V0[free]
    A = np.vstack([XG, math.sqrt(lam) * np.eye(XG.shape[1])])
    b = np.vstack([R, np.zeros((XG.shape[1], Y.shape[1]))])
    dV = np.linalg.lstsq(A, b, rcond=None)[0]
    np.testing.assert_allclose(V[free], V0[free] + dV, atol=1e-11)
    np.testing.assert_array_equal(V[~free], V0[~free])


def test_value_step_minimises_the_objective_exactly():
    """Sympy: set the gradient of Eq. 6 (with F fixed, App. D.3) to zero in
    exact rational arithmetic; the oracle must land on that minimiser."""
    sympy = pytest.importorskip("sympy")
    R = sympy.Rational
    X = sympy.Matrix([[R(1, 2), R(1, 4), R(1, 4)], [R(1, 8), R(5, 8), R(1, 4)]])
    Y = sympy.Matrix([[R(1), R(-2)], [R(3, 2), R(1, 3)]])
    V0 = sympy.Matrix([[R(1), R(0)], [R(-1), R(2)], [R(1, 2), R(1, 2)]])
    lam = R(1, 10)
    free = [True, True, False]
    syms = sympy.symbols("v0:6")
    V = sympy.Matrix(3, 2, lambda i, j: syms[2 * i + j] if free[i] else V0[i, j])
    E = Y - X * V
    obj = sum(e ** 2 for e in E) + lam * sum((V[i, j] - V0[i, j]) ** 2 for i in range(3) for j in range(2))
    unknowns = [s for s in syms if any(V[i, j] == s for i in range(3) for j in range(2))]
    sol = sympy.solve([sympy.diff(obj, s) for s in unknowns], unknowns, dict=True)[0]
    Vs = np.array(V.subs(sol).tolist(), dtype=np.float64)
    Vo = O.value_step_dual(np.array(X.tolist(), float), np.array(Y.tolist(), float),
                           np.array(V0.tolist(), float), np.array(free), float(lam))
    np.testing.assert_allclose(Vo, Vs, atol=1e-13)


def test_single_row_closed_form():
    # m = 1: N = |x_G|^2 + lambda is a scalar, dV_j = x_j r / (|x_G|^2 + lambda)
    x = np.array([[0.5, 0.3, 0.2]])
    y = np.array([[2.0, -1.0]])
    V0 = np.array([[1.0, 0.0], [0.0, 1.0], [1.0, 1.0]])
    free = np.array([True, True, False])
    lam = 0.1
    r = y - x @ V0
    expect = V0.copy()
    expect[:2] += x[0, :2, None] * r / (0.25 + 0.09 + lam)
    np.testing.assert_allclose(O.value_step_dual(x, y, V0, free, lam), expect, atol=1e-15)


def test_large_lambda_leaves_values():
    X, Y, V0, free = _ridge_case(np.random.default_rng(4))
    lam = 1e8
    V = O.value_step_dual(X, Y, V0, free, lam)
    R = Y - X @ V0
    bound = np.linalg.norm(R) * np.linalg.norm(X[:, free], 2) / lam
    assert np.linalg.norm(V - V0) <= bound * (1 + 1e-9)


def test_stationarity_and_fixed_rows():
    X, Y, V0, free = _ridge_case(np.random.default_rng(5), m=8, c=20, d=6, nfix=5)
    lam = 0.02
    V = O.value_step_dual(X, Y, V0, free, lam)
    grad = X[:, free].T @ (X @ V - Y) + lam * (V[free] - V0[free])
    assert np.abs(grad).max() < 1e-12
    np.testing.assert_array_equal(V[~free], V0[~free])


def test_lambda_zero_interpolates_the_target():
    X, Y, V0, free = _ridge_case(np.random.default_rng(6), m=4, c=12, d=5, nfix=3)
    V = O.value_step_dual(X, Y, V0, free, 0.0)
    np.testing.assert_allclose(X @ V, Y, atol=1e-9)


def test_window_loss_monotone_in_lambda():
    X, Y, V0, free = _ridge_case(np.random.default_rng(8), m=6, c=14, d=4)
    losses = [np.linalg.norm(Y - X @ O.value_step_dual(X, Y, V0, free, lam))
              for lam in (10.0, 1.0, 0.1, 0.01, 0.0)]
    assert all(a >= b - 1e-12 for a, b in zip(losses, losses[1:]))
    assert losses[0] <= np.linalg.norm(Y - X @ V0) + 1e-12


def test_full_budget_gives_zero_update():
    rng = np.random.default_rng(9)
    g, w, n, d = 2, 4, 40, 8
    q, k, v = _rand_unit(rng, g, w, n, d)
    p = O.Params(group=g, n=n, d=d, window=w, budget=n, n_sink=2, beta=0.1)
    out = O.compress_unit(q, k, v, p)
    np.testing.assert_array_equal(out["idx"], np.arange(n))
    np.testing.assert_allclose(out["v_out"], v, atol=1e-12)


def test_compress_unit_structure():
    rng = np.random.default_rng(10)
    g, w, n, d, B = 2, 4, 64, 8, 20
    q, k, v = _rand_unit(rng, g, w, n, d)
    p = O.Params(group=g, n=n, d=d, window=w, budget=B)
    out = O.compress_unit(q, k, v, p)
    idx = out["idx"]
    assert idx.size == B and np.all(np.diff(idx) > 0)
    np.testing.assert_array_equal(idx[-w:], np.arange(n - w, n))
    np.testing.assert_array_equal(out["k_out"], k[idx])
    np.testing.assert_array_equal(out["v_out"][out["fixed"]], v[idx][out["fixed"]])
    primal = O.compress_unit(q, k, v, p, mode="primal")
    np.testing.assert_allclose(out["v_out"], primal["v_out"], atol=1e-10)
    # lambda = inf: values unchanged
    pinf = O.Params(group=g, n=n, d=d, window=w, budget=B, lambda_v=math.inf)
    np.testing.assert_array_equal(O.compress_unit(q, k, v, pinf)["v_out"], v[idx])


# ------------------------------------------------------------- key step (NEXT)
def _key_case(rng, g=2, w=2, n=9, d=3, causal=True):
    """A tiny unit with its retained attention X at K0 and merged values V."""
    q, k, v = _rand_unit(rng, g, w, n, d, peaked=False)
    p = O.Params(group=g, n=n, d=d, window=w, budget=n - 2, causal=causal, update_k=True)
    idx = np.sort(rng.choice(n - w, size=n - 2 - w, replace=False))
    idx = np.concatenate([idx, np.arange(n - w, n)])
    K0 = k[idx]
    V = rng.standard_normal((idx.size, d))
    X = O.retained_attention(q, k, idx, p)
    Y = rng.standard_normal((p.m, d))
    return p, q.reshape(p.m, d), K0, V, X, Y, idx


def _autograd_jacobian(p, Q, K0, V, idx):
    """d vec(f)/d vec(K) of f(K) = softmax(s Q K^T + causal mask) V, by torch
    autograd in fp64 (row-major vec); independent of the oracle's JVP/VJP."""
    s = O.effective_scale(p)
    a = np.arange(p.m) % p.window
    mask = np.asarray(idx)[None, :] <= (p.n - p.window + a)[:, None] if p.causal else np.ones((p.m, len(idx)), bool)
    Qt, Vt = torch.from_numpy(Q), torch.from_numpy(V)
    bias = torch.from_numpy(np.where(mask, 0.0, -np.inf))

    def f(Kflat):
        K = Kflat.reshape(K0.shape)
        return (torch.softmax(s * Qt @ K.T + bias, dim=1) @ Vt).reshape(-1)

    return torch.autograd.functional.jacobian(f, torch.from_numpy(K0.reshape(-1))).numpy()


@pytest.mark.parametrize("causal", [True, False])
def test_key_jvp_vjp_match_autograd(causal):
    rng = np.random.default_rng(71 + causal)
    p, Q, K0, V, X, Y, idx = _key_case(rng, causal=causal)
    J = _autograd_jacobian(p, Q, K0, V, idx)
    s = O.effective_scale(p)
    dK = rng.standard_normal(K0.shape)
    W = rng.standard_normal((p.m, p.d))
    np.testing.assert_allclose(O.key_jvp(X, Q, V, dK, s).reshape(-1), J @ dK.reshape(-1),
                               rtol=0, atol=1e-13)
    np.testing.assert_allclose(O.key_vjp(X, Q, V, W, s).reshape(-1), J.T @ W.reshape(-1),
                               rtol=0, atol=1e-13)


@pytest.mark.parametrize("lam", [1e-2, 1e-1, 3.0])
def test_key_step_matches_dense_ridge(lam):
    """Full CG (md iterations) reaches the linearised ridge solution of App.
    D.2, computed densely in both forms from the autograd Jacobian:
    primal (J_G^T J_G + lam I) z = J_G^T e and dual J_G^T (J_G J_G^T + lam I)^-1 e."""
    rng = np.random.default_rng(int(lam * 1000) + 5)
    p, Q, K0, V, X, Y, idx = _key_case(rng)
    free = np.ones(idx.size, bool)
    free[[0, idx.size - 1]] = False
    J = _autograd_jacobian(p, Q, K0, V, idx)
    cols = np.repeat(free, p.d)                       # row-major vec(K): row i -> d entries
    JG = J[:, cols]
    e = (Y - X @ V).reshape(-1)
    z_primal = np.linalg.solve(JG.T @ JG + lam * np.eye(JG.shape[1]), JG.T @ e)
    z_dual = JG.T @ np.linalg.solve(JG @ JG.T + lam * np.eye(JG.shape[0]), e)
    np.testing.assert_allclose(z_dual, z_primal, rtol=0, atol=1e-10)
    # CG reaches the solution in md steps in exact arithmetic; in fp64 at small
    # lambda the lost orthogonality needs a few times more
    K, hist = O.key_step_dual(X, Q, K0, V, Y, free, lam, O.effective_scale(p), iters=20 * p.m * p.d)
    want = K0.copy()
    want[free] = K0[free] + z_primal.reshape(-1, p.d)
    np.testing.assert_allclose(K, want, rtol=0, atol=1e-9)
    assert hist[-1] <= 1e-9 * hist[0]
    assert np.array_equal(K[~free], K0[~free])


def test_key_step_large_lambda_leaves_keys():
    rng = np.random.default_rng(9)
    p, Q, K0, V, X, Y, idx = _key_case(rng)
    free = np.ones(idx.size, bool)
    s = O.effective_scale(p)
    lam = 1e8
    K, _ = O.key_step_dual(X, Q, K0, V, Y, free, lam, s, iters=p.m * p.d)
    bound = np.linalg.norm(O.key_vjp(X, Q, V, Y - X @ V, s)) / lam
    assert np.linalg.norm(K - K0) <= 1.0001 * bound


def test_key_step_stationarity():
    """z = K* - K0 solves J_G^T (J_G z - e) + lam z = 0 (normal equation of
    the local ridge problem), with J applied through autograd."""
    rng = np.random.default_rng(13)
    p, Q, K0, V, X, Y, idx = _key_case(rng, g=1, w=3, n=10, d=4)
    free = np.ones(idx.size, bool)
    free[1] = False
    lam = 0.05
    K, _ = O.key_step_dual(X, Q, K0, V, Y, free, lam, O.effective_scale(p), iters=20 * p.m * p.d)
    J = _autograd_jacobian(p, Q, K0, V, idx)[:, np.repeat(free, p.d)]
    z = (K - K0)[free].reshape(-1)
    e = (Y - X @ V).reshape(-1)
    g = J.T @ (J @ z - e) + lam * z
    assert np.abs(g).max() <= 1e-10 * max(1.0, np.abs(J.T @ e).max())


def test_merge_unit_key_step_uses_merged_values():
    """With update_k the key step linearises f around K0 with the merged
    values V* of the value step, and keeps fixed rows (Algorithm 1)."""
    rng = np.random.default_rng(21)
    g, w, n, d = 2, 3, 24, 8
    q, k, v = _rand_unit(rng, g, w, n, d)
    p = O.Params(group=g, n=n, d=d, window=w, budget=12, n_sink=2, beta=0.2, update_k=True,
                 lambda_k=0.05, cg_iters=g * w * d, cg_tol=1e-8)
    base = O.compress_unit(q, k, v, dataclasses_replace(p, update_k=False))
    out = O.compress_unit(q, k, v, p)
    np.testing.assert_array_equal(out["idx"], base["idx"])
    np.testing.assert_array_equal(out["v_out"], base["v_out"])
    K0 = np.asarray(k, dtype=np.float64)[out["idx"]]
    Q = np.asarray(q, dtype=np.float64).reshape(p.m, d)
    want, _ = O.key_step_dual(out["x"], Q, K0, out["v_out"], out["y"], ~out["fixed"],
                              np.float64(np.float32(p.lambda_k)), O.effective_scale(p), p.cg_iters,
                              p.cg_tol)
    np.testing.assert_array_equal(out["k_out"], want)
    assert np.array_equal(out["k_out"][out["fixed"]], K0[out["fixed"]])
    assert np.abs(out["k_out"] - K0).max() > 0


def dataclasses_replace(p, **kw):
    import dataclasses
    return dataclasses.replace(p, **kw)


def test_key_step_stops_at_the_residual_tolerance():
    rng = np.random.default_rng(31)
    p, Q, K0, V, X, Y, idx = _key_case(rng, g=2, w=3, n=14, d=4)
    free = np.ones(idx.size, bool)
    s = O.effective_scale(p)
    _, full = O.key_step_dual(X, Q, K0, V, Y, free, 0.1, s, iters=400)
    K, hist = O.key_step_dual(X, Q, K0, V, Y, free, 0.1, s, iters=400, tol=1e-3)
    assert hist[-1] <= 1e-3 * hist[0] and all(h > 1e-3 * hist[0] for h in hist[:-1])
    assert len(hist) < len(full)


# ------------------------------------------------- multi-step alternation --
def test_alternation_one_step_is_the_single_step_merge():
    rng = np.random.default_rng(41)
    g, w, n, d = 2, 3, 30, 8
    q, k, v = _rand_unit(rng, g, w, n, d)
    p = O.Params(group=g, n=n, d=d, window=w, budget=14, n_sink=2, beta=0.2, update_k=True,
                 lambda_k=0.05, cg_iters=500, cg_tol=1e-12)
    one = O.compress_unit(q, k, v, p)
    alt = O.alternate(q, k, v, one["scores32"], one["y"], one["idx"], p, steps=1)
    np.testing.assert_allclose(alt["v_out"], one["v_out"], rtol=0, atol=1e-13)
    np.testing.assert_allclose(alt["k_out"], one["k_out"], rtol=0, atol=1e-11)


def test_alternation_converges_to_a_stationary_point():
    """At a fixed point of the alternation, the key step's linearised update
    reproduces K (G = K - K0), which by the ridge identity means
    lambda_k (K - K0)_G = J_G^T (Y - f(K)): K is a stationary point of the
    nonlinear key objective ||Y - f(K)||^2 + lambda_k ||K - K0||^2 with V
    fixed; V is the exact value step at the final X.  Gradients by autograd."""
    rng = np.random.default_rng(43)
    g, w, n, d = 1, 3, 16, 4
    q, k, v = _rand_unit(rng, g, w, n, d, peaked=False)
    p = O.Params(group=g, n=n, d=d, window=w, budget=9, n_sink=1, beta=0.2, update_k=True,
                 lambda_v=0.5, lambda_k=0.5, cg_iters=500, cg_tol=1e-13)
    base = O.compress_unit(q, k, v, dataclasses_replace(p, update_k=False))
    out = O.alternate(q, k, v, base["scores32"], base["y"], base["idx"], p, steps=200, stop=1e-11)
    assert max(out["deltas"][-1]) <= 1e-11, out["deltas"][-3:]
    idx, K, V, Y = base["idx"], out["k_out"], out["v_out"], base["y"]
    free = ~out["fixed"]
    s = O.effective_scale(p)
    a = np.arange(p.m) % p.window
    mask = idx[None, :] <= (p.n - p.window + a)[:, None]
    Qt = torch.from_numpy(np.asarray(q, dtype=np.float64).reshape(p.m, d))
    Kt = torch.from_numpy(K.copy()).requires_grad_(True)
    f = torch.softmax(s * Qt @ Kt.T + torch.from_numpy(np.where(mask, 0.0, -np.inf)), dim=1) \
        @ torch.from_numpy(V)
    loss = ((torch.from_numpy(Y) - f) ** 2).sum() + p.lambda_k * ((Kt - torch.from_numpy(
        np.asarray(k, dtype=np.float64)[idx])) ** 2).sum()
    loss.backward()
    grad = Kt.grad.numpy()
    assert np.abs(grad[free]).max() <= 1e-8
    X, _, _ = O.softmax_rows(O.window_logits(q, K, p, cols=idx))
    V_want = O.value_step_dual(X, Y, np.asarray(v, dtype=np.float64)[idx], free, 0.5)
    np.testing.assert_allclose(V, V_want, rtol=0, atol=1e-12)


# ----------------------------------------------- decode-side transfer check --
@pytest.mark.parametrize("window_rule", [True, False])
def test_cache_output_matches_sdpa(window_rule):
    """Y = A V over a cache of c slots: SDPA with the bottom-right causal mask
    on slots (window rule) or with no mask (decoding queries)."""
    rng = np.random.default_rng(31 + window_rule)
    g, h, c, d = 2, 5, 17, 8
    q, kc, vc = rng.standard_normal((g, h, d)), rng.standard_normal((c, d)), rng.standard_normal((c, d))
    p = O.Params(group=g, n=40, d=d, window=h, budget=c)
    sub = O.Params(group=g, n=c, d=d, window=h, budget=c)
    np.testing.assert_allclose(O.cache_output(q, kc, vc, p, window_rule),
                               _sdpa(q, kc, vc, sub, window_rule), rtol=0, atol=1e-12)


def test_cache_output_single_slot_returns_its_value():
    rng = np.random.default_rng(5)
    q, kc, vc = rng.standard_normal((3, 4, 8)), rng.standard_normal((1, 8)), rng.standard_normal((1, 8))
    p = O.Params(group=3, n=10, d=8, window=4, budget=1, causal=False)
    np.testing.assert_allclose(O.cache_output(q, kc, vc, p, False), np.repeat(vc, 12, 0), atol=1e-15)


def _transfer_case(seed=3, g=2, w=4, h=6, n=60, d=8, B=16, lam=1e-2):
    rng = np.random.default_rng(seed)
    q, k, v = _rand_unit(rng, g, w, n, d)
    qh = 1.5 * k[rng.integers(0, n, size=(g, h))] + 0.3 * rng.standard_normal((g, h, d))
    p = O.Params(group=g, n=n, d=d, window=w, budget=B, lambda_v=lam)
    return q, qh, k, v, p


def test_transfer_check_full_cache_has_no_error():
    """B = n and lambda = inf keep the whole cache unchanged: every error is 0."""
    q, qh, k, v, p = _transfer_case(B=60)
    p = O.Params(**{**p.__dict__, "lambda_v": math.inf})
    o = O.compress_unit(q, k, v, p)
    r = O.transfer_check(q, qh, k, v, o["idx"], o["k_out"], o["v_out"], p)
    for key in ("e_win_base", "e_win_comp", "e_held_base", "e_held_comp"):
        assert r[key] <= 1e-24 * r["y_win2"], key
    assert not r["fail"]


def test_transfer_window_error_is_the_value_step_data_term():
    """e_win of the compressed cache is ||Y - X V*||^2 of the value step
    (Algorithm 1, slot rule on the retained cache = position rule on idx),
    and the ridge lowers it below the eviction-only cache's."""
    q, qh, k, v, p = _transfer_case()
    o = O.compress_unit(q, k, v, p)
    X = O.retained_attention(q, k, o["idx"], p)
    r = O.transfer_check(q, qh, k, v, o["idx"], o["k_out"], o["v_out"], p)
    np.testing.assert_allclose(r["e_win_comp"], ((o["y"] - X @ o["v_out"]) ** 2).sum(), rtol=1e-10)
    V0 = v[o["idx"]]
    np.testing.assert_allclose(r["e_win_base"], ((o["y"] - X @ V0) ** 2).sum(), rtol=1e-10)
    assert r["e_win_comp"] < r["e_win_base"]


def test_transfer_window_error_vanishes_as_lambda_goes_to_zero():
    """lambda -> 0 with X_G of full row rank interpolates the target (the
    lambda -> 0 limit of Eq. 7): the compressed cache's window error -> 0."""
    q, qh, k, v, p = _transfer_case(B=40, lam=1e-9)
    o = O.compress_unit(q, k, v, p)
    r = O.transfer_check(q, qh, k, v, o["idx"], o["k_out"], o["v_out"], p)
    assert r["e_win_comp"] <= 1e-10 * r["y_win2"]


def test_transfer_similarity_and_l_common():
    """cos is 1 when the held-out queries are the window queries seen without
    the window rule, and is invariant to scaling V; L_common is the ratio of
    summed squared errors to summed squared targets (App. G)."""
    q, _, k, v, p = _transfer_case()
    pn = O.Params(**{**p.__dict__, "causal": False})
    o = O.compress_unit(q, k, v, pn)
    r = O.transfer_check(q, q, k, v, o["idx"], o["k_out"], o["v_out"], pn)
    assert abs(r["cos"] - 1.0) < 1e-12
    q2, qh, k2, v2, p2 = _transfer_case(seed=9)
    o2 = O.compress_unit(q2, k2, v2, p2)
    r2 = O.transfer_check(q2, qh, k2, v2, o2["idx"], o2["k_out"], o2["v_out"], p2)
    o3 = O.compress_unit(q2, k2, 3.0 * v2, p2)
    r3 = O.transfer_check(q2, qh, k2, 3.0 * v2, o3["idx"], o3["k_out"], o3["v_out"], p2)
    assert abs(r2["cos"] - r3["cos"]) < 1e-12
    reps = [r, r2]
    want = (r["e_held_comp"] + r2["e_held_comp"]) / (r["y_held2"] + r2["y_held2"])
    assert abs(O.l_common(reps) - want) <= 1e-15 * want
    assert abs(O.l_common(reps, "base", "win") -
               (r["e_win_base"] + r2["e_win_base"]) / (r["y_win2"] + r2["y_win2"])) < 1e-14

"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Each test names the passage it follows.  None of them re-types the oracle's
own formula: they compare with the paper's worked example (tests/golden),
closed forms written a different way (normal equations, QR projectors,
finite differences), invariants and brute force.
"""
import json
import os

import numpy as np
import pytest

import oracle as O
from workloads import all_patterns, get, make_R

HERE = os.path.dirname(os.path.abspath(__file__))


def _golden():
    with open(os.path.join(HERE, "golden", "worked_example.json")) as f:
        return json.load(f)


def _tiny_inputs(ell, seed=11):
    rng = np.random.default_rng(seed)
    N = m = 6
    delta = 3
    order = O.cyclic_order(N, m, delta)
    R = rng.standard_normal((ell, m))
    d, n_c = 64, 32
    X = rng.standard_normal((N * n_c, d))
    y = rng.standard_normal(N * n_c)
    w = rng.standard_normal(d) / 8
    return N, m, delta, order, R, X, y, w, d, n_c


def _projector(R, S):
    """Orthogonal projector onto the column space of R[:, S] from a QR
    factorisation (independent of the oracle's pseudo-inverse route)."""
    ell = R.shape[0]
    if len(S) == 0:
        return np.zeros((ell, ell))
    if len(S) >= ell:
        return np.eye(ell)  # full row rank a.s. (Sec. II-A)
    Q, _ = np.linalg.qr(R[:, S])
    return Q @ Q.T


# ---------------------------------------------------------------- Sec. II-B
def test_worked_example_supports_and_classification():
    """Sec. II-B: psi=[5 2 0 2 3] gives the support of eq. (3) and is exact
    for l=2; psi=[4 2 0 2 3] gives eq. (8) with a single copy of D5."""
    g = _golden()
    order = np.array(g["order"], dtype=np.int32)
    N, ell = g["N"], g["ell"]
    for case in g["cases"]:
        psi = np.array(case["psi"])
        sup = O.support(order, psi, N)            # N x m
        assert np.array_equal(sup.T, np.array(case["B_support_worker_by_chunk"]))
        assert list(O.copies(order, psi, N)) == case["Delta"]
        assert O.is_exact(order, psi, N, ell) == case["exact"]
        assert O.error_estimate(order, psi, N, ell) == case["estimate"]
        # the solved B has exactly that support (Gaussian R: no accidental zeros)
        R = np.random.default_rng(5).standard_normal((ell, g["m"]))
        B = O.encoding_matrix(R, order, psi, N)
        nz = np.zeros((g["m"], N), dtype=int)
        for i in range(N):
            nz[:, i] = np.any(B[:, i * ell:(i + 1) * ell] != 0, axis=1)
        assert np.array_equal(nz, np.array(case["B_support_worker_by_chunk"]))


def test_worked_example_w5_underdetermined_closed_form():
    """Sec. II-B: the first column of B^(1) is the minimum-norm solution of
    [[r01 r02 r05],[r11 r12 r15]] [a1 b1 d1]^T = [1 0]^T.  For a full-row-rank
    X that is X^T (X X^T)^{-1} e_0 (normal equations of the row space)."""
    g = _golden()
    order = np.array(g["order"], dtype=np.int32)
    N, ell, m = g["N"], g["ell"], g["m"]
    pr = g["w5_first_column_problem"]
    R = np.random.default_rng(7).standard_normal((ell, m))
    psi = np.array(g["cases"][0]["psi"])
    X = R[:, pr["workers"]]
    e0 = np.array([1.0, 0.0])
    expect = X.T @ np.linalg.solve(X @ X.T, e0)
    B = O.encoding_matrix(R, order, psi, N)
    col = pr["chunk"] * ell + pr["column"]
    got = B[pr["workers"], col]
    assert np.allclose(got, expect, rtol=0, atol=1e-12)
    # W5 solves the same problem independently and agrees (Sec. II-B)
    _, solved5 = O.find_encoding_coeff(R, order, psi, N, 4, return_solved=True)
    assert np.allclose(solved5[pr["workers"], col], expect, rtol=0, atol=1e-12)


def test_worked_example_w5_overdetermined_closed_form():
    """Sec. II-B: with psi=[4 2 0 2 3], d'9 solves || [r05 r15]^T d'9 - [1 0]^T ||;
    for a single column x the least-squares solution is x_0 / ||x||^2 and the
    squared residual 1 - x_0^2/||x||^2; column e_1 gives x_1/||x||^2."""
    g = _golden()
    order = np.array(g["order"], dtype=np.int32)
    N, ell, m = g["N"], g["ell"], g["m"]
    pr = g["w5_overdetermined_problem"]
    R = np.random.default_rng(8).standard_normal((ell, m))
    psi = np.array(g["cases"][1]["psi"])
    x = R[:, pr["workers"][0]]
    nn = float(x @ x)
    B = O.encoding_matrix(R, order, psi, N)
    i = pr["chunk"]
    assert abs(B[4, i * ell + 0] - x[0] / nn) < 1e-12
    assert abs(B[4, i * ell + 1] - x[1] / nn) < 1e-12
    C = O.decode_matrix(R, B)
    resid0 = 1.0 - C[0, i * ell + 0]
    assert abs(resid0 - (1.0 - x[0] ** 2 / nn)) < 1e-12
    # that chunk alone carries the whole error: l - Delta = 1 (eq. 7)
    assert abs(O.coefficient_error(R, B, N) - 1.0) < 1e-10


# ---------------------------------------------------------------- Alg. 1
@pytest.mark.parametrize("ell", [1, 2, 3])
def test_projector_blocks_match_qr(ell):
    """R B block i is the orthogonal projector onto range(R[:, S_i]) (the
    min-norm LS solution gives X X^+): I when Delta_i >= l (Sec. II-A), a
    rank-Delta_i projector otherwise, 0 when no copy was processed."""
    N, m, delta, order, R, *_ = _tiny_inputs(ell)
    rng = np.random.default_rng(100 + ell)
    for _ in range(40):
        psi = rng.integers(0, delta + 1, size=m)
        B = O.encoding_matrix(R, order, psi, N)
        C = O.decode_matrix(R, B)
        S = O.completed_sets(order, psi, N)
        for i in range(N):
            P = _projector(R, S[i])
            assert np.allclose(C[:, i * ell:(i + 1) * ell], P, rtol=0, atol=1e-11)


@pytest.mark.parametrize("ell", [2, 3])
def test_holders_agree(ell):
    """Sec. II: every holder of D_i solves the same min-norm problem and gets
    the same block column, so the assembled B is consistent."""
    N, m, delta, order, R, *_ = _tiny_inputs(ell)
    rng = np.random.default_rng(200 + ell)
    for _ in range(10):
        psi = rng.integers(0, delta + 1, size=m)
        S = O.completed_sets(order, psi, N)
        solved = {j: O.find_encoding_coeff(R, order, psi, N, j, return_solved=True)[1]
                  for j in range(m) if psi[j] > 0}
        for i in range(N):
            blocks = [solved[j][:, i * ell:(i + 1) * ell] for j in S[i]]
            for b in blocks[1:]:
                assert np.allclose(b, blocks[0], rtol=0, atol=1e-12)


def test_rank_identity_error_equals_estimate():
    """Sec. II-A, eq. (7): the estimate is sum_i max(0, l - Delta_i).  For a
    projector P of rank r on R^l, ||I - P||_F^2 = l - r, and rank(R[:, S_i]) =
    min(l, Delta_i) for Gaussian R, so the coefficient error equals the
    estimate for every pattern, not only in expectation."""
    for ell in (1, 2, 3):
        N, m, delta, order, R, *_ = _tiny_inputs(ell, seed=ell)
        rng = np.random.default_rng(300 + ell)
        for _ in range(60):
            psi = rng.integers(0, delta + 1, size=m)
            B = O.encoding_matrix(R, order, psi, N)
            assert abs(O.coefficient_error(R, B, N) - O.error_estimate(order, psi, N, ell)) < 1e-10


def test_expected_single_chunk_error():
    """Eq. (7): E||X X^+ e_i - e_i||^2 = (l - Delta)/l over Gaussian X; Monte
    Carlo over R for one chunk with Delta = 1 copy and l = 3."""
    ell = 3
    order = np.array([[0]], dtype=np.int32)
    psi = np.array([1])
    rng = np.random.default_rng(9)
    errs = []
    for _ in range(4000):
        R = rng.standard_normal((ell, 1))
        B = O.encoding_matrix(R, order, psi, 1)
        C = O.decode_matrix(R, B)
        errs.append((C[0, 0] - 1.0) ** 2 + C[1, 0] ** 2 + C[2, 0] ** 2)
    assert abs(np.mean(errs) - (ell - 1) / ell) < 0.03


# ---------------------------------------------------------------- encode/decode
@pytest.mark.parametrize("ell", [1, 2, 3])
def test_exact_recovery_whenever_condition_holds(ell):
    """Sec. II-A: if every D_i was processed >= l times the PS recovers
    sum_i g_{D_i}; the transmit path (eq. 2 then Sec. II-B decode) and the
    fused R B form agree."""
    N, m, delta, order, R, X, y, w, d, n_c = _tiny_inputs(ell)
    G = O.chunk_gradients(X, y, w, N, n_c, O.LSQ)
    gsum = G.sum(axis=0)
    rng = np.random.default_rng(400 + ell)
    hits = 0
    for t in range(80):
        lo = 0 if t % 2 else max(0, delta - 1)   # half the draws near completion
        psi = rng.integers(lo, delta + 1, size=m)
        B = O.encoding_matrix(R, order, psi, N)
        T = O.encode(B, G, order, psi, ell)
        gh = O.decode(R, T, d)
        gf = O.decode_fused(R, B, G)
        assert np.allclose(gh, gf, rtol=0, atol=1e-12 * np.abs(gsum).max())
        if O.is_exact(order, psi, N, ell):
            hits += 1
            assert np.allclose(gh, gsum, rtol=0, atol=1e-10 * np.abs(gsum).max())
    assert hits > 0


def test_all_workers_finish_is_baseline_gradient():
    """Sec. I: with psi = delta everywhere the decoded vector is the baseline
    scheme's sum of chunk gradients, i.e. the one-shot full-batch gradient
    X^T (X w - y) for least squares and X^T (sigmoid(X w) - y01) for logistic."""
    for loss in (O.LSQ, O.LOGISTIC):
        N, m, delta, order, R, X, y, w, d, n_c = _tiny_inputs(3)
        if loss == O.LOGISTIC:
            y = np.where(y > 0, 1.0, -1.0)
            full = X.T @ (1.0 / (1.0 + np.exp(-(X @ w))) - (y + 1) / 2)
        else:
            full = X.T @ (X @ w - y)
        G = O.chunk_gradients(X, y, w, N, n_c, loss)
        psi = np.full(m, delta)
        for ell in (1, 2, 3):
            Rl = np.random.default_rng(ell).standard_normal((ell, m))
            B = O.encoding_matrix(Rl, order, psi, N)
            gh = O.decode(Rl, O.encode(B, G, order, psi, ell), d)
            assert np.allclose(gh, full, rtol=0, atol=1e-10 * np.abs(full).max())


def test_ell1_weighted_partial_sums():
    """Remark 1 (l = 1): the decoded vector is the sum of the chunk gradients
    with at least one processed copy; projector blocks are 1 or 0."""
    N, m, delta, order, R, X, y, w, d, n_c = _tiny_inputs(1)
    G = O.chunk_gradients(X, y, w, N, n_c, O.LSQ)
    rng = np.random.default_rng(13)
    for _ in range(50):
        psi = rng.integers(0, delta + 1, size=m)
        Delta = O.copies(order, psi, N)
        B = O.encoding_matrix(R, order, psi, N)
        gh = O.decode(R, O.encode(B, G, order, psi, 1), d)
        expect = G[Delta >= 1].sum(axis=0) if np.any(Delta >= 1) else np.zeros(d)
        assert np.allclose(gh, expect, rtol=0, atol=1e-10 * (np.abs(G).max() + 1))
        # MSE closed form for l = 1: the missing chunks' sum
        miss = G[Delta == 0].sum(axis=0) if np.any(Delta == 0) else np.zeros(d)
        assert abs(O.gradient_mse(gh, G.sum(axis=0)) - float(miss @ miss) / d) < 1e-9 * (1 + float(miss @ miss))


def test_order_invariance_of_full_gradient():
    """With every worker done, permuting chunks inside workers changes
    nothing: the decoded vector is the full gradient either way."""
    N, m, delta, order, R, X, y, w, d, n_c = _tiny_inputs(2)
    G = O.chunk_gradients(X, y, w, N, n_c, O.LSQ)
    rng = np.random.default_rng(17)
    psi = np.full(m, delta)
    ref = O.decode(R, O.encode(O.encoding_matrix(R, order, psi, N), G, order, psi, 2), d)
    for _ in range(5):
        perm = np.array([rng.permutation(row) for row in order], dtype=np.int32)
        gh = O.decode(R, O.encode(O.encoding_matrix(R, perm, psi, N), G, perm, psi, 2), d)
        assert np.allclose(gh, ref, rtol=0, atol=1e-10 * np.abs(ref).max())


def test_monotone_in_psi():
    """More processed chunks never increase the coefficient error."""
    N, m, delta, order, R, *_ = _tiny_inputs(3)
    rng = np.random.default_rng(19)
    for _ in range(30):
        psi = rng.integers(0, delta, size=m)
        j = rng.integers(0, m)
        psi2 = psi.copy()
        psi2[j] += 1
        e1 = O.coefficient_error(R, O.encoding_matrix(R, order, psi, N), N)
        e2 = O.coefficient_error(R, O.encoding_matrix(R, order, psi2, N), N)
        assert e2 <= e1 + 1e-10


def test_brute_force_tiny_all_patterns():
    """Every psi in {0..3}^6 on the tiny cyclic workload, l = 1, 2, 3:
    exact flag <=> min Delta >= l; error = estimate; decoded vector =
    sum_i P_i g_i with QR projectors P_i (and = sum g_i when exact)."""
    cfg = get("tiny")
    pats = all_patterns(cfg.m, cfg.delta)
    assert pats.shape == (4096, 6)
    N, m, delta = cfg.N, cfg.m, cfg.delta
    order = O.cyclic_order(N, m, delta)
    rng = np.random.default_rng(23)
    d = 16
    G = rng.standard_normal((N, d))
    for ell in (1, 2, 3):
        R = make_R(cfg, ell)
        L = O.block_length(d, ell)
        Gb = np.stack([O.blocks(G[i], ell) for i in range(N)])  # N x ell x L
        for psi in pats[:: (1 if ell == 2 else 4)]:
            r = O.run_pattern(R, order, psi, N, G, want_transmit=True)
            exact = r.Delta.min() >= ell
            assert O.is_exact(order, psi, N, ell) == exact
            assert abs(r.coef_err - r.est) < 1e-9
            expect = np.zeros((ell, L))
            for i in range(N):
                expect += _projector(R, r.S[i]) @ Gb[i]
            expect = expect.reshape(-1)[:d]
            assert np.allclose(r.ghat, expect, rtol=0, atol=1e-9)
            if exact:
                assert np.allclose(r.ghat, G.sum(axis=0), rtol=0, atol=1e-9)


# ---------------------------------------------------------------- gradients
@pytest.mark.parametrize("loss", [O.LSQ, O.LOGISTIC])
def test_chunk_gradients_finite_difference(loss):
    """Sec. I: grad L = (1/N~) sum_j g_{D_j}.  Central differences of the
    loss L = (1/N~) sum l (h = 1e-6) agree to 1e-6 relative."""
    N, m, delta, order, R, X, y, w, d, n_c = _tiny_inputs(2)
    if loss == O.LOGISTIC:
        y = np.where(y > 0, 1.0, -1.0)
    Ntil = N * n_c
    G = O.chunk_gradients(X, y, w, N, n_c, loss)
    grad = G.sum(axis=0) / Ntil
    h = 1e-6
    fd = np.zeros(d)
    for k in range(d):
        e = np.zeros(d)
        e[k] = h
        fd[k] = (O.full_loss(X, y, w + e, Ntil, 64, loss) - O.full_loss(X, y, w - e, Ntil, 64, loss)) / (2 * h)
    assert np.max(np.abs(fd - grad)) <= 1e-6 * np.max(np.abs(grad))


def test_sgd_step_is_gradient_descent_on_L():
    """One step w - lr * (sum g)/N~ equals w - lr * grad L with grad L from
    finite differences (pins the 1/N~ normalisation of Sec. I)."""
    N, m, delta, order, R, X, y, w, d, n_c = _tiny_inputs(2)
    Ntil = N * n_c
    G = O.chunk_gradients(X, y, w, N, n_c, O.LSQ)
    w1 = O.sgd_step(w, G.sum(axis=0), 0.1, Ntil)
    h = 1e-6
    fd = np.array([(O.full_loss(X, y, w + h * e, Ntil, 64, O.LSQ)
                    - O.full_loss(X, y, w - h * e, Ntil, 64, O.LSQ)) / (2 * h) for e in np.eye(d)])
    assert np.allclose(w1, w - 0.1 * fd, rtol=0, atol=1e-7)


# ---------------------------------------------------------------- ordering
@pytest.mark.parametrize("N,delta", [(6, 3), (20, 4), (64, 8), (128, 6), (256, 16)])
def test_cyclic_order_is_optimal_ordering(N, delta):
    """Sec. III: every column of O holds 1..delta once; the lower bound
    max_i sum_j O_ij >= delta(delta+1)/2 is met with equality by the cyclic
    order, so Q_max = delta(delta+1)/2 + (m - delta - 1) delta."""
    order = O.cyclic_order(N, N, delta)
    A, Om = O.ordering_matrix(order, N)
    for j in range(N):
        col = sorted(int(v) for v in Om[:, j] if v)
        assert col == list(range(1, delta + 1))
    assert np.all(A.sum(axis=0) == delta) and np.all(A.sum(axis=1) == delta)
    rows = Om.astype(int).sum(axis=1)
    assert rows.max() == delta * (delta + 1) // 2
    Q = O.q_metric(Om, delta)
    assert Q.max() == delta * (delta + 1) // 2 + (N - delta - 1) * delta

"""Completion times and the encode-and-transmit trigger (Sec. IV simulation).

CPU: the oracle's order-statistic form is pinned against the definition
(scan the events in time order and evaluate the error estimate of eq. (7)
with the pinned oracle functions), a closed form at equal speeds, and the
impossible case.  GPU: the library is bit-exact with the oracle on the
paper's exact-GC (cyclic, N = m = 200, delta = 8, delta - ell failures) and
approximate-GC (random 8-regular G1 with m = 200, Algorithm 2 order, 7
failures) scenarios, and the psi it returns feeds the batched decode."""
import math

import numpy as np
import pytest
import torch

import oracle as O
from workloads import make_worker_times, random_regular_graph


def _scan_definition(order, tau_r, N, ell, theta):
    """First event time at which sum_i max(0, ell - Delta_i) <= theta, with
    psi(T) and Delta_i from the oracle's completed-set functions."""
    m, delta = order.shape
    dj = (order >= 0).sum(axis=1)
    events = sorted({float(p) * float(tau_r[j]) for j in range(m) if math.isfinite(tau_r[j])
                     for p in range(1, dj[j] + 1)})
    for t in [0.0] + events:
        psi = np.array([sum(1 for p in range(1, dj[j] + 1)
                            if math.isfinite(tau_r[j]) and float(p) * float(tau_r[j]) <= t)
                        for j in range(m)])
        if O.error_estimate(order, psi, N, ell) <= theta:
            return t, psi
    return math.inf, None


@pytest.mark.parametrize("ell,theta,alpha", [(1, 0, 0), (2, 0, 2), (3, 4, 1), (2, 30, 6)])
def test_trigger_is_first_time_estimate_reaches_theta(ell, theta, alpha):
    N, delta = 12, 4
    order = O.cyclic_order(N, N, delta)
    tau = make_worker_times(N, 40, 3, alpha=alpha)
    T, psi, _ = O.completion_times(order, tau, N, ell, theta)
    for r in range(tau.shape[0]):
        t_ref, psi_ref = _scan_definition(order, tau[r], N, ell, theta)
        assert T[r] == t_ref
        if psi_ref is not None:
            assert np.array_equal(psi[r], psi_ref)
            if theta == 0:
                assert O.is_exact(order, psi[r], N, ell)


def test_trigger_full_finishers_definition():
    """T_full: copies count only at delta_j tau_j (the original protocol)."""
    N, delta, ell = 10, 3, 2
    order = O.cyclic_order(N, N, delta)
    tau = make_worker_times(N, 30, 4, alpha=1)
    _, _, TF = O.completion_times(order, tau, N, ell)
    for r in range(tau.shape[0]):
        fin = sorted(float(delta) * t for t in tau[r] if math.isfinite(t))
        best = math.inf
        for t in fin:  # first finishing time at which every chunk has ell finished holders
            done = [j for j in range(N) if math.isfinite(tau[r, j]) and float(delta) * tau[r, j] <= t]
            cnt = np.zeros(N, dtype=int)
            for j in done:
                cnt[order[j]] += 1
            if cnt.min() >= ell:
                best = t
                break
        assert TF[r] == best


def test_equal_speeds_closed_form():
    """All tau_j = 1: every chunk sits in slots 1..delta of its holders
    (cyclic), so T = ell and T_full = delta (ratio delta / ell)."""
    N, delta = 20, 4
    order = O.cyclic_order(N, N, delta)
    tau = np.ones((3, N))
    for ell in range(1, delta + 1):
        T, psi, TF = O.completion_times(order, tau, N, ell)
        assert np.all(T == ell) and np.all(TF == delta) and np.all(psi == ell)


def test_impossible_is_inf_and_theta_monotone():
    N, delta = 8, 3
    order = O.cyclic_order(N, N, delta)
    tau = np.ones((1, N))
    tau[0, :delta] = np.inf  # every holder of chunk delta-1... fails
    T, _, TF = O.completion_times(order, tau, N, 1)
    assert math.isinf(T[0]) and math.isinf(TF[0])
    tau = make_worker_times(N, 20, 9)
    prev = None
    for theta in range(0, 3 * N, 3):
        T, _, _ = O.completion_times(order, tau, N, 3, theta)
        if prev is not None:
            assert np.all(T <= prev)
        prev = T


# ------------------------------------------------------------------ GPU
@pytest.fixture(scope="module")
def gc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2405_19509_gb300 as m
    return m


def _gpu_vs_oracle(gc, order, N, ell, theta, tau):
    m, delta = order.shape
    dev = torch.device("cuda")
    res = gc.gc_trigger_times(torch.from_numpy(order).to(dev), N, m, delta,
                              torch.from_numpy(np.ascontiguousarray(tau)).to(dev), ell, theta)
    T, psi, TF = O.completion_times(order, tau, N, ell, theta)
    assert np.array_equal(res["T"].cpu().numpy(), T)
    assert np.array_equal(res["T_full"].cpu().numpy(), TF)
    assert np.array_equal(res["psi"].cpu().numpy(), psi)
    return res


@pytest.mark.gpu
@pytest.mark.parametrize("ell", [1, 2, 3, 4])
def test_gpu_trigger_exact_gc_cyclic_200(gc, ell):
    N, delta = 200, 8
    order = O.cyclic_order(N, N, delta)
    tau = make_worker_times(N, 300, 11, alpha=delta - ell)
    res = _gpu_vs_oracle(gc, order, N, ell, 0, tau)
    r = (res["T_full"] / res["T"]).mean().item()
    assert 1.5 < r < 3.0  # the proposed protocol finishes about twice as early


@pytest.mark.gpu
@pytest.mark.parametrize("ell,theta", [(1, 0), (2, 5), (3, 50), (8, 0)])
def test_gpu_trigger_regular_graph_alg2(gc, ell, theta):
    m, nu = 200, 8
    A = random_regular_graph(m, nu, 1)
    order, _ = gc.gc_chunk_ordering(A)
    tau = make_worker_times(m, 200, 12, alpha=nu - 1)
    _gpu_vs_oracle(gc, order, m, ell, theta, tau)


@pytest.mark.gpu
def test_gpu_trigger_edge_cases(gc):
    N, delta = 16, 4
    order = O.cyclic_order(N, N, delta)
    tau = np.ones((5, N))
    tau[1, :delta] = np.inf                 # chunk delta-1 has no live holder
    tau[2, :] = np.inf                      # everyone failed
    tau[3] = np.arange(1, N + 1)            # distinct speeds
    for ell in (1, 3):
        for theta in (0, 7, N * ell, N * ell + 5):
            _gpu_vs_oracle(gc, order, N, ell, theta, tau)
    # uneven explicit order (empty slots)
    ex = O.cyclic_order(N, N, delta).copy()
    ex[3, 2:] = -1
    ex[7, 1:] = -1
    _gpu_vs_oracle(gc, ex, N, 2, 0, make_worker_times(N, 50, 13, alpha=2))


@pytest.mark.gpu
@pytest.mark.parametrize("ell", [1, 2, 3])
def test_gpu_trigger_feeds_decode_on_g1(gc, ell):
    """Simulate -> trigger at a theta -> psi -> batched Algorithm 1 and
    decode on the G1-like graph with the Algorithm 2 order; per-pattern
    coefficient error equals the oracle's and the estimate equals the
    trigger's threshold bound."""
    from workloads import get, make_R
    m, nu, theta = 200, 8, 20
    A = random_regular_graph(m, nu, 1)
    order, _ = gc.gc_chunk_ordering(A)
    tau = make_worker_times(m, 256, 14, alpha=nu - 1)
    dev = torch.device("cuda")
    od = torch.from_numpy(order).to(dev)
    res = gc.gc_trigger_times(od, m, m, nu, torch.from_numpy(tau).to(dev), ell, theta)
    psi = res["psi"]
    R = np.random.default_rng(100 + ell).standard_normal((ell, m))
    Rd = torch.from_numpy(R).to(dev)
    rng = np.random.default_rng(7)
    G = torch.from_numpy(rng.standard_normal((m, 64 * ell)).astype(np.float32)).to(dev)
    out = gc.gc_decode_batch(Rd, ell, od, m, m, nu, psi, G)
    est = out["est"].cpu().numpy()
    ce = out["coef_err"].cpu().numpy()
    Tn = res["T"].cpu().numpy()
    psi_np = psi.cpu().numpy()
    for b in range(0, psi_np.shape[0], 16):
        if math.isfinite(Tn[b]):
            assert est[b] <= theta
        r = O.run_pattern(R, order, psi_np[b], m, G.cpu().numpy().astype(np.float64),
                          want_transmit=False)
        assert est[b] == r.est
        assert abs(ce[b] - r.coef_err) <= 1e-9 * max(1.0, r.coef_err)
        ref = r.ghat
        gh = out["Ghat"][b].cpu().numpy()
        assert np.max(np.abs(gh - ref)) <= 1e-4 * max(np.max(np.abs(ref)), 1e-30)

"""GPU vs oracle parity on the five synthetic workloads at their full sizes.

Where the oracle cannot redo a whole batch (it takes seconds per pattern at
d = 2^20), it checks sampled patterns one by one, and properties that hold at
any size are checked on every pattern: the per-pattern rank identity
coef_err == estimate (eq. 7 with rank(R_S) = min(l, Delta)), and exact
recovery of sum_i g_i whenever every chunk has >= l processed copies.
Chunk gradients fed to the decode tests are the oracle's (cast to fp32) or
given synthetic data, never the CUDA path's own output.
"""
import dataclasses
import math

import numpy as np
import pytest
import torch

import oracle as O
from _parity import (assert_grad_close, assert_mse_close, dev_tensors, rel_inf, to_np)
from workloads import get, make_chunk_grads, make_data, make_patterns, make_R

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2405_19509_gb300 as m
    return m


def _sample(npat, k, seed):
    rng = np.random.default_rng(seed)
    first = list(range(min(k // 2, npat)))
    rest = rng.choice(npat, size=min(k - len(first), npat), replace=False)
    return sorted(set(first) | set(int(x) for x in rest))


def _edge_patterns(m, delta, ell):
    """Patterns at the edges of the method under the cyclic assignment (chunk
    i0's holders are the workers i0 - p, slot p): every worker finished (exact,
    the baseline gradient), none started (every Delta_i = 0), chunk i0 with
    exactly ell - 1 copies (the holders at slots >= ell - 1 stop just before
    it; every other chunk keeps >= ell), and chunk i0 with no copy."""
    full = np.full(m, delta, dtype=np.int32)
    i0 = m // 2
    short = full.copy()
    for p in range(ell - 1, delta):
        short[(i0 - p) % m] = p
    none = full.copy()
    for p in range(delta):
        none[(i0 - p) % m] = p
    return np.stack([full, np.zeros(m, dtype=np.int32), short, none])


def _copies_cyclic(psi, N, delta):
    p = np.arange(delta)
    holders = (np.arange(N)[:, None] - p[None, :]) % N            # N x delta
    return (psi[:, holders] > p[None, None, :]).sum(axis=2)       # npat x N


def _check_batch(gc, cfg, ell, psi, G32, res, samples, transmit):
    """Full-batch properties plus sampled oracle comparisons."""
    N, m, delta, d = cfg.N, cfg.m, cfg.delta, cfg.d
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    Gref = G32.astype(np.float64)
    gsum = Gref.sum(axis=0)
    floor = 1e-8 * float(gsum @ gsum) / d
    ce, est = to_np(res["coef_err"]), to_np(res["est"])
    # copies per chunk from psi (cyclic: holders of chunk i are workers i - p at slot p)
    p = np.arange(delta)
    holders = (np.arange(N)[:, None] - p[None, :]) % N            # N x delta
    Delta = (psi[:, holders] > p[None, None, :]).sum(axis=2)     # npat x N
    est_ref = np.maximum(0, ell - Delta).sum(axis=1)
    assert np.array_equal(est, est_ref.astype(np.float64))
    assert np.max(np.abs(ce - est)) <= 1e-8 * max(1.0, N * ell)  # rank identity, every pattern
    exact = np.where(Delta.min(axis=1) >= ell)[0]
    if res.get("Ghat") is not None and exact.size:
        Gh = res["Ghat"]
        gs = torch.from_numpy(gsum.astype(np.float32)).cuda()
        idx = torch.from_numpy(exact[:512]).cuda()
        err = (Gh.index_select(0, idx) - gs).abs().max().item()
        assert err <= 1e-4 * float(np.max(np.abs(gsum))), "exact recovery"
    if res.get("grad_mse") is not None and exact.size:
        assert np.all(to_np(res["grad_mse"])[exact] <= floor)
    for b in samples:
        r = O.run_pattern(R, order, psi[b], N, Gref, want_transmit=transmit)
        assert abs(ce[b] - r.coef_err) <= 1e-8, b
        if res.get("Ghat") is not None:
            assert_grad_close(to_np(res["Ghat"][b]), r.ghat, f"{cfg.name} l={ell} b={b}")
        if res.get("grad_mse") is not None:
            assert_mse_close(float(res["grad_mse"][b]), r.grad_mse, floor, f"{cfg.name} l={ell} b={b}")


# ------------------------------------------------------------------ logistic (m = 20)
@pytest.fixture(scope="module")
def logistic_data():
    cfg = get("logistic")
    data = make_data(cfg, "cpu")
    G64 = O.chunk_gradients(data["X"].numpy(), data["y"].numpy(), data["w"].numpy(), cfg.N,
                            cfg.n_c, O.LOGISTIC)
    return cfg, data, G64


def test_logistic_chunk_grads_full(gc, logistic_data):
    cfg, data, G64 = logistic_data
    Xd, yd, wd = data["X"].cuda(), data["y"].cuda(), data["w"].cuda()
    lo = torch.zeros(1, dtype=torch.float64, device="cuda")
    G = gc.gc_chunk_grads(Xd, yd, wd, cfg.N, cfg.n_c, gc.GC_LOGISTIC, loss_out=lo)
    Gn = to_np(G)
    for i in range(cfg.N):
        assert_grad_close(Gn[i], G64[i], f"chunk {i}")
    Lo = O.full_loss(data["X"].numpy(), data["y"].numpy(), data["w"].numpy(), cfg.Ntil, 4096,
                     O.LOGISTIC)
    assert abs(lo.item() - Lo) <= 1e-5 * Lo


@pytest.mark.parametrize("ell", [1, 2, 4])
def test_logistic_decode_batch_full(gc, logistic_data, ell):
    """10^4 shifted-exponential realizations, the batch the benchmark times."""
    cfg, data, G64 = logistic_data
    psi = make_patterns(cfg)
    R = make_R(cfg, ell)
    order = O.cyclic_order(cfg.N, cfg.m, cfg.delta)
    G32 = G64.astype(np.float32)
    Rd, od, pd = dev_tensors(R, order, psi)
    res = gc.gc_decode_batch(Rd, ell, od, cfg.N, cfg.m, cfg.delta, pd, torch.from_numpy(G32).cuda())
    torch.cuda.synchronize()
    _check_batch(gc, cfg, ell, psi, G32, res, _sample(psi.shape[0], 64, ell), transmit=True)


def test_logistic_encode_transmit(gc, logistic_data):
    cfg, data, G64 = logistic_data
    ell = 2
    psi = make_patterns(cfg, npat=32)
    R = make_R(cfg, ell)
    order = O.cyclic_order(cfg.N, cfg.m, cfg.delta)
    G32 = G64.astype(np.float32)
    Rd, od, pd = dev_tensors(R, order, psi)
    T = gc.gc_encode(Rd, ell, od, cfg.N, cfg.m, cfg.delta, pd, torch.from_numpy(G32).cuda())
    gh = gc.gc_decode_tx(Rd, ell, cfg.m, T, cfg.d)
    for b in range(psi.shape[0]):
        r = O.run_pattern(R, order, psi[b], cfg.N, G32.astype(np.float64), want_transmit=True)
        assert rel_inf(to_np(T[b]), r.T) <= 1e-4
        assert_grad_close(to_np(gh[b]), r.ghat, f"b={b}")


# ------------------------------------------------------------------ mse sweep (m = 64, bf16 X)
@pytest.fixture(scope="module")
def sweep_data():
    cfg = get("mse_sweep")
    data = make_data(cfg, "cuda")   # 8.6 GB of bf16 features, generated on the device
    Xh = data["X"].cpu()
    yh, wh = data["y"].cpu().numpy(), data["w"].cpu().numpy()
    G64 = O.chunk_gradients(Xh, yh, wh, cfg.N, cfg.n_c, O.LSQ)
    return cfg, data, G64, Xh, yh, wh


def test_sweep_chunk_grads_full(gc, sweep_data):
    cfg, data, G64, Xh, yh, wh = sweep_data
    lo = torch.zeros(1, dtype=torch.float64, device="cuda")
    G = gc.gc_chunk_grads(data["X"], data["y"], data["w"], cfg.N, cfg.n_c, gc.GC_LSQ, loss_out=lo)
    Gn = to_np(G)
    for i in range(cfg.N):
        assert_grad_close(Gn[i], G64[i], f"chunk {i}")
    Lo = O.full_loss(Xh, yh, wh, cfg.Ntil, 8192, O.LSQ)
    assert abs(lo.item() - Lo) <= 1e-5 * Lo


@pytest.mark.parametrize("p", [0.3, 0.5, 0.7])
@pytest.mark.parametrize("ell", [1, 2, 3])
def test_sweep_mse_full(gc, sweep_data, p, ell):
    """10^5 Binomial(8, p) patterns, errors only (nothing written)."""
    cfg, data, G64, *_ = sweep_data
    psi = make_patterns(cfg, p=p)
    edges = _edge_patterns(cfg.m, cfg.delta, ell)
    psi[:len(edges)] = edges
    D = _copies_cyclic(psi[:len(edges)], cfg.N, cfg.delta)
    assert D[0].min() == cfg.delta and D[1].max() == 0 and D[2].min() == ell - 1 and D[3].min() == 0
    R = make_R(cfg, ell)
    order = O.cyclic_order(cfg.N, cfg.m, cfg.delta)
    G32 = G64.astype(np.float32)
    Rd, od, pd = dev_tensors(R, order, psi)
    res = gc.gc_mse(Rd, ell, od, cfg.N, cfg.m, cfg.delta, pd, torch.from_numpy(G32).cuda())
    torch.cuda.synchronize()
    samples = sorted(set(range(len(edges))) | set(_sample(psi.shape[0], 32, int(p * 10) + ell)))
    _check_batch(gc, cfg, ell, psi, G32, res, samples, transmit=False)


# ------------------------------------------------------------------ decode-dominated (m = 256)
@pytest.fixture(scope="module")
def decode_data():
    cfg = get("decode")
    Gd = make_chunk_grads(cfg, "cuda")
    return cfg, Gd, Gd.cpu().numpy()


@pytest.mark.parametrize("ell,nsamp", [(2, 64), (1, 64), (4, 16)])
def test_decode_full(gc, decode_data, ell, nsamp):
    """4096 patterns x d = 2^20 (Ghat is 17 GB), the edge patterns inside the
    batch.  Every pattern: estimate, rank identity, exact recovery.  Sampled
    patterns (the edges, then the first and random ones): Algorithm 1's
    coefficient error in full and the decoded gradient against the oracle on
    4096 columns of every block (the decode treats columns independently, so
    the oracle on those columns gives those entries exactly); the first
    patterns' gradient MSE against the oracle over all of d."""
    cfg, Gd, G32 = decode_data
    N, m, delta, d = cfg.N, cfg.m, cfg.delta, cfg.d
    psi = make_patterns(cfg)
    edges = _edge_patterns(m, delta, ell)
    psi[:len(edges)] = edges
    R = make_R(cfg, ell)
    order = O.cyclic_order(N, m, delta)
    Rd, od, pd = dev_tensors(R, order, psi)
    res = gc.gc_decode_batch(Rd, ell, od, N, m, delta, pd, Gd)
    torch.cuda.synchronize()
    Gref = G32.astype(np.float64)
    gsum = Gref.sum(axis=0)
    floor = 1e-8 * float(gsum @ gsum) / d
    _check_batch(gc, cfg, ell, psi, G32, {k: v for k, v in res.items() if k != "Ghat"}, [], False)
    L = d // ell
    rng = np.random.default_rng(100 + ell)
    cols = np.unique(np.concatenate([np.arange(1024), np.arange(L - 1024, L),
                                     rng.choice(L, size=2048, replace=False)]))
    full_cols = np.concatenate([k * L + cols for k in range(ell)])
    Gs = Gref[:, full_cols]
    samples = sorted(set(range(len(edges))) | set(_sample(psi.shape[0], nsamp - len(edges), ell)))
    idx = torch.from_numpy(np.array(samples)).cuda()
    cidx = torch.from_numpy(full_cols).cuda()
    Gh = to_np(res["Ghat"].index_select(0, idx).index_select(1, cidx))
    ce = to_np(res["coef_err"])
    mse = to_np(res["grad_mse"])
    for n, b in enumerate(samples):
        B = O.encoding_matrix(R, order, psi[b], N)
        assert abs(ce[b] - O.coefficient_error(R, B, N)) <= 1e-8, b
        assert_grad_close(Gh[n], O.decode_fused(R, B, Gs), f"decode l={ell} b={b} (sampled columns)")
        if n < 4:
            gm = O.gradient_mse(O.decode_fused(R, B, Gref), gsum)
            assert_mse_close(float(mse[b]), gm, floor, f"decode l={ell} b={b} mse")
    del res
    torch.cuda.empty_cache()


@pytest.mark.parametrize("npat", [1, 8])
def test_decode_encode_full(gc, decode_data, npat):
    """Eq. (2) at the decode batch's shape (m = N = 256, delta = 16, the
    16-slot ring, L = 2^19) for one pattern and for eight: the transmissions
    of every worker on 4096 columns of each block against the oracle on those
    columns (the encode treats columns independently); patterns: every worker
    done, a mixed straggler pattern, and the rest drawn from the workload."""
    cfg, Gd, G32 = decode_data
    N, m, delta, d, ell = cfg.N, cfg.m, cfg.delta, cfg.d, 2
    L = d // ell
    psi = make_patterns(cfg)[:npat].copy()
    psi[0] = delta
    if npat > 1:
        psi[1] = np.random.default_rng(41).integers(0, delta + 1, size=m)
    R = make_R(cfg, ell)
    order = O.cyclic_order(N, m, delta)
    Rd, od, pd = dev_tensors(R, order, psi)
    T = gc.gc_encode(Rd, ell, od, N, m, delta, pd, Gd)
    torch.cuda.synchronize()
    rng = np.random.default_rng(300 + npat)
    cols = np.unique(np.concatenate([np.arange(1024), np.arange(L - 1024, L),
                                     rng.choice(L, size=2048, replace=False)]))
    full_cols = np.concatenate([k * L + cols for k in range(ell)])
    Gs = G32[:, full_cols].astype(np.float64)
    Ts = to_np(T.index_select(2, torch.from_numpy(cols).cuda()))
    for b in sorted({0, npat - 1} | ({1} if npat > 1 else set())):
        r = O.run_pattern(R, order, psi[b], N, Gs, want_transmit=True)
        assert rel_inf(Ts[b], r.T) <= 1e-4, f"encode npat={npat} b={b} (sampled columns)"
    del T
    torch.cuda.empty_cache()


# ------------------------------------------------------------------ coded SGD (m = 128)
def _sgd_run_gpu(gc, cfg, data, ell, iters):
    N, m, delta = cfg.N, cfg.m, cfg.delta
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    Rd = torch.from_numpy(R).cuda()
    od = torch.from_numpy(order).cuda()
    w = torch.zeros(cfg.d, dtype=torch.float32, device="cuda")
    losses = torch.zeros(iters, dtype=torch.float64, device="cuda")
    ws = gc.Workspace()
    ws2 = gc.Workspace()
    ws_hist, gh_hist = [], []
    for t in range(iters):
        psi = torch.from_numpy(make_patterns(cfg, npat=1, stream=t)).cuda()
        G = gc.gc_chunk_grads(data["X"], data["y"], w, N, cfg.n_c, gc.GC_LOGISTIC,
                              loss_out=losses[t:t + 1], ws=ws)
        T = gc.gc_encode(Rd, ell, od, N, m, delta, psi, G, ws=ws2)
        gh = gc.gc_decode_tx(Rd, ell, m, T, cfg.d)
        gh_hist.append(gh[0].clone())
        gc.gc_sgd_step(w, gh[0], cfg.lr, cfg.Ntil)
        ws_hist.append(w.clone())
    gc.gc_status(ws)
    gc.gc_status(ws2)
    return to_np(losses), [to_np(x) for x in ws_hist], [to_np(x) for x in gh_hist]


def _sgd_run_oracle(cfg, X, y, ell, iters, w_force=None):
    N, m, delta = cfg.N, cfg.m, cfg.delta
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    w = np.zeros(cfg.d)
    losses, ws, ghs = [], [], []
    for t in range(iters):
        if w_force is not None and t > 0:
            w = w_force[t - 1].astype(np.float64)   # teacher forcing on the GPU's w_t
        psi = make_patterns(cfg, npat=1, stream=t)[0]
        G = O.chunk_gradients(X, y, w, N, cfg.n_c, O.LOGISTIC)
        losses.append(O.full_loss(X, y, w, cfg.Ntil, 16384, O.LOGISTIC))
        B = O.encoding_matrix(R, order, psi, N)
        gh = O.decode(R, O.encode(B, G, order, psi, ell), cfg.d)
        ghs.append(gh)
        w = O.sgd_step(w, gh, cfg.lr, cfg.Ntil)
        ws.append(w)
    return np.array(losses), ws, ghs


def test_sgd_reduced_trajectory_free_running(gc):
    """All 64 iterations, free running, on the m = 128 cluster with 64 points
    per chunk: loss trajectory within 1e-3 relative, final w within 1e-4."""
    cfg = dataclasses.replace(get("sgd"), n_c=64)
    data = make_data(cfg, "cpu", w_which="zero")
    dd = {k: v.cuda() for k, v in data.items()}
    ell = cfg.ell
    lg, wg, _ = _sgd_run_gpu(gc, cfg, dd, ell, cfg.iters)
    lo, wo, _ = _sgd_run_oracle(cfg, data["X"].numpy(), data["y"].numpy(), ell, cfg.iters)
    assert abs(lg[0] - math.log(2.0)) <= 1e-7          # w_0 = 0: every point costs log 2
    assert np.max(np.abs(lg - lo) / lo) <= 1e-3
    assert rel_inf(wg[-1], wo[-1]) <= 1e-4


def _chunk_pass_threaded(X, y, w, N, n_c, pool):
    """The oracle's chunk gradients and total loss at w, one chunk per task
    (the oracle's own per-chunk functions; NumPy releases the GIL in its
    casts and products, so the chunks run side by side)."""
    def one(i):
        rows = slice(i * n_c, (i + 1) * n_c)
        return (O.chunk_gradient(X[rows], y[rows], w, O.LOGISTIC),
                float(np.sum(O.point_losses(X[rows], y[rows], w, O.LOGISTIC))))
    out = list(pool.map(one, range(N)))
    return np.stack([g for g, _ in out]), sum(l for _, l in out)


def test_sgd_full_size_free_running(gc):
    """Full size (X is 8.6 GB, N~ = 262,144 points): all 64 coded-SGD
    iterations on the GPU and, free running from w_0 = 0, in the oracle (Sec.
    I: w <- w - lr * ghat / N~ with ghat the decoded sum of chunk gradients):
    the loss trajectory within 1e-3 relative, the decoded gradient of every
    8th iteration within 1e-4, and the final w within 1e-4."""
    import os
    from concurrent.futures import ThreadPoolExecutor

    cfg = get("sgd")
    data = make_data(cfg, "cuda", w_which="zero")
    ell = cfg.ell
    lg, wg, gg = _sgd_run_gpu(gc, cfg, data, ell, cfg.iters)
    assert abs(lg[0] - math.log(2.0)) <= 1e-7
    X = data["X"].cpu().numpy()
    y = data["y"].cpu().numpy()
    del data
    torch.cuda.empty_cache()
    N, m, delta = cfg.N, cfg.m, cfg.delta
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    w = np.zeros(cfg.d)
    lo, go = [], []
    with ThreadPoolExecutor(max_workers=max(2, os.cpu_count() or 2)) as pool:
        for t in range(cfg.iters):
            psi = make_patterns(cfg, npat=1, stream=t)[0]
            G, tot = _chunk_pass_threaded(X, y, w, N, cfg.n_c, pool)
            lo.append(tot / cfg.Ntil)
            B = O.encoding_matrix(R, order, psi, N)
            gh = O.decode(R, O.encode(B, G, order, psi, ell), cfg.d)
            go.append(gh)
            w = O.sgd_step(w, gh, cfg.lr, cfg.Ntil)
    lo = np.array(lo)
    assert np.max(np.abs(lg - lo) / lo) <= 1e-3
    assert lg[-1] < lg[0]
    for t in range(0, cfg.iters, 8):
        assert_grad_close(gg[t], go[t], f"iteration {t}")
    assert rel_inf(wg[-1], w) <= 1e-4

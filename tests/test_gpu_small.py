"""GPU vs oracle parity on small inputs: the 6-worker workload brute-forced
over every straggler pattern, ragged and degenerate shapes, explicit
(non-uniform) orders, every cluster width of the chunk-gradient kernel, and
device-detected bad data.  All calls go through the C-ABI (ctypes binding)."""
import json
import os

import numpy as np
import pytest
import torch

import oracle as O
from _parity import (COEF_RTOL, assert_grad_close, assert_mse_close, dev_tensors, rel_inf, to_np)
from workloads import all_patterns, get, make_data, make_patterns, make_R

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.fixture(scope="module")
def gc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2405_19509_gb300 as m
    return m


def _tiny_patterns(cfg):
    return np.concatenate([all_patterns(cfg.m, cfg.delta), make_patterns(cfg)])


# ------------------------------------------------------------------ Algorithm 1
@pytest.mark.parametrize("ell", [1, 2, 3])
def test_tiny_coefficients_all_patterns(gc, ell):
    """Every psi in {0..3}^6 plus the 256 seeded ones: Delta and the supports
    bit-exact, E (Algorithm 1) to 1e-9, C = R B, coefficient error and
    estimate, through both the memo-table path and the direct path."""
    cfg = get("tiny")
    N, m, delta = cfg.N, cfg.m, cfg.delta
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    psi = _tiny_patterns(cfg)
    Rd, od, pd = dev_tensors(R, order, psi)
    big = gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, pd, support=True)   # table path
    ws = gc.Workspace()
    small = gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, pd[:3], support=True, ws=ws)  # direct
    gc.gc_status(ws)
    for k in ("E", "C", "coef_err", "delta"):
        assert torch.equal(small[k], big[k][:3]), f"table and direct paths differ in {k}"
    E, C, D, S = to_np(big["E"]), to_np(big["C"]), to_np(big["delta"]), to_np(big["support"])
    ce, est = to_np(big["coef_err"]), to_np(big["est"])
    for b in range(psi.shape[0]):
        r = O.run_pattern(R, order, psi[b], N)
        assert np.array_equal(D[b], r.Delta), b
        assert np.array_equal(S[b], r.support), b
        assert rel_inf(E[b], r.E) <= COEF_RTOL, b
        assert np.max(np.abs(C[b] - r.C)) <= 2e-6, b
        assert abs(ce[b] - r.coef_err) <= 1e-9, b
        assert est[b] == r.est, b


def test_worked_example_explicit_order(gc):
    """Sec. II-B's five-worker example (non-uniform loads, a failed worker,
    -1 slots): supports of eqs. (3) and (8) and the coefficients."""
    with open(os.path.join(HERE, "golden", "worked_example.json")) as f:
        g = json.load(f)
    ex = np.array(g["order"], dtype=np.int32)
    N, m, ell = g["N"], g["m"], g["ell"]
    delta = ex.shape[1]
    A, order, Om = gc.gc_make_assignment(N, m, delta, gc.GC_EXPLICIT, ex)
    R = np.random.default_rng(31).standard_normal((ell, m))
    psi = np.array([c["psi"] for c in g["cases"]], dtype=np.int32)
    Rd, od, pd = dev_tensors(R, order, psi)
    res = gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, pd, support=True)
    for b, case in enumerate(g["cases"]):
        assert np.array_equal(to_np(res["support"][b]).T, np.array(case["B_support_worker_by_chunk"]))
        assert list(to_np(res["delta"][b])) == case["Delta"]
        assert res["est"][b].item() == case["estimate"]
        r = O.run_pattern(R, order, psi[b], N)
        assert rel_inf(to_np(res["E"][b]), r.E) <= COEF_RTOL
        assert abs(res["coef_err"][b].item() - r.coef_err) <= 1e-9


# ------------------------------------------------------------------ decode paths
@pytest.mark.parametrize("ell", [1, 2, 3])
def test_tiny_decode_batch_and_transmit_all_patterns(gc, ell):
    """Batched decode-combine and the worker-encode / PS-decode path against
    the oracle's transmit path, every pattern; l = 3 does not divide d = 64
    (zero-padded last block)."""
    cfg = get("tiny")
    N, m, delta, d = cfg.N, cfg.m, cfg.delta, cfg.d
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    psi = _tiny_patterns(cfg)
    data = make_data(cfg)
    G64 = O.chunk_gradients(data["X"].numpy(), data["y"].numpy(), data["w"].numpy(), N, cfg.n_c, O.LSQ)
    G32 = G64.astype(np.float32)
    Gref = G32.astype(np.float64)
    Rd, od, pd = dev_tensors(R, order, psi)
    Gd = torch.from_numpy(G32).cuda()
    res = gc.gc_decode_batch(Rd, ell, od, N, m, delta, pd, Gd)
    T = gc.gc_encode(Rd, ell, od, N, m, delta, pd, Gd)
    gh = gc.gc_decode_tx(Rd, ell, m, T, d)
    Gh, Tn, ghn = to_np(res["Ghat"]), to_np(T), to_np(gh)
    mse = to_np(res["grad_mse"])
    gsum = Gref.sum(axis=0)
    floor = 1e-8 * float(gsum @ gsum) / d
    for b in range(psi.shape[0]):
        r = O.run_pattern(R, order, psi[b], N, Gref, want_transmit=True)
        assert_grad_close(Gh[b], r.ghat, f"combine b={b}")
        assert_grad_close(ghn[b], r.ghat, f"transmit b={b}")
        if np.max(np.abs(r.T)) > 0:
            assert rel_inf(Tn[b], r.T) <= 1e-4, b
        else:
            assert np.all(Tn[b] == 0)
        assert_mse_close(mse[b], r.grad_mse, floor, f"mse b={b}")


def test_degenerate_shapes(gc):
    """d < ell (empty trailing blocks), psi all zero (nothing decoded), all
    finished (baseline gradient), npat = 0 (no launch)."""
    rng = np.random.default_rng(3)
    N = m = 5
    delta = 3
    order = O.cyclic_order(N, m, delta)
    for d, ell in [(2, 3), (5, 4), (1, 1), (7, 8)]:
        if ell > 8:
            continue
        R = rng.standard_normal((ell, m))
        G = rng.standard_normal((N, d)).astype(np.float32)
        psi = np.array([[0] * m, [delta] * m, [1, 0, 3, 2, 1]], dtype=np.int32)
        Rd, od, pd = dev_tensors(R, order, psi)
        res = gc.gc_decode_batch(Rd, ell, od, N, m, delta, pd, torch.from_numpy(G).cuda())
        Gh = to_np(res["Ghat"])
        assert np.all(Gh[0] == 0.0)
        for b in range(3):
            r = O.run_pattern(R, order, psi[b], N, G.astype(np.float64))
            assert_grad_close(Gh[b], r.ghat, f"d={d} ell={ell} b={b}")
            assert res["est"][b].item() == r.est
    # npat = 0: nothing to do, outputs untouched
    R = rng.standard_normal((2, m))
    Rd, od, pd = dev_tensors(R, order, np.zeros((0, m), dtype=np.int32))
    res = gc.gc_decode_batch(Rd, 2, od, N, m, delta, pd, torch.zeros(N, 8, device="cuda"))
    assert res["Ghat"].shape == (0, 8)


def test_large_ell_and_explicit_uneven(gc):
    """l = 8 (the build's maximum) with delta = 8, and an explicit order with
    N != m and uneven replication."""
    rng = np.random.default_rng(4)
    N = m = 16
    delta, ell, d = 8, 8, 40
    order = O.cyclic_order(N, m, delta)
    R = rng.standard_normal((ell, m))
    G = rng.standard_normal((N, d)).astype(np.float32)
    psi = rng.integers(0, delta + 1, size=(40, m)).astype(np.int32)
    psi[0] = delta
    Rd, od, pd = dev_tensors(R, order, psi)
    res = gc.gc_decode_batch(Rd, ell, od, N, m, delta, pd, torch.from_numpy(G).cuda())
    for b in range(psi.shape[0]):
        r = O.run_pattern(R, order, psi[b], N, G.astype(np.float64), want_transmit=False)
        assert_grad_close(to_np(res["Ghat"][b]), r.ghat, f"ell=8 b={b}")
        assert abs(res["coef_err"][b].item() - r.coef_err) <= 1e-8
    # explicit: 4 chunks, 6 workers, ragged loads
    ex = np.array([[0, 1, 2], [1, 3, -1], [2, -1, -1], [3, 0, 1], [0, -1, -1], [2, 3, 0]],
                  dtype=np.int32)
    N2, m2, dl2 = 4, 6, 3
    _, order2, _ = gc.gc_make_assignment(N2, m2, dl2, gc.GC_EXPLICIT, ex)
    ell = 2
    R2 = rng.standard_normal((ell, m2))
    G2 = rng.standard_normal((N2, 10)).astype(np.float32)
    psi2 = np.array([[3, 2, 1, 3, 1, 3], [1, 1, 0, 2, 0, 1], [0, 0, 0, 0, 0, 0], [2, 2, 1, 1, 1, 2]],
                    dtype=np.int32)
    Rd, od, pd = dev_tensors(R2, order2, psi2)
    res = gc.gc_decode_batch(Rd, ell, od, N2, m2, dl2, pd, torch.from_numpy(G2).cuda())
    for b in range(psi2.shape[0]):
        r = O.run_pattern(R2, order2, psi2[b], N2, G2.astype(np.float64))
        assert_grad_close(to_np(res["Ghat"][b]), r.ghat, f"explicit b={b}")
        assert res["est"][b].item() == r.est


# ------------------------------------------------------------------ chunk gradients
@pytest.mark.parametrize("d,n_c,N,dtype,loss", [
    (64, 32, 6, torch.float32, 0),       # tiny
    (65, 7, 3, torch.float32, 1),        # ragged d (no TMA), odd n_c
    (8, 1, 5, torch.float32, 0),         # one row per chunk
    (4096, 16, 2, torch.float32, 1),     # one CTA per row
    (16384, 8, 3, torch.float32, 0),     # cluster of 2
    (32768, 4, 2, torch.float32, 1),     # cluster of 4
    (65536, 4, 2, torch.float32, 0),     # cluster of 4 with 64 KB slices (8 vectors a thread)
    (40000, 3, 2, torch.float32, 1),     # cluster of 4, 8-vector threads partly past the slice
    (40001, 2, 2, torch.float32, 0),     # the same without TMA (row not a 16-byte multiple)
    (65536, 8, 2, torch.bfloat16, 0),    # bf16, cluster of 4 with 32 KB slices
    (131072, 2, 2, torch.bfloat16, 1),   # bf16, cluster of 8 with 32 KB slices
    (16384, 3, 3, torch.float32, 1),     # cluster of 2, one row per stage (3 rows a chunk)
    (32768, 6, 2, torch.bfloat16, 1),    # bf16 cluster of 4, two rows per stage
    (4000, 5, 3, torch.bfloat16, 0),     # bf16, 256 threads x 2 vectors, slice shorter than the stage row
    (2048, 8, 2, torch.float32, 1),      # 256 threads x 2 vectors
    (600, 4, 3, torch.float32, 0),       # 128 threads x 2 vectors
    (100, 6, 4, torch.bfloat16, 1),      # bf16 ragged (no TMA)
    (1024, 2048, 1, torch.float32, 1),   # one chunk spanning many clusters
])
def test_chunk_grads_shapes(gc, d, n_c, N, dtype, loss):
    g = torch.Generator().manual_seed(d * 7 + n_c)
    X = torch.randn(N * n_c, d, generator=g)
    if loss == 1:
        X /= d ** 0.5
        y = torch.where(torch.rand(N * n_c, generator=g) < 0.5, 1.0, -1.0)
    else:
        y = torch.randn(N * n_c, generator=g)
    w = (torch.randn(d, generator=g) / d ** 0.5).float()
    X = X.to(dtype)
    Xd, yd, wd = X.cuda(), y.cuda(), w.cuda()
    lo = torch.zeros(1, dtype=torch.float64, device="cuda")
    ws = gc.Workspace()
    G = gc.gc_chunk_grads(Xd, yd, wd, N, n_c, loss, loss_out=lo, ws=ws)
    gc.gc_status(ws)
    Go = O.chunk_gradients(X, y.numpy(), w.numpy(), N, n_c, loss)
    for i in range(N):
        assert_grad_close(to_np(G[i]), Go[i], f"chunk {i}")
    Lo = O.full_loss(X, y.numpy(), w.numpy(), N * n_c, 4096, loss)
    assert abs(lo.item() - Lo) <= 1e-5 * abs(Lo)


def test_chunk_grads_unaligned_X(gc):
    """An X view starting 4 bytes past a 16-byte boundary takes the plain-load path."""
    N, n_c, d = 3, 8, 256
    base = torch.randn(N * n_c * d + 1, generator=torch.Generator().manual_seed(9))
    X = base[1:].view(N * n_c, d)
    y = torch.randn(N * n_c, generator=torch.Generator().manual_seed(10))
    w = torch.randn(d, generator=torch.Generator().manual_seed(11)) / 16
    Xd = base.cuda()[1:].view(N * n_c, d)
    assert Xd.data_ptr() % 16 != 0
    G = gc.gc_chunk_grads(Xd, y.cuda(), w.cuda(), N, n_c, 0)
    Go = O.chunk_gradients(X, y.numpy(), w.numpy(), N, n_c, 0)
    assert_grad_close(to_np(G), Go, "unaligned")


def test_sgd_step(gc):
    d = 1000
    w = torch.randn(d, generator=torch.Generator().manual_seed(1))
    gh = torch.randn(d, generator=torch.Generator().manual_seed(2))
    wd = w.cuda()
    gc.gc_sgd_step(wd, gh.cuda(), 0.1, 4096)
    ref = O.sgd_step(w.numpy(), gh.numpy(), 0.1, 4096)
    assert np.max(np.abs(to_np(wd) - ref)) <= 1e-6 * (1 + np.max(np.abs(ref)))


# ------------------------------------------------------------------ device-detected bad data
def test_bad_psi_flagged(gc):
    N = m = 6
    delta, ell = 3, 2
    order = O.cyclic_order(N, m, delta)
    R = make_R(get("tiny"), ell)
    psi = np.array([[0, 1, 2, 3, 4, 0], [-1, 0, 0, 0, 0, 0]], dtype=np.int32)   # 4 > delta, -1 < 0
    Rd, od, pd = dev_tensors(R, order, psi)
    ws = gc.Workspace()
    gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, pd, ws=ws)
    with pytest.raises(gc.GCError) as ei:
        gc.gc_status(ws)
    assert ei.value.code == -7 and "psi" in str(ei.value)
    gc.gc_status(ws)  # cleared


def test_singular_R_flagged(gc):
    """Two identical columns of R make X = R[:, S] rank deficient for a chunk
    held by exactly those two workers."""
    N = m = 6
    delta, ell = 3, 2
    order = O.cyclic_order(N, m, delta)
    R = make_R(get("tiny"), ell)
    R[:, 1] = R[:, 0]
    psi = np.array([[2, 1, 0, 0, 0, 0]], dtype=np.int32)  # chunk 1 done by workers 0 and 1 only
    Rd, od, pd = dev_tensors(R, order, psi)
    ws = gc.Workspace()
    gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, pd, ws=ws)
    with pytest.raises(gc.GCError) as ei:
        gc.gc_status(ws)
    assert ei.value.code == -7 and "rank" in str(ei.value)


def test_encode_with_coeffs_matches_encode(gc):
    """Algorithm 1 then eq. (2) in two calls gives the same transmissions as
    gc_encode, and the oracle's."""
    cfg = get("tiny")
    N, m, delta, d, ell = cfg.N, cfg.m, cfg.delta, cfg.d, 3
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    psi = make_patterns(cfg, npat=40)
    G = np.random.default_rng(12).standard_normal((N, d)).astype(np.float32)
    Rd, od, pd = dev_tensors(R, order, psi)
    Gd = torch.from_numpy(G).cuda()
    E = gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, pd, C=False)["E"]
    T2 = gc.gc_encode_with_coeffs(E, ell, od, N, m, delta, pd, Gd)
    T1 = gc.gc_encode(Rd, ell, od, N, m, delta, pd, Gd)
    assert torch.equal(T1, T2)
    for b in range(psi.shape[0]):
        r = O.run_pattern(R, order, psi[b], N, G.astype(np.float64))
        if np.max(np.abs(r.T)) > 0:
            assert rel_inf(to_np(T2[b]), r.T) <= 1e-4


@pytest.mark.parametrize("explicit", [False, True])
@pytest.mark.parametrize("npat", [1, 3])
def test_encode_long_rows(gc, explicit, npat):
    """Eq. (2) on long rows (L = 2^18, 16-byte column vectors, blocks striding
    over many column stripes) for one pattern and for a group of three, with
    the cyclic order and with an explicit order of disjoint chunk lists (64
    chunks, one copy each): the transmissions equal the oracle's."""
    ell, d, delta = 2, 1 << 19, 4
    rng = np.random.default_rng(31 + 2 * npat + explicit)
    if explicit:
        N, m = 64, 16
        order = np.arange(N, dtype=np.int32).reshape(m, delta)
    else:
        N = m = 16
        order = O.cyclic_order(N, m, delta)
    R = rng.standard_normal((ell, m))
    psi = rng.integers(0, delta + 1, size=(npat, m)).astype(np.int32)
    G = rng.standard_normal((N, d)).astype(np.float32)
    Rd, od, pd = dev_tensors(R, order, psi)
    Gd = torch.from_numpy(G).cuda()
    T = gc.gc_encode(Rd, ell, od, N, m, delta, pd, Gd)
    torch.cuda.synchronize()
    G64 = G.astype(np.float64)
    for b in range(npat):
        r = O.run_pattern(R, order, psi[b], N, G64)
        if np.max(np.abs(r.T)) > 0:
            assert rel_inf(to_np(T[b]), r.T) <= 1e-4, f"pattern {b}"
        else:
            assert float(T[b].abs().max()) == 0.0


@pytest.mark.parametrize("delta,d,ell", [(5, 2600, 2), (9, 2599, 2), (16, 2600, 2), (16, 2599, 2),
                                         (17, 2600, 2), (32, 2600, 2), (16, 2600, 1), (16, 2600, 3),
                                         (16, 2604, 4), (16, 2601, 4)])
def test_encode_ring_sizes(gc, delta, d, ell):
    """Eq. (2) through every ring size of the chunk sweep (8, 16 and 32
    slots, with delta below and at the ring size), with one block of a chunk
    per step (l odd) and two (l even), on column stripes with a ragged last
    one (L = 1300 at l = 2), 16-byte vectors (d = 2600, 2604) and scalar
    columns with padded last blocks (d = 2599, 2601); the patterns include
    every worker done, none done, and mixed.  Few patterns, so the launch
    also splits the workers into groups (each group sweeps its own chunks)."""
    rng = np.random.default_rng(700 + delta + d + 10 * ell)
    N = m = 40
    order = O.cyclic_order(N, m, delta)
    R = rng.standard_normal((ell, m))
    psi = rng.integers(0, delta + 1, size=(4, m)).astype(np.int32)
    psi[0] = delta
    psi[1] = 0
    psi[2, ::3] = 0
    G = rng.standard_normal((N, d)).astype(np.float32)
    Rd, od, pd = dev_tensors(R, order, psi)
    T = to_np(gc.gc_encode(Rd, ell, od, N, m, delta, pd, torch.from_numpy(G).cuda()))
    G64 = G.astype(np.float64)
    for b in range(psi.shape[0]):
        r = O.run_pattern(R, order, psi[b], N, G64, want_transmit=True)
        if np.max(np.abs(r.T)) > 0:
            assert rel_inf(T[b], r.T) <= 1e-4, f"delta={delta} d={d} l={ell} pattern {b}"
        else:
            assert float(np.abs(T[b]).max()) == 0.0


@pytest.mark.parametrize("N,m,delta,d,ell,explicit", [
    (6, 6, 3, 64, 2, False),        # the tiny configuration
    (20, 20, 4, 4099, 3, False),    # padded last block (3 * 1367 > 4099)
    (128, 128, 6, 8192, 2, False),  # the coded-SGD shape
    (12, 6, 2, 130, 2, True),       # explicit, non-cyclic order
    (40, 40, 16, 1000, 1, False),   # l = 1
    (256, 256, 16, 2002, 2, False), # N*l too large to stage the columns: chunk gradients read directly
])
def test_live_step_matches_three_calls(gc, N, m, delta, d, ell, explicit):
    """gc_live_step (one launch) gives the same T, ghat and w, bit for bit, as
    gc_encode_with_coeffs + gc_decode_tx + gc_sgd_step; ghat agrees with the
    oracle's Sec. II-B decode of the eq. (2) transmissions."""
    rng = np.random.default_rng(900 + N + d + ell)
    if explicit:
        order = rng.permutation(N).astype(np.int32).reshape(m, delta)
    else:
        order = O.cyclic_order(N, m, delta)
    R = rng.standard_normal((ell, m))
    psi = rng.integers(0, delta + 1, size=(1, m)).astype(np.int32)
    psi[0, 0] = delta
    G = rng.standard_normal((N, d)).astype(np.float32)
    w0 = rng.standard_normal(d).astype(np.float32)
    Rd, od, pd = dev_tensors(R, order, psi)
    Gd = torch.from_numpy(G).cuda()
    E = gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, pd, C=False)["E"]
    lr, Ntil = 0.25, 1000
    T1 = gc.gc_encode_with_coeffs(E, ell, od, N, m, delta, pd, Gd)
    gh1 = gc.gc_decode_tx(Rd, ell, m, T1, d)
    w1 = torch.from_numpy(w0).cuda()
    gc.gc_sgd_step(w1, gh1[0], lr, Ntil)
    L = gc.block_length(d, ell)
    T2 = torch.empty(m, L, dtype=torch.float32, device="cuda")
    gh2 = torch.empty(d, dtype=torch.float32, device="cuda")
    w2 = torch.from_numpy(w0).cuda()
    gc.gc_live_step(E, Rd, ell, od, N, m, delta, pd, Gd, w2, lr, Ntil, T=T2, ghat=gh2)
    w3 = torch.from_numpy(w0).cuda()
    gc.gc_live_step(E, Rd, ell, od, N, m, delta, pd, Gd, w3, lr, Ntil)   # no T, no ghat
    torch.cuda.synchronize()
    assert torch.equal(T2, T1[0])
    assert torch.equal(gh2, gh1[0])
    assert torch.equal(w2, w1) and torch.equal(w3, w1)
    r = O.run_pattern(R, order, psi[0], N, G.astype(np.float64), want_transmit=True)
    assert_grad_close(to_np(gh2), r.ghat, "live step ghat")


@pytest.mark.parametrize("ell", [1, 3])
def test_decode_plan_then_apply(gc, ell):
    """gc_decode_plan (psi side) then gc_decode_apply (data side) equals
    gc_decode_batch bit for bit and the oracle within tolerance; l = 3 has
    padding columns (N*l = 18 of 64) that the plan must zero."""
    cfg = get("tiny")
    N, m, delta, d = cfg.N, cfg.m, cfg.delta, cfg.d
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    psi = make_patterns(cfg, npat=300, stream=77)
    G = np.random.default_rng(21).standard_normal((N, d)).astype(np.float32)
    Rd, od, pd = dev_tensors(R, order, psi)
    Gd = torch.from_numpy(G).cuda()
    # dirty plan buffer: every byte the apply reads must be written by the plan
    nb = gc.lib.gc_decode_plan_bytes(N, ell, psi.shape[0])
    plan = torch.full((nb,), 0x7f, dtype=torch.uint8, device="cuda")
    pl = gc.gc_decode_plan(Rd, ell, od, N, m, delta, pd, plan=plan)
    ap = gc.gc_decode_apply(pl["plan"], ell, N, psi.shape[0], Gd)
    ref = gc.gc_decode_batch(Rd, ell, od, N, m, delta, pd, Gd)
    assert torch.equal(ap["Ghat"], ref["Ghat"])
    assert torch.equal(ap["grad_mse"], ref["grad_mse"])
    assert torch.equal(pl["coef_err"], ref["coef_err"]) and torch.equal(pl["est"], ref["est"])
    for b in range(0, psi.shape[0], 7):
        r = O.run_pattern(R, order, psi[b], N, G.astype(np.float64), want_transmit=False)
        assert_grad_close(to_np(ap["Ghat"][b]), r.ghat, f"plan/apply b={b}")


@pytest.mark.parametrize("cfg_name,ell,npat", [("tiny", 2, 256), ("tiny", 3, 5), ("logistic", 2, 2000)])
def test_prepared_plan_matches_plan(gc, cfg_name, ell, npat):
    """gc_decode_plan_prepared equals gc_decode_plan bit for bit when the
    latter uses its memo table (npat >= 2^delta), to rounding otherwise; the
    prepared buffer serves several batches."""
    from workloads import get, make_R, make_patterns
    cfg = get(cfg_name)
    N, m, delta = cfg.N, cfg.m, cfg.delta
    order = O.cyclic_order(N, m, delta)
    dev = torch.device("cuda")
    Rd = torch.from_numpy(make_R(cfg, ell)).to(dev)
    od = torch.from_numpy(order).to(dev)
    prep = gc.gc_decode_prepare(Rd, ell, od, N, m, delta)
    for stream in (0, 1):
        psi = torch.from_numpy(make_patterns(cfg, npat=npat, stream=stream)).to(dev)
        a = gc.gc_decode_plan(Rd, ell, od, N, m, delta, psi)
        b = gc.gc_decode_plan_prepared(prep, Rd, ell, N, m, delta, psi)
        torch.cuda.synchronize()
        assert torch.equal(a["est"], b["est"])
        if npat >= 2 ** delta:
            assert torch.equal(a["plan"], b["plan"])
            assert torch.equal(a["coef_err"], b["coef_err"])
        else:
            assert torch.allclose(a["coef_err"], b["coef_err"], rtol=0, atol=1e-9)
            pa = a["plan"].view(torch.bfloat16).float()
            pb = b["plan"].view(torch.bfloat16).float()
            assert torch.allclose(pa, pb, rtol=2 ** -7, atol=1e-6)


def test_prepared_plan_direct_solves_for_large_delta(gc):
    """delta = 16 > 14: no memo table; the prepared call solves every block
    directly and agrees with the oracle's coefficient error."""
    from workloads import get, make_R, make_patterns
    cfg = get("decode")
    N, m, delta, ell = 64, 64, 16, 2
    order = O.cyclic_order(N, m, delta)
    dev = torch.device("cuda")
    R = np.random.default_rng(5).standard_normal((ell, m))
    Rd, od = torch.from_numpy(R).to(dev), torch.from_numpy(order).to(dev)
    psi_np = np.random.default_rng(6).integers(0, delta + 1, size=(40, m)).astype(np.int32)
    prep = gc.gc_decode_prepare(Rd, ell, od, N, m, delta)
    b = gc.gc_decode_plan_prepared(prep, Rd, ell, N, m, delta, torch.from_numpy(psi_np).to(dev))
    ce = b["coef_err"].cpu().numpy()
    for i in range(0, 40, 7):
        r = O.run_pattern(R, order, psi_np[i], N, None, want_transmit=False)
        assert abs(ce[i] - r.coef_err) <= 1e-9 * max(1.0, r.coef_err)
        assert b["est"][i].item() == r.est


def test_maximum_delta_and_replication(gc):
    """delta = 32 (GC_MAX_DELTA) in the cyclic assignment, so every chunk has
    32 holders (GC_MAX_REPL); l = 2 (l = 8 is covered above: the oracle's
    per-worker solve at l = 8 with 32 chunks a worker takes seconds per
    pattern).  Decode, errors and the transmit path against the oracle; the
    trigger kernel on the same assignment."""
    rng = np.random.default_rng(21)
    N = m = 40
    delta, ell, d = 32, 2, 48
    order = O.cyclic_order(N, m, delta)
    R = rng.standard_normal((ell, m))
    G = rng.standard_normal((N, d)).astype(np.float32)
    psi = rng.integers(0, delta + 1, size=(12, m)).astype(np.int32)
    psi[0] = delta
    psi[1] = 0
    psi[2] = rng.integers(0, 2, size=m)  # mostly too few copies: approximate
    Rd, od, pd = dev_tensors(R, order, psi)
    Gd = torch.from_numpy(G).cuda()
    res = gc.gc_decode_batch(Rd, ell, od, N, m, delta, pd, Gd)
    T = gc.gc_encode(Rd, ell, od, N, m, delta, pd[:4].contiguous(), Gd)
    gh = gc.gc_decode_tx(Rd, ell, m, T, d)
    for b in range(psi.shape[0]):
        r = O.run_pattern(R, order, psi[b], N, G.astype(np.float64), want_transmit=b < 4)
        assert_grad_close(to_np(res["Ghat"][b]), r.ghat, f"delta=32 b={b}")
        assert abs(res["coef_err"][b].item() - r.coef_err) <= 1e-8 * max(1.0, r.coef_err)
        assert res["est"][b].item() == r.est
        if b < 4:
            assert_grad_close(to_np(gh[b]), r.ghat, f"delta=32 transmit b={b}")
    from workloads import make_worker_times
    tau = make_worker_times(m, 64, 22, alpha=5)
    out = gc.gc_trigger_times(od, N, m, delta, torch.from_numpy(tau).cuda(), ell, 3)
    Tn, psin, TFn = O.completion_times(order, tau, N, ell, 3)
    assert np.array_equal(out["T"].cpu().numpy(), Tn)
    assert np.array_equal(out["psi"].cpu().numpy(), psin)
    assert np.array_equal(out["T_full"].cpu().numpy(), TFn)


# ------------------------------------------------------------------ the lean Algorithm 1 kernel
@pytest.mark.parametrize("N,delta,ell,npat", [
    (40, 4, 2, 300),     # two chunks a lane, the second group ragged (8 of 32 lanes)
    (64, 8, 2, 400),     # the MSE sweep's shape, memo table (npat >= 2^delta)
    (64, 8, 3, 9),       # direct solves (npat < 2^delta)
    (100, 6, 4, 200),    # four chunks a lane, ragged
    (128, 6, 1, 100),
    (72, 12, 2, 5000),   # twelve holders a chunk: holders past the eighth, table of 2^12 masks
    (48, 16, 2, 30),     # delta = 16: no table, sixteen holders a chunk
])
def test_lean_solve_matches_coefficient_path(gc, N, delta, ell, npat):
    """Without E, Algorithm 1 for N <= 128 runs one warp per pattern with
    several chunks a lane; it must give the Delta, supports, estimate, decode
    blocks and coefficient error of the per-chunk-thread kernel that also
    writes E (bit for bit where both solve; exactly I where that kernel
    rounds a solved full-rank block), and the oracle's within tolerance; bad
    psi entries are flagged and read as 0 on both paths."""
    m = N
    rng = np.random.default_rng(1000 + N + delta + ell)
    order = O.cyclic_order(N, m, delta)
    R = rng.standard_normal((ell, m))
    psi = rng.integers(0, delta + 1, size=(npat, m)).astype(np.int32)
    psi[0] = 0
    psi[1 % npat] = delta
    if npat > 3:
        psi[2, ::3] = ell - 1   # chunks with fewer than ell finishers
    Rd, od, pd = dev_tensors(R, order, psi)
    full = gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, pd, support=True)
    lean = gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, pd, E=False, support=True)
    for k in ("delta", "support", "est"):
        assert torch.equal(lean[k], full[k]), f"lean and coefficient kernels differ in {k}"
    ce, est, D = to_np(lean["coef_err"]), to_np(lean["est"]), to_np(lean["delta"])
    C = to_np(lean["C"])
    # blocks of chunks with Delta >= ell: exactly I on the lean path (Sec. II-A),
    # I to rounding where E is also wanted (that path solves them); the
    # others come from the same solve on both paths, bit for bit
    Cf = to_np(full["C"]).reshape(npat, ell, N, ell)
    Cl = C.reshape(npat, ell, N, ell)
    full_rank = (D >= ell)[:, None, :, None]
    eye = np.broadcast_to(np.eye(ell, dtype=np.float32)[None, :, None, :], Cl.shape)
    assert np.array_equal(np.where(full_rank, Cl, eye), eye)
    assert np.max(np.abs(np.where(full_rank, Cf, eye) - eye)) <= 1e-6
    assert np.array_equal(np.where(full_rank, 0, Cl), np.where(full_rank, 0, Cf))
    assert np.all(np.abs(ce - to_np(full["coef_err"])) <= 1e-12 * np.maximum(1.0, ce))
    for b in sorted({0, 1 % npat, 2 % npat, npat - 1}):
        r = O.run_pattern(R, order, psi[b], N)
        assert np.array_equal(D[b], r.Delta), b
        assert np.max(np.abs(C[b] - r.C)) <= 2e-6, b
        assert abs(ce[b] - r.coef_err) <= 1e-9 * max(1.0, r.coef_err), b
        assert est[b] == r.est, b
    # out-of-range entries: flagged, and read as 0 by both kernels
    bad = psi[:4].copy()
    bad[0, 0], bad[1 % 4, m - 1] = delta + 1, -2
    Rd, od, bd = dev_tensors(R, order, bad)
    outs = []
    for want_E in (True, False):
        ws = gc.Workspace()
        outs.append(gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, bd, E=want_E, ws=ws))
        with pytest.raises(gc.GCError) as ei:
            gc.gc_status(ws)
        assert ei.value.code == -7 and "psi" in str(ei.value)
    zeroed = bad.copy()
    zeroed[(zeroed < 0) | (zeroed > delta)] = 0
    Rd, od, zd = dev_tensors(R, order, zeroed)
    ref = gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, zd, E=False)
    for k in ("delta", "est"):
        assert torch.equal(outs[1][k], outs[0][k]) and torch.equal(outs[1][k], ref[k]), k
    for k in ("C", "coef_err"):
        assert torch.equal(outs[1][k], ref[k]), k

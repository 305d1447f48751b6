"""The two paths of the batched decode against the oracle and each other.

Every decode block Pi_{b,i} is I_ell when Delta_i >= ell (Sec. II-A), so the
library writes the rows of a 128-row tile either as sum_i g_{D_i} plus the
non-identity blocks (residual path) or by the tensor-core GEMM C . G; the
choice is made per tile on the device (gc_set_decode_policy).  These tests
force each policy and let the automatic one mix them: tiles of exact and of
approximate patterns side by side, patterns straddling two tiles (ell = 3),
lists longer than the residual path holds, ragged block lengths, and a
decode matrix that is not a projector (gc_decode_combine)."""
import numpy as np
import pytest
import torch

import oracle as O
from _parity import assert_grad_close, assert_mse_close, dev_tensors, to_np
from workloads import all_patterns, get, make_data, make_patterns, make_R

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2405_19509_gb300 as m
    yield m
    m.gc_set_decode_policy(m.GC_DECODE_AUTO)


def _policies(gc):
    return {"auto": gc.GC_DECODE_AUTO, "dense": gc.GC_DECODE_DENSE, "residual": gc.GC_DECODE_RESIDUAL}


def _decode(gc, policy, *args, **kw):
    gc.gc_set_decode_policy(policy)
    try:
        res = gc.gc_decode_batch(*args, **kw)
        torch.cuda.synchronize()
    finally:
        gc.gc_set_decode_policy(gc.GC_DECODE_AUTO)
    return res


def _copies(order, psi, N):
    """Delta per (pattern, chunk) for an order given as m x delta."""
    m, delta = order.shape
    D = np.zeros((psi.shape[0], N), dtype=np.int64)
    for j in range(m):
        for p in range(delta):
            i = order[j, p]
            if i >= 0:
                D[:, i] += psi[:, j] > p
    return D


def _residual_rows(nnz, ell, ksp):
    """Rows the residual policy leaves off the GEMM: a 128-row tile stays on
    the residual path unless a pattern overlapping it has more than `ksp`
    non-identity blocks or more than 32 of its rows need corrections."""
    npat = nnz.shape[0]
    M = npat * ell
    row_pat = np.arange(M) // ell
    res = np.zeros(M, dtype=bool)
    for t0 in range(0, M, 128):
        rows = np.arange(t0, min(M, t0 + 128))
        pats = np.unique(row_pat[rows])
        corrected = int((nnz[row_pat[rows]] > 0).sum())
        res[rows] = not (np.any(nnz[pats] > ksp) or corrected > 32)
    return res


def _tiny_G():
    cfg = get("tiny")
    data = make_data(cfg)
    G64 = O.chunk_gradients(data["X"].numpy(), data["y"].numpy(), data["w"].numpy(), cfg.N, cfg.n_c,
                            O.LSQ)
    return G64.astype(np.float32)


@pytest.mark.parametrize("ell", [1, 2, 3])
def test_policies_every_tiny_pattern(gc, ell):
    """All 4,096 patterns of the 6-worker workload plus 256 seeded ones under
    each policy: decoded gradients and errors against the oracle (tiles with
    more than 32 corrected rows stay on the GEMM under every policy)."""
    cfg = get("tiny")
    N, m, delta, d = cfg.N, cfg.m, cfg.delta, cfg.d
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    psi = np.concatenate([all_patterns(m, delta), make_patterns(cfg)])
    G32 = _tiny_G()
    Gref = G32.astype(np.float64)
    gsum = Gref.sum(axis=0)
    floor = 1e-8 * float(gsum @ gsum) / d
    Rd, od, pd = dev_tensors(R, order, psi)
    Gd = torch.from_numpy(G32).cuda()
    out = {k: _decode(gc, v, Rd, ell, od, N, m, delta, pd, Gd) for k, v in _policies(gc).items()}
    Gh = {k: to_np(v["Ghat"]) for k, v in out.items()}
    ms = {k: to_np(v["grad_mse"]) for k, v in out.items()}
    for b in range(psi.shape[0]):
        r = O.run_pattern(R, order, psi[b], N, Gref, want_transmit=False)
        for k in Gh:
            assert_grad_close(Gh[k][b], r.ghat, f"{k} b={b}")
            assert_mse_close(ms[k][b], r.grad_mse, floor, f"{k} mse b={b}")


@pytest.mark.parametrize("ell", [2, 3])
def test_mixed_and_straddling_tiles(gc, ell):
    """Runs of 64 exact patterns (all workers finished) alternate with runs of
    uniformly random ones, so the automatic policy sends some tiles to each
    path; with ell = 3 patterns straddle tile boundaries."""
    cfg = get("tiny")
    N, m, delta, d = cfg.N, cfg.m, cfg.delta, cfg.d
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    rnd = make_patterns(cfg, npat=512, stream=7)
    runs = []
    for r in range(8):
        runs.append(np.full((64, m), delta, dtype=np.int32) if r % 2 == 0 else rnd[64 * r:64 * r + 64])
    psi = np.concatenate(runs + [rnd[:5]])   # a ragged last tile
    G32 = _tiny_G()
    Gref = G32.astype(np.float64)
    gsum = Gref.sum(axis=0)
    floor = 1e-8 * float(gsum @ gsum) / d
    Rd, od, pd = dev_tensors(R, order, psi)
    res = _decode(gc, gc.GC_DECODE_AUTO, Rd, ell, od, N, m, delta, pd, torch.from_numpy(G32).cuda())
    dense = _decode(gc, gc.GC_DECODE_DENSE, Rd, ell, od, N, m, delta, pd, torch.from_numpy(G32).cuda())
    Gh, ms = to_np(res["Ghat"]), to_np(res["grad_mse"])
    if ell == 2:
        # a run of 64 exact patterns is one whole tile: residual path, ghat = sum_i g, zero error
        for r0 in (0, 128, 256, 384):
            assert np.all(ms[r0:r0 + 64] == 0.0)
            assert np.array_equal(Gh[r0], Gh[r0 + 63])
    for b in range(psi.shape[0]):
        r = O.run_pattern(R, order, psi[b], N, Gref, want_transmit=False)
        assert_grad_close(Gh[b], r.ghat, f"auto b={b}")
        assert_mse_close(ms[b], r.grad_mse, floor, f"auto mse b={b}")
    assert np.max(np.abs(Gh - to_np(dense["Ghat"]))) <= 1e-5 * np.max(np.abs(Gh))


def test_list_overflow_goes_to_the_gemm(gc):
    """m = N = 64, delta = 8, l = 2 with Binomial(8, 0.3) patterns: nearly every
    pattern needs corrections, more rows than a residual tile holds (32), so
    even the residual policy must decode those tiles on the GEMM; sampled
    patterns, the heaviest included, against the oracle."""
    cfg = get("mse_sweep")
    N, m, delta, ell, d = cfg.N, cfg.m, cfg.delta, 2, 2048
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    psi = make_patterns(cfg, npat=384, p=0.3)
    nnz = (_copies(order, psi, N) < ell).sum(axis=1)
    assert nnz.max() > 16
    rng = np.random.default_rng(3)
    G32 = rng.standard_normal((N, d)).astype(np.float32)
    Gref = G32.astype(np.float64)
    gsum = Gref.sum(axis=0)
    floor = 1e-8 * float(gsum @ gsum) / d
    Rd, od, pd = dev_tensors(R, order, psi)
    Gd = torch.from_numpy(G32).cuda()
    outs = [_decode(gc, v, Rd, ell, od, N, m, delta, pd, Gd) for v in _policies(gc).values()]
    picks = sorted(set([int(np.argmax(nnz)), int(np.argmin(nnz))] + list(range(0, 384, 29))))
    for b in picks:
        r = O.run_pattern(R, order, psi[b], N, Gref, want_transmit=False)
        for res in outs:
            assert_grad_close(to_np(res["Ghat"][b]), r.ghat, f"b={b} nnz={nnz[b]}")
            assert_mse_close(float(res["grad_mse"][b]), r.grad_mse, floor, f"b={b}")


def _sparse_stragglers(rng, npat, m, delta, every):
    """Every worker finished, except in every `every`-th pattern (offset 1),
    whose counts are uniform in 0..delta: residual tiles with corrected rows."""
    psi = np.full((npat, m), delta, dtype=np.int32)
    idx = np.arange(1, npat, every)
    psi[idx] = rng.integers(0, delta + 1, size=(idx.size, m))
    return psi


@pytest.mark.parametrize("ell", [1, 2, 3])
def test_sparse_stragglers_tiny(gc, ell):
    """4096 patterns of the 6-worker workload, one in five with stragglers:
    the residual tiles now hold corrected rows (the list and slot machinery);
    every pattern against the oracle under each policy."""
    cfg = get("tiny")
    N, m, delta, d = cfg.N, cfg.m, cfg.delta, cfg.d
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    psi = _sparse_stragglers(np.random.default_rng(40 + ell), 4096, m, delta, 5)
    G32 = _tiny_G()
    Gref = G32.astype(np.float64)
    gsum = Gref.sum(axis=0)
    floor = 1e-8 * float(gsum @ gsum) / d
    Rd, od, pd = dev_tensors(R, order, psi)
    Gd = torch.from_numpy(G32).cuda()
    out = {k: _decode(gc, v, Rd, ell, od, N, m, delta, pd, Gd) for k, v in _policies(gc).items()}
    nnz = (_copies(order, psi, N) < ell).sum(axis=1)
    res_rows = _residual_rows(nnz, ell, N).reshape(-1, ell).all(axis=1)
    assert res_rows.mean() > 0.5, "most tiles should stay on the residual path"
    exact_res = (nnz == 0) & res_rows
    assert np.all(to_np(out["residual"]["grad_mse"])[exact_res] == 0.0)
    cache = {}
    for b in range(psi.shape[0]):
        key = psi[b].tobytes()
        if key not in cache:
            cache[key] = O.run_pattern(R, order, psi[b], N, Gref, want_transmit=False)
        r = cache[key]
        for k, res in out.items():
            assert_grad_close(to_np(res["Ghat"][b]), r.ghat, f"{k} b={b}")
            assert_mse_close(float(res["grad_mse"][b]), r.grad_mse, floor, f"{k} mse b={b}")


@pytest.mark.parametrize("d,ell,npat", [(67, 2, 1), (5, 4, 3), (64, 3, 129), (1, 1, 130), (1030, 2, 200)])
def test_ragged_shapes_both_paths(gc, d, ell, npat):
    """Block lengths that are not multiples of 4 (scalar loads and stores),
    zero padding past d, a single pattern, a last tile of one row."""
    N = m = 6
    delta = 3
    order = O.cyclic_order(N, m, delta)
    rng = np.random.default_rng(d * 100 + ell)
    R = rng.standard_normal((ell, m))
    psi = _sparse_stragglers(rng, npat, m, delta, 3)
    if npat == 1:
        psi[0] = rng.integers(0, delta + 1, size=m)
    G32 = rng.standard_normal((N, d)).astype(np.float32)
    Gref = G32.astype(np.float64)
    gsum = Gref.sum(axis=0)
    floor = 1e-8 * float(gsum @ gsum) / d
    Rd, od, pd = dev_tensors(R, order, psi)
    Gd = torch.from_numpy(G32).cuda()
    for pol in (gc.GC_DECODE_DENSE, gc.GC_DECODE_RESIDUAL):
        res = _decode(gc, pol, Rd, ell, od, N, m, delta, pd, Gd)
        for b in range(npat):
            r = O.run_pattern(R, order, psi[b], N, Gref, want_transmit=False)
            assert_grad_close(to_np(res["Ghat"][b]), r.ghat, f"policy {pol} b={b}")
            assert_mse_close(float(res["grad_mse"][b]), r.grad_mse, floor, f"policy {pol} b={b}")


def test_combine_non_projector_matrix(gc):
    """gc_decode_combine with a decode matrix whose blocks, in one pattern in
    four, are near but not exactly I (every block of such a pattern differs
    from I): both paths against the plain product C . G in fp64 and against
    each other; MSE-only as well, and errors only under the automatic policy,
    which forms each MSE as a quadratic form in the Gram matrix of the chunk
    blocks."""
    N, ell, npat, d = 6, 2, 300, 1024
    rng = np.random.default_rng(17)
    C = np.tile(np.kron(np.ones((1, N)), np.eye(ell)), (npat, 1, 1))
    # perturbations far from rounding (the GEMM forms ghat - s by difference;
    # the decode blocks of the method are projectors, Pi - I either 0 or O(1))
    C += 0.05 * rng.standard_normal(C.shape)
    keep = np.arange(npat) % 4 != 1
    C[keep] = np.kron(np.ones((1, N)), np.eye(ell))  # three patterns in four exact
    C = C.astype(np.float32)
    G32 = rng.standard_normal((N, d)).astype(np.float32)
    L = d // ell
    Gv = G32.astype(np.float64).reshape(N, ell, L).reshape(N * ell, L)
    ref = np.einsum("bkj,jc->bkc", C.astype(np.float64), Gv).reshape(npat, d)
    gsum = G32.astype(np.float64).sum(axis=0)
    mref = ((ref - gsum) ** 2).sum(axis=1) / d
    floor = 1e-8 * float(gsum @ gsum) / d
    Cd, Gd = torch.from_numpy(C).cuda(), torch.from_numpy(G32).cuda()
    got = {}
    for name, pol in (("dense", gc.GC_DECODE_DENSE), ("residual", gc.GC_DECODE_RESIDUAL)):
        gc.gc_set_decode_policy(pol)
        try:
            res = gc.gc_decode_combine(Cd, ell, N, Gd)
            mo = gc.gc_decode_combine(Cd, ell, N, Gd, Ghat=False)["grad_mse"]
            torch.cuda.synchronize()
        finally:
            gc.gc_set_decode_policy(gc.GC_DECODE_AUTO)
        got[name] = to_np(res["Ghat"])
        for b in range(npat):
            assert_grad_close(got[name][b], ref[b], f"{name} b={b}")
            assert_mse_close(float(res["grad_mse"][b]), mref[b], floor, f"{name} mse b={b}")
            assert_mse_close(float(mo[b]), mref[b], floor, f"{name} mse-only b={b}")
    assert np.max(np.abs(got["dense"] - got["residual"])) <= 1e-5 * np.max(np.abs(ref))
    # errors only under the automatic policy: the quadratic forms in the Gram
    # matrix of the chunk blocks (exact patterns give 0 exactly)
    mg = to_np(gc.gc_decode_combine(Cd, ell, N, Gd, Ghat=False)["grad_mse"])
    for b in range(npat):
        assert_mse_close(float(mg[b]), mref[b], floor, f"gram mse-only b={b}")
    assert np.all(mg[keep] == 0.0)


@pytest.mark.parametrize("ell", [5, 8])
def test_large_ell_both_paths(gc, ell):
    """The widest communication factors of the build: N = m = 10 chunks and
    workers, delta = 8, l = 5 and 8 (at l = 8 exact recovery needs every copy;
    lists hold 8 blocks, so longer ones send their tiles to the GEMM), d not a
    multiple of l.  Mostly exact patterns, mild stragglers and a few uniform
    ones; every pattern against the oracle under each policy."""
    N = m = 10
    delta, d, npat = 8, 1003, 300
    order = O.cyclic_order(N, m, delta)
    rng = np.random.default_rng(70 + ell)
    R = rng.standard_normal((ell, m))
    # exact patterns; mild stragglers (a few consecutive workers stop up to 6
    # chunks early: a few blocks below l copies); every 12th pattern uniform
    psi = np.full((npat, m), delta, dtype=np.int32)
    every = 3 if ell == 5 else 8   # a 128-row tile holds 25 patterns at l = 5, 16 at l = 8
    for b in range(npat):
        if b % (4 * every) == 5:
            psi[b] = rng.integers(0, delta + 1, size=m)
        elif b % every == 1:
            j0 = rng.integers(0, m)
            for t in range(int(rng.integers(1, 4))):
                psi[b, (j0 + t) % m] = delta - int(rng.integers(1, 7))
    G32 = rng.standard_normal((N, d)).astype(np.float32)
    Gref = G32.astype(np.float64)
    gsum = Gref.sum(axis=0)
    floor = 1e-8 * float(gsum @ gsum) / d
    Rd, od, pd = dev_tensors(R, order, psi)
    Gd = torch.from_numpy(G32).cuda()
    out = {k: _decode(gc, v, Rd, ell, od, N, m, delta, pd, Gd) for k, v in _policies(gc).items()}
    nnz = (_copies(order, psi, N) < ell).sum(axis=1)
    assert (nnz == 0).any() and (nnz > 8).any()
    res_rows = _residual_rows(nnz, ell, 8)
    assert res_rows.mean() > 0.3 and (np.repeat(nnz, ell)[res_rows] > 0).any()
    cache = {}
    for b in range(npat):
        key = psi[b].tobytes()
        if key not in cache:
            cache[key] = O.run_pattern(R, order, psi[b], N, Gref, want_transmit=False)
        r = cache[key]
        for k, res in out.items():
            assert_grad_close(to_np(res["Ghat"][b]), r.ghat, f"{k} l={ell} b={b}")
            assert_mse_close(float(res["grad_mse"][b]), r.grad_mse, floor, f"{k} l={ell} mse b={b}")


@pytest.mark.parametrize("N,delta,ell,d", [(10, 4, 3, 1001), (20, 8, 8, 997), (40, 6, 5, 1500)])
def test_errors_only_gram_path(gc, N, delta, ell, d):
    """Errors only under the automatic policy (npat * ell >= 2 N ell): each
    pattern's gradient MSE as a quadratic form in the Gram matrix of the chunk
    blocks, with a padded last block (l does not divide d), H in shared memory
    (N l <= 128) or read through the cache (N l = 160, 200); against the
    oracle's decoded gradients, against the residual/GEMM decode of the same
    batch, and exactly 0 for exact patterns."""
    m = N
    rng = np.random.default_rng(50 + N + ell)
    order = O.cyclic_order(N, m, delta)
    R = rng.standard_normal((ell, m))
    npat = 2 * N + 7
    psi = rng.integers(0, delta + 1, size=(npat, m)).astype(np.int32)
    psi[0] = delta                      # every worker done: exact
    psi[1] = 0                          # none started
    G = rng.standard_normal((N, d)).astype(np.float32)
    Gref = G.astype(np.float64)
    gsum = Gref.sum(axis=0)
    floor = 1e-8 * float(gsum @ gsum) / d
    Rd, od, pd = dev_tensors(R, order, psi)
    Gd = torch.from_numpy(G).cuda()
    res = gc.gc_mse(Rd, ell, od, N, m, delta, pd, Gd)               # the Gram path
    full = gc.gc_decode_batch(Rd, ell, od, N, m, delta, pd, Gd)     # decoded gradients and MSE
    torch.cuda.synchronize()
    mg, mf = to_np(res["grad_mse"]), to_np(full["grad_mse"])
    assert mg[0] == 0.0
    for b in range(npat):
        r = O.run_pattern(R, order, psi[b], N, Gref, want_transmit=False)
        assert_mse_close(float(mg[b]), r.grad_mse, floor, f"gram b={b}")
        assert_mse_close(float(mg[b]), float(mf[b]), floor, f"gram vs decode b={b}")

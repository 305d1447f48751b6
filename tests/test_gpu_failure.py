"""Failure path without a GPU fault.  A loader is made to withhold its copy
(gc_inject_stall), so its consumers wait on a barrier that nothing completes;
with a short wait limit (gc_set_wait_limit) the wait expires, the kernel
records GC_ERR_TIMEOUT in the workspace status and returns, and the next call
on the same context is correct again."""
import numpy as np
import pytest
import torch

import oracle as O
from _parity import assert_grad_close, to_np

pytestmark = pytest.mark.gpu

SHORT = 1 << 22  # clock cycles, about 2 ms


@pytest.fixture(scope="module")
def gc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2405_19509_gb300 as m
    return m


def _expect_timeout(gc, ws):
    with pytest.raises(gc.GCError) as ei:
        gc.gc_status(ws)
    assert ei.value.code == -5 and "wait" in str(ei.value)


def test_chunk_grads_stall_times_out_then_recovers(gc):
    N, n_c, d = 20, 512, 4096
    g = torch.Generator().manual_seed(5)
    X = torch.randn(N * n_c, d, generator=g) / d ** 0.5
    y = torch.randn(N * n_c, generator=g)
    w = torch.randn(d, generator=g) / d ** 0.5
    Xd, yd, wd = X.cuda(), y.cuda(), w.cuda()
    ws = gc.Workspace()
    gc.gc_set_wait_limit(SHORT)
    try:
        gc.gc_inject_stall(gc.GC_STALL_CHUNK_GRADS)
        gc.gc_chunk_grads(Xd, yd, wd, N, n_c, gc.GC_LSQ, ws=ws)
        torch.cuda.synchronize()
        _expect_timeout(gc, ws)
    finally:
        gc.gc_inject_stall(0)
        gc.gc_set_wait_limit(0)
    # the status was cleared by the read; the context is usable and results right
    G = gc.gc_chunk_grads(Xd, yd, wd, N, n_c, gc.GC_LSQ, ws=ws)
    gc.gc_status(ws)
    Go = O.chunk_gradients(X.numpy(), y.numpy(), w.numpy(), N, n_c, O.LSQ)
    for i in range(N):
        assert_grad_close(to_np(G[i]), Go[i], f"chunk {i} after recovery")


def test_combine_stall_times_out_then_recovers(gc):
    from workloads import get, make_R, make_patterns

    cfg = get("tiny")
    N, m, delta, ell = cfg.N, cfg.m, cfg.delta, 2
    L = 1024
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    psi = make_patterns(cfg, npat=300)
    rng = np.random.default_rng(11)
    G = rng.standard_normal((N, ell * L)).astype(np.float32)
    dev = torch.device("cuda")
    Rd, od = torch.from_numpy(R).to(dev), torch.from_numpy(order).to(dev)
    pd, Gd = torch.from_numpy(psi).to(dev), torch.from_numpy(G).to(dev)
    ws = gc.Workspace()
    gc.gc_set_wait_limit(SHORT)
    # every row tile on the tensor-core GEMM, so the withheld copy is waited on
    gc.gc_set_decode_policy(gc.GC_DECODE_DENSE)
    try:
        gc.gc_inject_stall(gc.GC_STALL_COMBINE)
        gc.gc_decode_batch(Rd, ell, od, N, m, delta, pd, Gd, ws=ws)
        torch.cuda.synchronize()
        _expect_timeout(gc, ws)
    finally:
        gc.gc_inject_stall(0)
        gc.gc_set_wait_limit(0)
        gc.gc_set_decode_policy(gc.GC_DECODE_AUTO)
    res = gc.gc_decode_batch(Rd, ell, od, N, m, delta, pd, Gd, ws=ws)
    gc.gc_status(ws)
    Gh = to_np(res["Ghat"])
    for b in range(0, psi.shape[0], 7):
        ref = O.run_pattern(R, order, psi[b], N, G.astype(np.float64)).ghat
        assert_grad_close(Gh[b], ref, f"pattern {b} after recovery")


def test_stall_bit_is_consumed(gc):
    """An armed stall affects one launch only: the following call is clean."""
    N, n_c, d = 4, 64, 256
    X = torch.randn(N * n_c, d, device="cuda")
    y = torch.randn(N * n_c, device="cuda")
    w = torch.randn(d, device="cuda")
    ws = gc.Workspace()
    gc.gc_set_wait_limit(SHORT)
    try:
        gc.gc_inject_stall(gc.GC_STALL_CHUNK_GRADS)
        gc.gc_chunk_grads(X, y, w, N, n_c, gc.GC_LSQ, ws=ws)
        _expect_timeout(gc, ws)
        gc.gc_chunk_grads(X, y, w, N, n_c, gc.GC_LSQ, ws=ws)
        gc.gc_status(ws)
    finally:
        gc.gc_inject_stall(0)
        gc.gc_set_wait_limit(0)


def test_batched_gemm_stall_times_out_then_recovers(gc):
    N, n_c, d, n_w = 4, 128, 256, 32
    g = torch.Generator().manual_seed(9)
    X = (torch.randn(N * n_c, d, generator=g) / d ** 0.5).to(torch.bfloat16)
    y = torch.randn(N * n_c, generator=g)
    W = torch.randn(n_w, d, generator=g)
    Xd, yd, Wd = X.cuda(), y.cuda(), W.cuda()
    ws = gc.Workspace()
    gc.gc_set_wait_limit(SHORT)
    try:
        gc.gc_inject_stall(gc.GC_STALL_BATCHED)
        gc.gc_chunk_grads_batched(Xd, yd, Wd, N, n_c, O.LSQ, ws=ws)
        torch.cuda.synchronize()
        _expect_timeout(gc, ws)
    finally:
        gc.gc_inject_stall(0)
        gc.gc_set_wait_limit(0)
    G = gc.gc_chunk_grads_batched(Xd, yd, Wd, N, n_c, O.LSQ, ws=ws)
    gc.gc_status(ws)
    Xf = X.float().numpy().astype(np.float64)
    for w in (0, 31):
        ref = O.chunk_gradients(Xf, y.numpy(), W[w].numpy(), N, n_c, O.LSQ)
        for i in range(N):
            assert_grad_close(to_np(G[w, i]), ref[i], f"w {w} chunk {i} after recovery")

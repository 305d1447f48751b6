"""The allocation-free variant of Algorithm 1 (gc_find_encoding_coeff_noalloc).

It exists for callers that cannot allocate device memory (a runtime that
reserves its memory once at start-up and forbids later cudaMalloc, an
embedding without a CUDA allocator): its scratch is a fixed array inside the
library instead of a caller workspace.  This test calls it through the C-ABI
twice in a row -- a large batch that uses the memo table, then a small one
solved directly, so the second call runs on scratch the first one left
behind -- and checks both against gc_find_encoding_coeff with a workspace.
This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle as O
from _parity import COEF_RTOL, dev_tensors, rel_inf, to_np
from workloads import get, make_patterns, make_R

pytestmark = pytest.mark.gpu


def _noalloc(gc, Rd, ell, od, N, m, delta, pd):
    npat = pd.shape[0]
    dev = pd.device
    E = torch.empty(npat, m, delta, ell, dtype=torch.float64, device=dev)
    C = torch.empty(npat, ell, N * ell, dtype=torch.float32, device=dev)
    D = torch.empty(npat, N, dtype=torch.uint8, device=dev)
    ce = torch.empty(npat, dtype=torch.float64, device=dev)
    es = torch.empty(npat, dtype=torch.float64, device=dev)
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    rc = gc.lib.gc_find_encoding_coeff_noalloc(
        p(Rd), ell, p(od), N, m, delta, p(pd), npat, p(E), p(C), p(D), None, p(ce), p(es),
        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == 0, gc.gc_last_error()
    return {"E": E, "C": C, "delta": D, "coef_err": ce, "est": es}


def test_noalloc_matches_workspace_variant_twice():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2405_19509_gb300 as gc

    cfg = get("logistic")
    N, m, delta, ell = cfg.N, cfg.m, cfg.delta, 2
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    big = make_patterns(cfg, npat=4000, stream=901)      # memo-table path
    small = make_patterns(cfg, npat=3, stream=902)       # direct path
    for psi in (big, small):
        Rd, od, pd = dev_tensors(R, order, psi)
        got = _noalloc(gc, Rd, ell, od, N, m, delta, pd)
        ref = gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, pd)
        torch.cuda.synchronize()
        assert torch.equal(got["delta"], ref["delta"])
        assert torch.equal(got["est"], ref["est"])
        for b in range(psi.shape[0]):
            assert rel_inf(to_np(got["E"][b]), to_np(ref["E"][b])) <= COEF_RTOL
        assert torch.max(torch.abs(got["C"] - ref["C"])).item() <= 2e-6
        assert torch.max(torch.abs(got["coef_err"] - ref["coef_err"])).item() <= 1e-9
    # and the second call against the oracle directly, pattern by pattern
    for b in range(small.shape[0]):
        r = O.run_pattern(R, order, small[b], N)
        assert rel_inf(to_np(got["E"][b]), r.E) <= COEF_RTOL
        assert np.array_equal(to_np(got["delta"][b]), r.Delta)


def test_noalloc_rejects_oversized_scratch():
    """A shape whose holder table alone exceeds the static scratch is
    rejected on the host, with a message naming the limit."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2405_19509_gb300 as gc
    N, m, delta, ell = 100_000, 1, 1, 1          # ~100 bytes of holder table per chunk
    order = np.zeros((m, delta), dtype=np.int32)
    R = np.ones((ell, m))
    psi = np.zeros((1, m), dtype=np.int32)
    Rd, od, pd = dev_tensors(R, order, psi)
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    rc = gc.lib.gc_find_encoding_coeff_noalloc(p(Rd), ell, p(od), N, m, delta, p(pd), 1, None, None,
                                               None, None, None, None, None)
    assert rc == -6
    assert "static scratch" in gc.gc_last_error()

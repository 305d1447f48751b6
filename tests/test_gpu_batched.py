"""Chunk gradients for several parameter vectors on the tensor cores
(gc_chunk_grads_batched) against the fp64 oracle, one w at a time, on the
same bf16 features (Sec. I: g_{D_i} = X_i^T (f(X_i w) - y01_i))."""
import numpy as np
import pytest
import torch

import oracle as O
from _parity import assert_grad_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2405_19509_gb300 as m
    return m


def _case(N, n_c, d, n_w, loss, seed):
    g = torch.Generator().manual_seed(seed)
    X = (torch.randn(N * n_c, d, generator=g) / d ** 0.5).to(torch.bfloat16)
    if loss == O.LSQ:
        y = torch.randn(N * n_c, generator=g)
    else:
        y = torch.where(torch.rand(N * n_c, generator=g) < 0.5, -1.0, 1.0)
    W = torch.randn(n_w, d, generator=g)
    return X, y, W


@pytest.mark.parametrize("N,n_c,d,n_w,loss", [
    (4, 128, 256, 32, 0), (4, 128, 256, 32, 1),
    (2, 192, 384, 64, 1),
    (8, 256, 1024, 128, 0),
    (2, 128, 512, 256, 1),
    (16, 512, 2048, 96, 1),
])
def test_batched_chunk_grads_match_oracle(gc, N, n_c, d, n_w, loss):
    X, y, W = _case(N, n_c, d, n_w, loss, 100 + n_w + d)
    ws = gc.Workspace()
    G = gc.gc_chunk_grads_batched(X.cuda(), y.cuda(), W.cuda(), N, n_c, loss, ws=ws)
    gc.gc_status(ws)
    Xf = X.float().numpy().astype(np.float64)
    Gn = G.cpu().numpy()
    yn = y.numpy()
    for w in range(n_w):
        ref = O.chunk_gradients(Xf, yn, W[w].numpy(), N, n_c, loss)
        for i in range(N):
            assert_grad_close(Gn[w, i], ref[i], f"w {w} chunk {i}")


def test_batched_matches_single_w_path(gc):
    """Column w of the batched result equals gc_chunk_grads at w (bf16 X)."""
    N, n_c, d, n_w = 8, 256, 1024, 64
    X, y, W = _case(N, n_c, d, n_w, 1, 7)
    Xd, yd, Wd = X.cuda(), y.cuda(), W.cuda()
    G = gc.gc_chunk_grads_batched(Xd, yd, Wd, N, n_c, 1)
    for w in (0, 17, 63):
        Gs = gc.gc_chunk_grads(Xd, yd, Wd[w].contiguous(), N, n_c, 1)
        a, b = G[w].cpu().numpy(), Gs.cpu().numpy()
        assert np.max(np.abs(a - b)) <= 2e-4 * np.max(np.abs(b))


def test_batched_status_and_shapes(gc):
    ws = gc.Workspace()
    X, y, W = _case(2, 128, 256, 32, 0, 3)
    gc.gc_chunk_grads_batched(X.cuda(), y.cuda(), W.cuda(), 2, 128, 0, ws=ws)
    gc.gc_status(ws)
    # d = 200 is not a multiple of 128: rejected before any launch
    X2 = X[:, :200].contiguous().cuda()
    with pytest.raises(gc.GCError) as e:
        gc.gc_chunk_grads_batched(X2, y.cuda(), W[:, :200].contiguous().cuda(), 2, 128, 0)
    assert e.value.code == -3

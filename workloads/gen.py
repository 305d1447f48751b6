"""Seeded generators for the synthetic workloads (data only, no protocol math).

Every generator is keyed by (config seed, purpose tag, index) so that any
chunk of X can be regenerated on its own.  Small workloads are generated on
the CPU; the multi-GB feature matrices can be generated chunk by chunk on a
CUDA device with torch's seeded device generator (the same call, so the same
bits, every time it runs on a given torch build).
"""
from __future__ import annotations

import itertools
import math

import numpy as np
import torch

from .configs import Config

(_TAG_R, _TAG_WSTAR, _TAG_W, _TAG_X, _TAG_NOISE, _TAG_LABEL, _TAG_PSI, _TAG_G, _TAG_GRAPH,
 _TAG_ORDER, _TAG_TIMES) = range(11)


def _np_rng(*key: int) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([int(k) for k in key]))


def _torch_seed(*key: int) -> int:
    s = 0x9E3779B97F4A7C15
    for k in key:
        s = (s * 0x100000001B3 + int(k) + 1) & 0x7FFFFFFFFFFFFFFF
    return s


def make_R(cfg: Config, ell: int) -> np.ndarray:
    """The PS's ell x m matrix with i.i.d. N(0,1) entries (Sec. II), fp64."""
    return _np_rng(cfg.seed, _TAG_R, ell).standard_normal((ell, cfg.m))


def make_w(cfg: Config, which: str = "eval") -> np.ndarray:
    """Parameter vectors (fp32 values, returned as float32 numpy):
    which="star": the generating w*; which="eval": the point where chunk
    gradients are evaluated (random, so that X w matters); which="zero"."""
    d = cfg.d
    if which == "zero":
        return np.zeros(d, dtype=np.float32)
    tag = _TAG_WSTAR if which == "star" else _TAG_W
    v = _np_rng(cfg.seed, tag).standard_normal(d)
    if cfg.loss == "lsq" or which == "eval":
        v = v / math.sqrt(d)
    return v.astype(np.float32)


def _x_scale(cfg: Config) -> float:
    return 1.0 / math.sqrt(cfg.d) if cfg.loss == "logistic" else 1.0


def _torch_dtype(cfg: Config):
    return torch.bfloat16 if cfg.x_dtype == "bf16" else torch.float32


def make_X_chunk(cfg: Config, i: int, device="cpu") -> torch.Tensor:
    """Rows [i*n_c, (i+1)*n_c) of X, generated from their own seed."""
    dev = torch.device(device)
    g = torch.Generator(device=dev).manual_seed(_torch_seed(cfg.seed, _TAG_X, i))
    x = torch.randn(cfg.n_c, cfg.d, generator=g, device=dev, dtype=torch.float32)
    if cfg.loss == "logistic":
        x.mul_(_x_scale(cfg))
    return x.to(_torch_dtype(cfg))


def make_data(cfg: Config, device="cpu", w_which: str = "eval") -> dict:
    """X (N*n_c x d, fp32 or bf16), y (fp32; +-1 for logistic), w (fp32),
    w_star, all as torch tensors on `device`.  Labels:
      least squares: y = X w* + 0.1 * N(0,1), w* ~ N(0,1)/sqrt(d)
      logistic:      y = +1 with probability sigmoid(x^T w*), else -1, w* ~ N(0,1)
    """
    dev = torch.device(device)
    Ntil = cfg.Ntil
    X = torch.empty(Ntil, cfg.d, dtype=_torch_dtype(cfg), device=dev)
    for i in range(cfg.N):
        X[i * cfg.n_c:(i + 1) * cfg.n_c] = make_X_chunk(cfg, i, dev)
    w_star = torch.from_numpy(make_w(cfg, "star")).to(dev)
    z = torch.empty(Ntil, dtype=torch.float32, device=dev)
    for i in range(cfg.N):
        rows = slice(i * cfg.n_c, (i + 1) * cfg.n_c)
        z[rows] = X[rows].float() @ w_star
    gy = torch.Generator(device=dev).manual_seed(_torch_seed(cfg.seed, _TAG_LABEL))
    if cfg.loss == "lsq":
        noise = torch.randn(Ntil, generator=gy, device=dev, dtype=torch.float32)
        y = z + 0.1 * noise
    else:
        u = torch.rand(Ntil, generator=gy, device=dev, dtype=torch.float32)
        y = torch.where(u < torch.sigmoid(z), 1.0, -1.0).to(torch.float32)
    w = torch.from_numpy(make_w(cfg, w_which)).to(dev)
    return {"X": X, "y": y.contiguous(), "w": w, "w_star": w_star}


def make_chunk_grads(cfg: Config, device="cpu") -> torch.Tensor:
    """Given chunk gradients for the decode-only workload: N x d fp32 ~ N(0,1)."""
    dev = torch.device(device)
    G = torch.empty(cfg.N, cfg.d, dtype=torch.float32, device=dev)
    for i in range(cfg.N):
        g = torch.Generator(device=dev).manual_seed(_torch_seed(cfg.seed, _TAG_G, i))
        G[i] = torch.randn(cfg.d, generator=g, device=dev, dtype=torch.float32)
    return G


def make_patterns(cfg: Config, npat: int | None = None, p: float | None = None,
                  stream: int = 0) -> np.ndarray:
    """npat x m int32 state vectors psi under the workload's straggler model.
    `stream` separates independent batches (e.g. SGD iterations)."""
    npat = cfg.npat if npat is None else npat
    m, delta = cfg.m, cfg.delta
    key_p = 0 if p is None else int(round(p * 1000))
    rng = _np_rng(cfg.seed, _TAG_PSI, key_p, stream)
    model = cfg.pattern_model
    if model == "uniform":
        psi = rng.integers(0, delta + 1, size=(npat, m))
    elif model == "shifted_exp":
        tau = 1.0 + rng.exponential(1.0, size=(npat, m))
        T = 0.5 * delta * tau.max(axis=1, keepdims=True)
        psi = np.minimum(delta, np.floor(T / tau)).astype(np.int64)
    elif model == "binomial":
        if p is None:
            raise ValueError("binomial straggler model needs p")
        psi = rng.binomial(delta, p, size=(npat, m))
    elif model == "frac_binom":
        f = rng.uniform(0.2, 1.0, size=(npat, 1))
        psi = rng.binomial(delta, np.broadcast_to(f, (npat, m)))
    else:
        raise ValueError(model)
    return np.ascontiguousarray(psi, dtype=np.int32)


def all_patterns(m: int, delta: int) -> np.ndarray:
    """Every psi in {0..delta}^m, in lexicographic order (brute force)."""
    return np.array(list(itertools.product(range(delta + 1), repeat=m)), dtype=np.int32)


def random_regular_graph(m: int, nu: int, seed: int) -> np.ndarray:
    """Adjacency matrix (m x m uint8, symmetric, zero diagonal) of a random
    nu-regular simple graph: the pairing model with pairs drawn among the
    points that can still be joined (no loop, no repeated edge), restarted
    when it gets stuck (Steger and Wormald, 1999).  Used as the assignment
    matrix A of the approximate-GC workloads (Sec. IV: N = m, every row and
    column sum nu)."""
    assert (m * nu) % 2 == 0 and nu < m
    rng = _np_rng(seed, _TAG_GRAPH, m, nu)
    while True:
        A = np.zeros((m, m), dtype=np.uint8)
        pts = list(np.repeat(np.arange(m), nu))
        stuck = False
        while pts:
            n = len(pts)
            done = False
            for _ in range(64):
                a, b = rng.integers(0, n, size=2)
                u, v = pts[a], pts[b]
                if a != b and u != v and not A[u, v]:
                    done = True
                    break
            if not done:
                # exhaustive search for any suitable pair before giving up
                cand = [(a, b) for a in range(n) for b in range(a + 1, n)
                        if pts[a] != pts[b] and not A[pts[a], pts[b]]]
                if not cand:
                    stuck = True
                    break
                a, b = cand[rng.integers(0, len(cand))]
                u, v = pts[a], pts[b]
            A[u, v] = A[v, u] = 1
            for k in sorted((a, b), reverse=True):
                pts[k] = pts[-1]
                pts.pop()
        if not stuck:
            return A


def second_eigenvalue(A: np.ndarray) -> float:
    """Second-largest absolute eigenvalue of a symmetric adjacency matrix
    (a nu-regular graph is Ramanujan when it is below 2 sqrt(nu - 1))."""
    ev = np.sort(np.abs(np.linalg.eigvalsh(A.astype(np.float64))))
    return float(ev[-2])


def random_order(A: np.ndarray, seed: int, index: int = 0) -> np.ndarray:
    """A uniformly random processing order for assignment A: worker j takes
    its chunks {i : A_ij != 0} in a random permutation (m x delta int32,
    -1 padded).  Sec. IV compares the optimal ordering with the best of 100
    such orderings."""
    N, m = A.shape
    delta = int((A != 0).sum(axis=0).max())
    rng = _np_rng(seed, _TAG_ORDER, index)
    order = -np.ones((m, delta), dtype=np.int32)
    for j in range(m):
        ch = np.flatnonzero(A[:, j])
        order[j, :len(ch)] = rng.permutation(ch)
    return order


def make_worker_times(m: int, nsim: int, seed: int, alpha: int = 0, shift: float = 0.0):
    """Per-realization worker speeds for the completion-time simulation of
    Sec. IV: tau[r, j] = time W_j takes per chunk, i.i.d. shift + Exp(1); in
    every realization alpha workers chosen uniformly at random have failed
    (tau = +inf).  Returns float64 nsim x m."""
    rng = _np_rng(seed, _TAG_TIMES, m, alpha)
    tau = shift + rng.exponential(1.0, size=(nsim, m))
    for r in range(nsim):
        if alpha:
            tau[r, rng.choice(m, size=alpha, replace=False)] = np.inf
    return tau

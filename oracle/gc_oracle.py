"""Plain fp64 CPU oracle for the partial-straggler gradient-coding protocol.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import this module:
only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline /
``--impl reference`` leg use it.  It shares no code with the CUDA library.

Everything here is written from "Leveraging partial stragglers within gradient
coding" (Ramamoorthy, Meng, Girimaji, 2024) and follows its notation:

  N chunks D_1..D_N, m workers W_1..W_m (0-based in code), load delta,
  communication factor ell, parameter dimension d, block length L = ceil(d/ell),
  state vector psi (chunks processed per worker), R (ell x m, N(0,1)),
  encoding-coefficient matrix B (m x N*ell, block columns B^(i) of ell columns).

Layout conventions (the same ones the C-ABI documents, restated here, not
shared):
  * order[j, p]   chunk processed p-th by worker j (top to bottom), -1 = empty.
  * O[i, j]       position (1-based) of D_i inside W_j, 0 = not assigned (Sec. III).
  * X             (N*n_c) x d row-major; chunk i = rows [i*n_c, (i+1)*n_c).
  * G             N x d chunk gradients g_{D_i}.
  * blocks        g[k] = g[k*L : (k+1)*L], zero padded to length L (Sec. II).
  * T             m x L transmissions (eq. 2).
  * B             m x (N*ell); column i*ell + k belongs to g_{D_i}[k].

All arithmetic is float64.  Library primitives (lstsq, matmul) serve as single
steps; no blocking or fusion beyond what the paper states.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

LSQ = 0
LOGISTIC = 1


# --------------------------------------------------------------------------
# Assignment and ordering (Sec. I: assignment matrix A; Sec. III: ordering
# matrix O; the cyclic assignment of Tandon et al. that Sec. III and Sec. IV use)
# --------------------------------------------------------------------------
def cyclic_order(N: int, m: int, delta: int) -> np.ndarray:
    """Cyclic assignment (Sec. III, Sec. IV): W_j holds delta cyclically
    consecutive chunks D_j, D_{j+1}, ..., D_{j+delta-1} (mod N) and processes
    them top to bottom."""
    order = np.empty((m, delta), dtype=np.int32)
    for j in range(m):
        for p in range(delta):
            order[j, p] = (j + p) % N
    return order


def ordering_matrix(order: np.ndarray, N: int) -> tuple[np.ndarray, np.ndarray]:
    """Assignment matrix A (Sec. I: A_ij != 0 iff D_i is assigned to W_j) and
    ordering matrix O (Sec. III: O_ij = alpha if D_i is the alpha-th chunk of
    W_j, else 0), both N x m uint8."""
    m, delta = order.shape
    O = np.zeros((N, m), dtype=np.uint8)
    for j in range(m):
        for p in range(delta):
            i = int(order[j, p])
            if i >= 0:
                O[i, j] = p + 1
    A = (O > 0).astype(np.uint8)
    return A, O


def q_metric(O: np.ndarray, delta: int) -> np.ndarray:
    """Q_i(O) of Sec. III: the most chunks the cluster can process with no copy
    of D_i processed: sum_j 1{O_ij != 0}(O_ij - 1) + (m - delta) * delta."""
    N, m = O.shape
    Q = np.zeros(N, dtype=np.int64)
    for i in range(N):
        s = 0
        for j in range(m):
            if O[i, j] != 0:
                s += int(O[i, j]) - 1
        Q[i] = s + (m - delta) * delta
    return Q


def chunk_ordering(A: np.ndarray) -> np.ndarray:
    """Algorithm 2 (Sec. III): for an N == m assignment with every row and
    column sum delta, peel delta perfect matchings P_1..P_delta off the
    bipartite graph of A (each exists by Claim 1) and return the ordering
    matrix O = sum_p p * P_p (N x m uint8).  The matching step is a library
    maximum bipartite matching; which optimal O comes out depends on it."""
    from scipy.sparse import csr_matrix
    from scipy.sparse.csgraph import maximum_bipartite_matching

    At = (np.asarray(A) != 0).astype(np.int64)
    N, m = At.shape
    assert N == m, "Algorithm 2 needs N == m"
    delta = int(At[0].sum())
    assert np.all(At.sum(axis=0) == delta) and np.all(At.sum(axis=1) == delta)
    O = np.zeros((N, m), dtype=np.uint8)
    for p in range(1, delta + 1):
        match = maximum_bipartite_matching(csr_matrix(At), perm_type="column")  # row i -> column
        assert np.all(match >= 0), "Claim 1: a perfect matching exists"
        P = np.zeros_like(At)
        P[np.arange(N), match] = 1
        O[P == 1] = p
        At = At - P
    assert At.sum() == 0
    return O


def order_from_O(O: np.ndarray) -> np.ndarray:
    """Per-worker processing order (m x delta, -1 padded) from an ordering
    matrix: column j lists D_i by increasing O_ij."""
    N, m = O.shape
    delta = int(max((O[:, j] > 0).sum() for j in range(m)))
    order = -np.ones((m, delta), dtype=np.int32)
    for j in range(m):
        for i in range(N):
            if O[i, j]:
                order[j, int(O[i, j]) - 1] = i
    return order


def completion_times(order: np.ndarray, tau: np.ndarray, N: int, ell: int, theta: int = 0):
    """Completion-time simulation of Sec. IV.  Realization r: W_j needs
    tau[r, j] per chunk (+inf = failed) and finishes its p-th chunk (1-based)
    at p * tau_j.  Returns, per realization,
      T      the first time at which the error estimate sum_i max(0, ell -
             n_i(T)) is <= theta, n_i(T) = copies of D_i processed by T
             (theta = 0: every chunk processed ell times);
      psi    chunks each worker has processed by T;
      T_full the same time when a copy counts only once its worker has
             processed all of its chunks (the original protocol of Sec. IV).
    The estimate only drops at the ell earliest completion times of each
    chunk, so T is the (N ell - theta)-th smallest of those N ell times."""
    tau = np.asarray(tau, dtype=np.float64)
    m, delta = order.shape
    dj = [int((order[j] >= 0).sum()) for j in range(m)]
    nsim = tau.shape[0]
    T = np.zeros(nsim)
    TF = np.zeros(nsim)
    psi = np.zeros((nsim, m), dtype=np.int32)
    k = N * ell - theta
    for r in range(nsim):
        times = [[] for _ in range(N)]
        times_full = [[] for _ in range(N)]
        for j in range(m):
            t = float(tau[r, j])
            if not math.isfinite(t):
                continue
            for p in range(dj[j]):
                i = int(order[j, p])
                times[i].append(float(p + 1) * t)
                times_full[i].append(float(dj[j]) * t)
        vals, vals_full = [], []
        for i in range(N):
            vals += (sorted(times[i]) + [math.inf] * ell)[:ell]
            vals_full += (sorted(times_full[i]) + [math.inf] * ell)[:ell]
        T[r] = sorted(vals)[k - 1] if k >= 1 else 0.0
        TF[r] = sorted(vals_full)[k - 1] if k >= 1 else 0.0
        for j in range(m):
            t = float(tau[r, j])
            if math.isfinite(t):
                psi[r, j] = sum(1 for p in range(1, dj[j] + 1) if float(p) * t <= T[r])
    return T, psi, TF


# --------------------------------------------------------------------------
# Chunk gradients (Sec. I): g_{D_j} = sum_{i in D_j} grad l(x_i, y_i, w)
# --------------------------------------------------------------------------
def _sigmoid(z: np.ndarray) -> np.ndarray:
    out = np.empty_like(z)
    pos = z >= 0
    out[pos] = 1.0 / (1.0 + np.exp(-z[pos]))
    ez = np.exp(z[~pos])
    out[~pos] = ez / (1.0 + ez)
    return out


def point_losses(X: np.ndarray, y: np.ndarray, w: np.ndarray, loss: int) -> np.ndarray:
    """Per-point prediction error l(x_i, y_i, w) (Sec. I).
    Least squares: l = (x^T w - y)^2 / 2.  Logistic with y in {-1,+1}:
    l = log(1 + exp(-y x^T w))."""
    X = np.asarray(X, dtype=np.float64)
    z = X @ np.asarray(w, dtype=np.float64)
    y = np.asarray(y, dtype=np.float64)
    if loss == LSQ:
        return 0.5 * (z - y) ** 2
    t = -y * z
    return np.logaddexp(0.0, t)


def chunk_gradient(Xc: np.ndarray, yc: np.ndarray, w: np.ndarray, loss: int) -> np.ndarray:
    """g_{D} = sum over the chunk's points of grad_w l (Sec. I), un-normalised.
    Least squares: X^T (X w - y).  Logistic (y in {-1,+1}): X^T (sigma(X w) - y01)
    with y01 = (y + 1) / 2, which equals sum_i -y_i x_i sigma(-y_i x_i^T w)."""
    Xc = np.asarray(Xc, dtype=np.float64)
    yc = np.asarray(yc, dtype=np.float64)
    z = Xc @ np.asarray(w, dtype=np.float64)
    if loss == LSQ:
        r = z - yc
    else:
        r = _sigmoid(z) - (yc + 1.0) / 2.0
    return Xc.T @ r


def chunk_gradients(X, y, w, N: int, n_c: int, loss: int, chunks=None) -> np.ndarray:
    """All chunk gradients g_{D_i}, i in `chunks` (default all), streamed chunk
    by chunk so that a large X is never materialised in fp64.  `X` may be any
    array-like supporting row slicing (numpy array or torch CPU tensor)."""
    idx = range(N) if chunks is None else chunks
    out = []
    for i in idx:
        rows = slice(i * n_c, (i + 1) * n_c)
        Xc = _as_f64(X[rows])
        yc = _as_f64(y[rows])
        out.append(chunk_gradient(Xc, yc, w, loss))
    return np.stack(out) if out else np.zeros((0, 0))


def full_loss(X, y, w, Ntil: int, n_rows_per_block: int, loss: int) -> float:
    """L = (1/N~) sum_i l(x_i, y_i, w) (Sec. I), streamed in row blocks."""
    tot = 0.0
    for a in range(0, Ntil, n_rows_per_block):
        b = min(Ntil, a + n_rows_per_block)
        tot += float(np.sum(point_losses(_as_f64(X[a:b]), _as_f64(y[a:b]), _as_f64(w), loss)))
    return tot / Ntil


def _as_f64(a) -> np.ndarray:
    if hasattr(a, "detach"):  # torch tensor (bf16 has no numpy dtype)
        import torch  # local: only for CPU tensor conversion
        return a.detach().to(device="cpu", dtype=torch.float64).numpy()
    return np.asarray(a, dtype=np.float64)


# --------------------------------------------------------------------------
# Blocks (Sec. II): each g_{D_i} is split into ell disjoint parts g[k].
# --------------------------------------------------------------------------
def block_length(d: int, ell: int) -> int:
    return -(-d // ell)


def blocks(g: np.ndarray, ell: int) -> np.ndarray:
    """g -> ell x L matrix of contiguous blocks, zero padded to ell*L."""
    d = g.shape[-1]
    L = block_length(d, ell)
    pad = np.zeros(ell * L)
    pad[:d] = g
    return pad.reshape(ell, L)


def unblock(gb: np.ndarray, d: int) -> np.ndarray:
    return gb.reshape(-1)[:d]


# --------------------------------------------------------------------------
# The state vector psi and the support of B (Sec. II)
# --------------------------------------------------------------------------
def processed_chunks(order: np.ndarray, psi, j: int) -> list[int]:
    """Chunks W_j has processed: the first psi_j entries of its order (an
    empty slot, -1, holds no chunk)."""
    return [int(c) for c in order[j, : int(psi[j])] if c >= 0]


def completed_sets(order: np.ndarray, psi, N: int) -> list[list[int]]:
    """S_i = sorted workers that processed D_i (row support of B^(i))."""
    m = order.shape[0]
    S: list[list[int]] = [[] for _ in range(N)]
    for j in range(m):
        for i in processed_chunks(order, psi, j):
            S[i].append(j)
    return [sorted(s) for s in S]


def copies(order: np.ndarray, psi, N: int) -> np.ndarray:
    """Delta_i = |S_i|, the number of processed copies of D_i."""
    return np.array([len(s) for s in completed_sets(order, psi, N)], dtype=np.int64)


def support(order: np.ndarray, psi, N: int) -> np.ndarray:
    """N x m 0/1 matrix: entry (i, j) = 1 iff row j of B^(i) holds
    indeterminates, i.e. W_j processed D_i (Sec. II, eqs. 3 and 8)."""
    m = order.shape[0]
    s = np.zeros((N, m), dtype=np.uint8)
    for j in range(m):
        for i in processed_chunks(order, psi, j):
            s[i, j] = 1
    return s


def is_exact(order: np.ndarray, psi, N: int, ell: int) -> bool:
    """Exact-GC condition of Sec. II / II-A: every D_i processed >= ell times."""
    return bool(np.min(copies(order, psi, N)) >= ell)


def error_estimate(order: np.ndarray, psi, N: int, ell: int) -> float:
    """Overall approximate-GC error estimate, eq. (7) and the sentence after
    it: sum_i max(0, ell - Delta_i)."""
    return float(sum(max(0, ell - int(D)) for D in copies(order, psi, N)))


# --------------------------------------------------------------------------
# Algorithm 1, Find-Encoding-Coeff
# --------------------------------------------------------------------------
def find_encoding_coeff(R: np.ndarray, order: np.ndarray, psi, N: int, beta: int,
                        return_solved: bool = False):
    """Algorithm 1 run by worker W_beta; returns eps_beta = B(beta, :).

    Step 1: form the indeterminate matrix B from psi (support(...)).
    Step 2: extract B~_beta, the block columns of the chunks W_beta processed,
            in increasing chunk index i_1 < ... < i_alpha (eq. 5).
    Step 3: minimum-l2-norm least-squares solution of eq. (6),
            min || 1_alpha^T (x) I_ell - R B~_beta ||   (Frobenius norm),
            over all indeterminates of B~_beta, written as one linear system
            in the vector of indeterminates and solved with a minimum-norm
            least-squares routine (SVD based).
    Step 4: eps_beta = row beta of the solved matrix.

    With return_solved=True the whole m x N*ell matrix W_beta solved (its
    block columns filled, the others zero) is returned as well, so that the
    agreement between workers (Sec. II: the same minimisation is performed
    independently by every holder) can be checked.
    """
    ell, m = R.shape
    sup = support(order, psi, N)                          # step 1
    mine = sorted(processed_chunks(order, psi, beta))     # step 2
    alpha = len(mine)
    eps = np.zeros(N * ell)
    solved = np.zeros((m, N * ell))
    if alpha == 0:
        return (eps, solved) if return_solved else eps
    ncols = alpha * ell                                   # columns of B~_beta
    unknowns = []                                         # (row j, column c of B~)
    for a, i in enumerate(mine):
        for k in range(ell):
            c = a * ell + k
            for j in range(m):
                if sup[i, j]:
                    unknowns.append((j, c))
    # vec of the ell x ncols residual, entry (r, c) at r * ncols + c
    M = np.zeros((ell * ncols, len(unknowns)))
    for t, (j, c) in enumerate(unknowns):
        for r in range(ell):
            M[r * ncols + c, t] = R[r, j]
    target = np.zeros((ell, ncols))
    for a in range(alpha):
        target[:, a * ell:(a + 1) * ell] = np.eye(ell)   # 1_alpha^T (x) I_ell
    u = np.linalg.lstsq(M, target.reshape(-1), rcond=None)[0]   # step 3
    Bt = np.zeros((m, ncols))
    for t, (j, c) in enumerate(unknowns):
        Bt[j, c] = u[t]
    for a, i in enumerate(mine):                          # step 4
        eps[i * ell:(i + 1) * ell] = Bt[beta, a * ell:(a + 1) * ell]
        solved[:, i * ell:(i + 1) * ell] = Bt[:, a * ell:(a + 1) * ell]
    return (eps, solved) if return_solved else eps


def encoding_matrix(R: np.ndarray, order: np.ndarray, psi, N: int) -> np.ndarray:
    """The m x N*ell matrix B the workers agree on: row beta is the eps_beta
    that W_beta computes on its own with Algorithm 1 (rows of workers with
    psi_beta = 0 are zero: they transmit nothing useful)."""
    ell, m = R.shape
    B = np.zeros((m, N * ell))
    for beta in range(m):
        if int(psi[beta]) > 0:
            B[beta] = find_encoding_coeff(R, order, psi, N, beta)
    return B


def worker_coefficients(B: np.ndarray, order: np.ndarray, psi, ell: int) -> np.ndarray:
    """Per-worker encoding coefficients in processing order: E[j, p, k] =
    B[j, order[j,p]*ell + k] for p < psi_j, else 0.  (A re-indexing of
    eps_j that the C-ABI returns; m x delta x ell.)"""
    m, delta = order.shape
    E = np.zeros((m, delta, ell))
    for j in range(m):
        for p in range(int(psi[j])):
            i = int(order[j, p])
            E[j, p, :] = B[j, i * ell:(i + 1) * ell]
    return E


# --------------------------------------------------------------------------
# Encoding (eq. 2) and PS decoding (Sec. II-B)
# --------------------------------------------------------------------------
def encode(B: np.ndarray, G: np.ndarray, order: np.ndarray, psi, ell: int) -> np.ndarray:
    """Worker transmissions, eq. (2): g_beta = sum_i sum_{j<ell}
    B^(i)_{beta,j} g_{D_i}[j].  Terms with B^(i)_{beta,.} = 0 (chunks W_beta
    did not process) vanish, so the sum runs over W_beta's processed chunks."""
    m = B.shape[0]
    d = G.shape[1]
    L = block_length(d, ell)
    T = np.zeros((m, L))
    for beta in range(m):
        for i in processed_chunks(order, psi, beta):
            gb = blocks(G[i], ell)
            for j in range(ell):
                T[beta] += B[beta, i * ell + j] * gb[j]
    return T


def decode(R: np.ndarray, T: np.ndarray, d: int) -> np.ndarray:
    """PS decoding (Sec. II-B): sum_i g_{D_i}[k] ~= sum_j r_{kj} g_j for each
    block k; blocks are concatenated and the zero padding dropped."""
    ell, m = R.shape
    L = T.shape[1]
    out = np.zeros((ell, L))
    for k in range(ell):
        for j in range(m):
            out[k] += R[k, j] * T[j]
    return unblock(out, d)


def decode_fused(R: np.ndarray, B: np.ndarray, G: np.ndarray) -> np.ndarray:
    """The same decoded vector through the identity sum_j r_kj g_j =
    sum_i sum_k' (R B)[k, i*ell+k'] g_{D_i}[k'] (eq. 1 generalised to
    blocks).  Used as a self-check of the transmit path."""
    ell = R.shape[0]
    N, d = G.shape
    C = R @ B
    L = block_length(d, ell)
    out = np.zeros((ell, L))
    for i in range(N):
        gb = blocks(G[i], ell)
        for k in range(ell):
            for kp in range(ell):
                out[k] += C[k, i * ell + kp] * gb[kp]
    return unblock(out, d)


def decode_matrix(R: np.ndarray, B: np.ndarray) -> np.ndarray:
    """C = R B (ell x N*ell): row k gives the weight of every g_{D_i}[k'] in
    the decoded block k."""
    return R @ B


def coefficient_error(R: np.ndarray, B: np.ndarray, N: int) -> float:
    """Squared error of the decoding in coefficient space: the sum over
    k < ell of the least-squares errors for z_k (eq. 4, Sec. IV):
    || (1_N (x) I_ell)^T - R B ||_F^2."""
    ell = R.shape[0]
    Z = np.kron(np.ones((1, N)), np.eye(ell))
    return float(np.sum((Z - R @ B) ** 2))


def gradient_mse(ghat: np.ndarray, gtrue: np.ndarray) -> float:
    """Mean squared error of a decoded gradient against sum_i g_{D_i}."""
    diff = np.asarray(ghat, dtype=np.float64) - np.asarray(gtrue, dtype=np.float64)
    return float(diff @ diff) / diff.shape[0]


def sgd_step(w: np.ndarray, ghat: np.ndarray, lr: float, Ntil: int) -> np.ndarray:
    """w_{t+1} = w_t - lr * grad L with grad L = (1/N~) sum_j g_{D_j} (Sec. I)."""
    return np.asarray(w, dtype=np.float64) - lr * np.asarray(ghat, dtype=np.float64) / Ntil


# --------------------------------------------------------------------------
# One straggler pattern end to end
# --------------------------------------------------------------------------
@dataclass
class PatternResult:
    S: list
    Delta: np.ndarray
    support: np.ndarray
    B: np.ndarray
    E: np.ndarray
    C: np.ndarray
    T: np.ndarray | None
    ghat: np.ndarray | None
    coef_err: float
    est: float
    grad_mse: float | None


def run_pattern(R, order, psi, N, G=None, want_transmit=True) -> PatternResult:
    """psi -> S_i -> Algorithm 1 -> eq. (2) encode -> Sec. II-B decode -> errors."""
    ell, m = R.shape
    S = completed_sets(order, psi, N)
    Delta = np.array([len(s) for s in S], dtype=np.int64)
    sup = support(order, psi, N)
    B = encoding_matrix(R, order, psi, N)
    E = worker_coefficients(B, order, psi, ell)
    C = decode_matrix(R, B)
    ce = coefficient_error(R, B, N)
    est = float(sum(max(0, ell - int(D)) for D in Delta))
    T = ghat = gm = None
    if G is not None:
        d = G.shape[1]
        if want_transmit:
            T = encode(B, G, order, psi, ell)
            ghat = decode(R, T, d)
        else:
            ghat = decode_fused(R, B, G)
        gm = gradient_mse(ghat, G.sum(axis=0))
    return PatternResult(S, Delta, sup, B, E, C, T, ghat, ce, est, gm)

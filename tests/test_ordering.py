"""Algorithm 2 (Sec. III) chunk ordering: the oracle pinned against the
paper's optimality bound, brute force on tiny graphs and the Q_i definition;
the library's host implementation checked for validity and optimality on the
paper's graph sizes (several optimal orderings exist, so the unique parts --
row sums, column value sets, support -- are compared)."""
import itertools

import numpy as np
import pytest

import oracle as O
from workloads import random_order, random_regular_graph, second_eigenvalue


def _valid(Om, A):
    N, m = Om.shape
    delta = int(A[:, 0].sum())
    assert np.array_equal(Om > 0, A != 0)
    for j in range(m):
        assert sorted(int(v) for v in Om[:, j] if v) == list(range(1, delta + 1))
    return delta


def _brute_min_max_rowsum(A):
    """min over all orderings of max_i sum_j O_ij (every column independently
    permuted), by enumeration."""
    N, m = A.shape
    cols = [np.flatnonzero(A[:, j]) for j in range(m)]
    delta = len(cols[0])
    perms = list(itertools.permutations(range(1, delta + 1)))
    best = None
    for choice in itertools.product(range(len(perms)), repeat=m):
        rows = np.zeros(N, dtype=int)
        for j, c in enumerate(choice):
            rows[cols[j]] += perms[c]
        v = rows.max()
        best = v if best is None else min(best, v)
    return best


@pytest.mark.parametrize("m,nu,seed", [(5, 2, 0), (6, 3, 1), (6, 2, 2)])
def test_alg2_oracle_matches_brute_force_optimum(m, nu, seed):
    A = random_regular_graph(m, nu, seed)
    Om = O.chunk_ordering(A)
    delta = _valid(Om, A)
    opt = _brute_min_max_rowsum(A)
    assert opt == delta * (delta + 1) // 2          # the counting bound is tight (Sec. III)
    assert Om.astype(int).sum(axis=1).max() == opt


def test_q_metric_matches_its_definition_by_enumeration():
    """Q_i(O): the most chunks the cluster can process with no copy of D_i
    processed, maximised over every psi in {0..delta}^m."""
    A = random_regular_graph(5, 2, 3)
    Om = O.chunk_ordering(A)
    N, m = Om.shape
    delta = 2
    order = O.order_from_O(Om)
    best = np.zeros(N, dtype=int)
    for psi in itertools.product(range(delta + 1), repeat=m):
        done = set()
        for j in range(m):
            done.update(int(c) for c in order[j, :psi[j]])
        for i in range(N):
            if i not in done:
                best[i] = max(best[i], sum(psi))
    assert np.array_equal(best, O.q_metric(Om, delta))


@pytest.mark.parametrize("m,nu,seed", [(20, 4, 0), (200, 8, 1), (300, 8, 2)])
def test_alg2_oracle_optimal_on_paper_graphs(m, nu, seed):
    A = random_regular_graph(m, nu, seed)
    assert second_eigenvalue(A) < 2 * np.sqrt(nu - 1)   # Ramanujan, as the paper's G1, G2
    Om = O.chunk_ordering(A)
    delta = _valid(Om, A)
    assert np.all(Om.astype(int).sum(axis=1) == delta * (delta + 1) // 2)
    Q = O.q_metric(Om, delta)
    assert Q.max() == delta * (delta + 1) // 2 + (m - delta - 1) * delta
    # best of 100 random orderings is no better (Sec. IV's comparison)
    qr = min(O.q_metric(O.ordering_matrix(random_order(A, seed, k), m)[1], delta).max()
             for k in range(100))
    assert qr >= Q.max()


def _lib():
    from paper_2405_19509_gb300 import binding
    return binding


@pytest.mark.parametrize("m,nu,seed", [(20, 4, 0), (200, 8, 1), (300, 8, 2), (6, 3, 1)])
def test_library_alg2_valid_optimal_deterministic(m, nu, seed):
    gc = _lib()
    A = random_regular_graph(m, nu, seed)
    order, Om = gc.gc_chunk_ordering(A)
    delta = _valid(Om, A)
    assert np.all(Om.astype(int).sum(axis=1) == delta * (delta + 1) // 2)
    assert np.array_equal(O.order_from_O(Om), order)
    order2, Om2 = gc.gc_chunk_ordering(A)
    assert np.array_equal(order, order2) and np.array_equal(Om, Om2)
    # the order is a valid explicit assignment with the same A and O
    A3, order3, Om3 = gc.gc_make_assignment(m, m, delta, gc.GC_EXPLICIT, order)
    assert np.array_equal(A3, A) and np.array_equal(Om3, Om) and np.array_equal(order3, order)


def test_library_alg2_on_cyclic_assignment_is_optimal():
    gc = _lib()
    A, _, _ = gc.gc_make_assignment(20, 20, 4, gc.GC_CYCLIC)
    order, Om = gc.gc_chunk_ordering(A)
    _valid(Om, A)
    assert np.all(Om.astype(int).sum(axis=1) == 10)


def test_library_alg2_rejects_irregular():
    gc = _lib()
    A = random_regular_graph(20, 4, 0).copy()
    A[0, :] = 0
    with pytest.raises(gc.GCError) as e:
        gc.gc_chunk_ordering(A)
    assert e.value.code == -2
    B = np.ones((4, 5), dtype=np.uint8)
    with pytest.raises(gc.GCError) as e:
        gc.gc_chunk_ordering(B)
    assert e.value.code == -2

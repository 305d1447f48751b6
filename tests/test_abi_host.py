"""C-ABI checks that need no GPU: the library loads, exports every symbol
include/gc.h declares, the host-only assignment is bit-exact with the oracle,
and argument validation returns its codes before any launch."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _lib():
    gc = pytest.importorskip("paper_2405_19509_gb300", reason="libgc.so not built")
    return gc


def _declared():
    with open(os.path.join(ROOT, "include", "gc.h")) as f:
        src = f.read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(gc_\w+)\s*\(", src)))


def test_header_symbols_exported():
    gc = _lib()
    names = _declared()
    assert len(names) >= 15
    for n in names:
        assert hasattr(gc.lib, n), f"{n} declared in gc.h but not exported"
        assert isinstance(getattr(gc.lib, n), ctypes._CFuncPtr)


def test_version_and_error_text():
    gc = _lib()
    assert gc.gc_version() >= 100
    assert isinstance(gc.gc_last_error(), str)


@pytest.mark.parametrize("N,delta", [(6, 3), (20, 4), (64, 8), (128, 6), (256, 16)])
def test_cyclic_assignment_bit_exact(N, delta):
    gc = _lib()
    A, order, Om = gc.gc_make_assignment(N, N, delta, gc.GC_CYCLIC)
    o_ref = O.cyclic_order(N, N, delta)
    A_ref, O_ref = O.ordering_matrix(o_ref, N)
    assert np.array_equal(order, o_ref)
    assert np.array_equal(A, A_ref)
    assert np.array_equal(Om, O_ref)


def test_explicit_assignment_worked_example():
    gc = _lib()
    import json
    with open(os.path.join(ROOT, "tests", "golden", "worked_example.json")) as f:
        g = json.load(f)
    ex = np.array(g["order"], dtype=np.int32)
    A, order, Om = gc.gc_make_assignment(g["N"], g["m"], ex.shape[1], gc.GC_EXPLICIT, ex)
    A_ref, O_ref = O.ordering_matrix(ex, g["N"])
    assert np.array_equal(order, ex)
    assert np.array_equal(A, A_ref) and np.array_equal(Om, O_ref)


def _code(fn, *args):
    gc = _lib()
    with pytest.raises(gc.GCError) as ei:
        fn(*args)
    return ei.value.code


def test_assignment_validation():
    gc = _lib()
    assert _code(gc.gc_make_assignment, 6, 5, 3, gc.GC_CYCLIC) == -2          # N != m
    assert _code(gc.gc_make_assignment, 6, 6, 33, gc.GC_CYCLIC) == -3         # delta > 32
    bad = np.array([[0, 0], [1, 2]], dtype=np.int32)                           # chunk twice
    assert _code(gc.gc_make_assignment, 3, 2, 2, gc.GC_EXPLICIT, bad) == -1
    gap = np.array([[-1, 0], [1, 2]], dtype=np.int32)                          # chunk after empty
    assert _code(gc.gc_make_assignment, 3, 2, 2, gc.GC_EXPLICIT, gap) == -1
    oob = np.array([[0, 3], [1, 2]], dtype=np.int32)                           # chunk >= N
    assert _code(gc.gc_make_assignment, 3, 2, 2, gc.GC_EXPLICIT, oob) == -1


def test_device_entry_validation_before_launch():
    """Raw C calls with NULL device pointers or bad shapes must return an error
    code without touching the GPU (no device here)."""
    gc = _lib()
    L = gc.lib
    p = ctypes.c_void_p(0)
    # NULL required pointers
    assert L.gc_chunk_grads(None, 0, None, None, 1, 1, 1, 0, None, None, None, 0, None) == -1
    assert L.gc_decode_batch(None, 2, None, 6, 6, 3, None, 4, None, 64, None, None, None, None,
                             None, 0, None) == -1
    # unsupported ell / delta
    assert L.gc_encode(p, 9, p, 6, 6, 3, p, 1, p, 64, p, p, 1 << 20, None) == -3
    assert L.gc_find_encoding_coeff(p, 2, p, 6, 6, 33, p, 1, None, None, None, None, None, None,
                                    p, 1 << 20, None) == -3
    # bad shapes
    q = ctypes.c_void_p(4096)
    assert L.gc_decode_tx(q, 0, 6, q, 1, 64, q, None) == -2
    assert L.gc_decode_tx(q, 9, 6, q, 1, 64, q, None) == -3
    assert L.gc_sgd_step(None, q, 8, ctypes.c_float(0.1), 10, None) == -1
    assert L.gc_sgd_step(ctypes.c_void_p(16), ctypes.c_void_p(16), 0, ctypes.c_float(0.1), 10, None) == -2
    # the live step: NULL inputs, bad shapes, unsupported ell, staging too large
    assert L.gc_live_step(None, q, 2, q, 6, 6, 3, q, q, 64, ctypes.c_float(0.1), 10, q, None, None,
                          None) == -1
    assert L.gc_live_step(q, q, 2, q, 6, 6, 3, q, q, 0, ctypes.c_float(0.1), 10, q, None, None,
                          None) == -2
    assert L.gc_live_step(q, q, 9, q, 6, 6, 3, q, q, 64, ctypes.c_float(0.1), 10, q, None, None,
                          None) == -3
    assert L.gc_live_step(q, q, 8, q, 4096, 4096, 32, q, q, 64, ctypes.c_float(0.1), 10, q, None,
                          None, None) == -3
    # workspace missing / too small / misaligned
    need = L.gc_decode_batch_workspace(6, 6, 3, 2, 4, 64)
    assert need > 256
    fake = ctypes.c_void_p(4096)
    assert L.gc_decode_batch(fake, 2, fake, 6, 6, 3, fake, 4, fake, 64, fake, None, None, None,
                             None, need, None) == -6
    assert L.gc_decode_batch(fake, 2, fake, 6, 6, 3, fake, 4, fake, 64, fake, None, None, None,
                             ctypes.c_void_p(4096), need - 1, None) == -6
    assert L.gc_decode_batch(fake, 2, fake, 6, 6, 3, fake, 4, fake, 64, fake, None, None, None,
                             ctypes.c_void_p(4096 + 8), need, None) == -6
    # neither output requested
    assert L.gc_decode_batch(fake, 2, fake, 6, 6, 3, fake, 4, fake, 64, None, None, None, None,
                             ctypes.c_void_p(4096), need, None) == -1
    assert "NULL" in gc.gc_last_error()


def test_workspace_sizes_monotone():
    gc = _lib()
    L = gc.lib
    a = L.gc_decode_batch_workspace(20, 20, 4, 2, 100, 4096)
    b = L.gc_decode_batch_workspace(20, 20, 4, 2, 10000, 4096)
    assert 0 < a < b
    assert L.gc_chunk_grads_workspace(20, 512, 4096, 0) > 256
    assert L.gc_coeff_workspace(6, 6, 3, 9, 4) == 0   # unsupported -> 0


def test_wait_limit_knob_validation():
    gc = _lib()
    assert gc.lib.gc_set_wait_limit(-1) == -1
    assert gc.lib.gc_set_wait_limit(0) == 0
    assert gc.lib.gc_inject_stall(8) == -1
    assert gc.lib.gc_inject_stall(0) == 0
    # decode path policy: the three documented values, anything else rejected
    assert gc.lib.gc_set_decode_policy(3) == -1
    assert gc.lib.gc_set_decode_policy(-1) == -1
    for pol in (gc.GC_DECODE_DENSE, gc.GC_DECODE_RESIDUAL, gc.GC_DECODE_AUTO):
        assert gc.lib.gc_set_decode_policy(pol) == 0


def test_batched_chunk_grads_validation():
    gc = _lib()
    L = gc.lib
    nul = None
    # unsupported shapes are rejected on the host before anything runs
    assert L.gc_chunk_grads_batched(nul, nul, nul, 2, 128, 256, 48, 0, nul, nul, 0, nul) == -3
    assert L.gc_chunk_grads_batched(nul, nul, nul, 2, 128, 200, 32, 0, nul, nul, 0, nul) == -3
    assert L.gc_chunk_grads_batched(nul, nul, nul, 2, 100, 256, 32, 0, nul, nul, 0, nul) == -3
    assert L.gc_chunk_grads_batched(nul, nul, nul, 2, 128, 256, 32, 0, nul, nul, 0, nul) == -1
    assert L.gc_chunk_grads_batched_workspace(2, 128, 256, 32) > 256


def test_binding_without_library_raises(tmp_path):
    """The package has no CPU fallback: a copy of its Python files without
    libgc.so beside them refuses to import, naming the missing library."""
    import shutil
    import subprocess
    import sys
    pkg = os.path.join(ROOT, "paper_2405_19509_gb300")
    dst = tmp_path / "paper_2405_19509_gb300"
    dst.mkdir()
    for name in os.listdir(pkg):
        if name.endswith(".py"):
            shutil.copy(os.path.join(pkg, name), dst / name)
    assert not (dst / "libgc.so").exists()
    r = subprocess.run([sys.executable, "-c", "import paper_2405_19509_gb300"], cwd=tmp_path,
                       capture_output=True, text=True, timeout=300,
                       env={**os.environ, "PYTHONPATH": str(tmp_path)})
    assert r.returncode != 0
    assert "ImportError" in r.stderr and "libgc.so is missing" in r.stderr

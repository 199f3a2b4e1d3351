"""The C ABI without a GPU: the library loads, exports every symbol that
include/agn.h declares, its host-side generator reproduces agn_inputs bit for
bit, and invalid arguments are rejected with the documented codes."""

import math
import os
import re
import subprocess

import numpy as np
import pytest

import agn_inputs as I
from agn_inputs import workloads as WL

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def agn():
    import __graft_entry__ as g
    g.build()
    import paper_1710_02368_gb300 as agn
    return agn


def _declared_symbols():
    syms = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            text = open(os.path.join(ROOT, "include", fn)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            syms |= set(re.findall(r"\b(agn_\w+)\s*\(", text))
    return syms


def test_library_exports_every_declared_symbol(agn):
    out = subprocess.run(["nm", "-D", "--defined-only", agn.library_path()],
                         capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\bT (agn_\w+)", out))
    declared = _declared_symbols()
    assert declared, "no declarations found"
    assert declared <= exported, declared - exported
    from paper_1710_02368_gb300 import _lib
    assert declared <= set(_lib.SIGNATURES), declared - set(_lib.SIGNATURES)
    lib = _lib.load()
    for s in declared:
        assert hasattr(lib, s)


@pytest.mark.parametrize("n,C,lo,hi,seed", [(4, 50, 0, 2, I.DEFAULT_SEED),
                                             (16, 2000, 0, 15, I.DEFAULT_SEED),
                                             (32, 300, 31, 31, 5), (3, 100, 1, 7, 99)])
def test_schedule_matches_python_generator(agn, n, C, lo, hi, seed):
    w, t = agn.agn_make_schedule(n, C, lo, hi, seed)
    pw, pt = I.make_schedule(n, C, lo, hi, seed)
    assert np.array_equal(w, pw) and np.array_equal(t, pt)


@pytest.mark.parametrize("w,rows", [
    (WL.SMALL, (0, 2048)),
    (WL.MNIST_SHAPED, (3750 * 5 - 7, 300)),
    (WL.WIDE_BF16, (1562 * 3, 40)),
    (WL.LARGE_BF16, (99000, 1000)),
], ids=lambda v: getattr(v, "name", str(v)))
def test_generated_inputs_match_python_generator(agn, w, rows):
    row0, nr = rows
    x, y, th = agn.agn_generate_inputs(w.dims, w.dist, I.DEFAULT_SEED, row0, nr,
                                       teacher_dims=w.teacher_dims,
                                       want_theta=(w.dims[1] <= 1000))
    r = np.arange(row0, row0 + nr)
    px = I.make_inputs_x(I.DEFAULT_SEED, w.dims[0], r, w.dist)
    assert np.array_equal(x, px)
    py = I.teacher_labels(px, I.teacher_params(I.DEFAULT_SEED, w.teacher_dims), w.dist)
    assert np.array_equal(y, py)
    if th is not None:
        assert np.array_equal(th, I.init_params(I.DEFAULT_SEED, w.dims))


def test_generate_inputs_rejects_bad_arguments(agn):
    with pytest.raises(agn.AGNError) as e:
        agn.agn_generate_inputs([784, 0, 10], 0, 1, 0, 4)
    assert e.value.code == agn.AGN_E_INVALID
    with pytest.raises(agn.AGNError) as e:
        agn.agn_generate_inputs([784, 10], 0, 1, 0, 4, teacher_dims=[700, 10])
    assert e.value.code == agn.AGN_E_INVALID


def test_make_schedule_rejects_bad_arguments(agn):
    for args in [(0, 10, 0, 0, 1), (4, 10, 3, 2, 1), (4, 10, -1, 2, 1)]:
        with pytest.raises(agn.AGNError) as e:
            agn.agn_make_schedule(*args)
        assert e.value.code == agn.AGN_E_INVALID


def test_create_validates_before_touching_the_device(agn):
    for dims, n, lam, eta in [((784,), 4, 5, 0.1), ((784, 0, 10), 4, 5, 0.1),
                              ((784, 10), 0, 5, 0.1), ((784, 10), 4, 0, 0.1),
                              ((784, 10), 4, 5, -1.0), ((784, 10), 300, 5, 0.1)]:
        with pytest.raises(agn.AGNError) as e:
            agn.agn_create(dims, n, lam, eta, 1)
        assert e.value.code == agn.AGN_E_INVALID
    o = agn.agn_default_options()
    o.precision = 7
    with pytest.raises(agn.AGNError) as e:
        agn.agn_create((8, 4), 2, 1, 0.1, 1, o)
    assert e.value.code == agn.AGN_E_INVALID
    o = agn.agn_default_options()
    assert o.commit_rule == agn.AGN_COMMIT_AGN
    o.commit_rule = 5
    with pytest.raises(agn.AGNError) as e:
        agn.agn_create((8, 4), 2, 1, 0.1, 1, o)
    assert e.value.code == agn.AGN_E_INVALID


def test_temporal_efficiency_through_the_abi(agn):
    """Eq. 4 in the library (host code) against the oracle's restatement."""
    import oracle as O
    rng = np.random.default_rng(5)
    for _ in range(20):
        na, nb = rng.integers(1, 12, 2)
        ta = np.sort(rng.uniform(0, 10, na)); ta[-1] = max(ta[-1], 0.5)
        tb = np.sort(rng.uniform(0, 10, nb)); tb[-1] = max(tb[-1], 0.5)
        fa, fb = rng.uniform(0.1, 1, na), rng.uniform(0.1, 1, nb)
        got = agn.agn_temporal_efficiency(ta, fa, tb, fb)
        assert math.isclose(got, O.temporal_efficiency(ta, fa, tb, fb), rel_tol=1e-12)
    for bad in [([], [], [0, 1], [1, 1]), ([0, 2, 1], [1, 1, 1], [0, 1], [1, 1]),
                ([0, 1], [1, 1], [0, 1], [0, 0])]:
        with pytest.raises(agn.AGNError) as e:
            agn.agn_temporal_efficiency(*bad)
        assert e.value.code == agn.AGN_E_INVALID


@pytest.mark.parametrize("entry", ["agn_commit_pull", "agn_commit_pull_noalloc"])
def test_commit_pull_rejects_pulls_without_buffers_before_reading_them(agn, entry):
    """Pull offsets that promise pulls with a null pull list (or no replicas)
    are rejected with AGN_E_INVALID before any pull index is read (no device
    is touched: validation comes first)."""
    import ctypes as C
    from paper_1710_02368_gb300 import _lib
    lib = _lib.load()
    fake = C.c_void_p(1 << 20)            # aligned, never dereferenced on the host
    cw = (C.c_int32 * 1)(0)
    po = (C.c_int32 * 2)(0, 2)
    pw = (C.c_int32 * 2)(0, 1)
    fn = getattr(lib, entry)
    rc = fn(fake, fake, fake, None, 64, 64, 2, 1, cw, po, None, 0.01, 10, 1, None, None)
    assert rc == agn.AGN_E_INVALID and "pulls need replicas" in agn.agn_last_error()
    rc = fn(fake, fake, None, None, 64, 64, 2, 1, cw, po, pw, 0.01, 10, 1, None, None)
    assert rc == agn.AGN_E_INVALID and "pulls need replicas" in agn.agn_last_error()


def test_debug_waits_validates_its_arguments(agn):
    """The bounded-wait test hook rejects a null handle and out-of-range values
    before touching anything."""
    import ctypes as C
    from paper_1710_02368_gb300 import _lib
    lib = _lib.load()
    assert lib.agn_debug_waits(None, 1000, 0) == agn.AGN_E_INVALID


def test_create_rejects_unknown_tc_mask_bits(agn):
    """tc_mask takes bits 0-9 (include/agn.h); anything outside is rejected
    before any device access."""
    for mask in (-1, 1024, 4096):
        o = agn.agn_default_options()
        o.tc_mask = mask
        with pytest.raises(agn.AGNError) as e:
            agn.agn_create((8, 4), 2, 1, 0.1, 1, o)
        assert e.value.code == agn.AGN_E_INVALID
        assert "tc_mask" in agn.agn_last_error()

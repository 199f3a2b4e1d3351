"""The bounds-checked build (-DAGN_BOUNDS_CHECK, libagn_gb300_check.so).

compute-sanitizer is not available on the GPUs these tests run on; this build
stands in for its memcheck on the library's kernels: every wrapped global
access is checked against the table of device buffers the library knows, an
access outside all of them is refused (not performed) and reported as
AGN_E_BOUNDS.  Each case (tests/bounds_cases.py) runs in a child process with
AGN_LIB_VARIANT=check: small ragged shapes through every kernel path, the
16-worker workload at full size, the standalone commit entry points, all
compared with the oracle; and the checker's own detection, with every buffer
registered 64 bytes short so that real in-allocation accesses are refused.
"""

import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def built():
    import __graft_entry__ as g
    g.build()
    from paper_1710_02368_gb300 import _lib
    assert os.path.exists(_lib.LIB_CHECK_PATH), "the bounds-checked library was not built"


def _case(name, extra_env=None):
    env = dict(os.environ, AGN_LIB_VARIANT="check", **(extra_env or {}))
    r = subprocess.run([sys.executable, os.path.join(ROOT, "tests", "bounds_cases.py"), name],
                       env=env, capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    return json.loads(r.stdout.strip().splitlines()[-1])


def test_fp32_tensor_core_path(built):
    r = _case("fp32_tc")
    assert r["rel"] <= 1e-5 and r["loss_err"] <= 1e-5, r


def test_fp32_separate_output_layer_tiled_dw_no_split_k(built):
    r = _case("fp32_tc_kernels")
    assert r["rel"] <= 1e-5 and r["loss_err"] <= 1e-5, r


def test_fp32_cuda_core_path(built):
    r = _case("fp32_simt")
    assert r["rel"] <= 1e-5 and r["loss_err"] <= 1e-5, r


def test_commit_rules_and_optimizers(built):
    r = _case("variants")
    assert all(v <= 1e-5 for v in r.values()), r


def test_bf16_path(built):
    r = _case("bf16")
    assert r["loss_err"] <= 2e-2, r


def test_mnist_shaped_workload_full_size(built):
    r = _case("mnist_shaped")
    assert r["rel"] <= 1e-5, r


def test_evaluation(built):
    r = _case("eval")
    assert r["loss_rel"] <= 1e-5, r


def test_standalone_commit_entry_points(built):
    r = _case("commit")
    assert all(r.values()), r


def test_checker_refuses_and_reports(built):
    r = _case("detect", {"AGN_BOUNDS_TEST_SHRINK": "64"})
    assert r["code"] == -8, r           # AGN_E_BOUNDS
    assert r["tail_untouched"] and r["head_committed"], r

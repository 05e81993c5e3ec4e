"""The range-checked build (libregmem_checked.so: the same sources compiled
with REGMEM_DEVICE_CHECKS, whose kernels check each index they derive before
a global access -- bank rows and tokens of the admission, sampled-query
tokens of the saliency, partial slots of the split units and of their merge
-- and record a failure in the status word, which the next call reports as
REGMEM_ERR_DEVICE_CHECK).  Parity tests that cover every kernel and the
split paths run again in a fresh process with that library loaded: no guard
may fail and the results must still match the oracle."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

TESTS = [
    "tests/test_gpu_parity.py::test_tiny_stream_full_oracle",
    "tests/test_gpu_parity.py::test_vggt_layer_first_frames",
    "tests/test_gpu_parity.py::test_split_units_across_many_ctas",
    "tests/test_gpu_parity.py::test_long_bank_sampled_rows",
    "tests/test_gpu_parity.py::test_admit_every_candidate",
    "tests/test_gpu_parity.py::test_fused_step_matches_two_calls",
    "tests/test_gpu_variants.py::test_shared_admission_matches_oracle",
    "tests/test_zz_no_alloc.py::test_noalloc_matches_handle_path_on_two_calls",
]


def test_parity_with_the_range_checked_library():
    from paper_2609_23286_gb300 import regmem
    assert os.path.exists(regmem.CHECKED_LIB_PATH), "build() makes libregmem_checked.so"
    code = ("import sys, pytest\n"
            "from paper_2609_23286_gb300 import regmem\n"
            "regmem.load(regmem.CHECKED_LIB_PATH)\n"
            f"sys.exit(pytest.main({TESTS!r} + ['-q', '-x', '-p', 'no:cacheprovider']))\n")
    r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, capture_output=True, text=True,
                       timeout=900)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-2000:]
    assert " passed" in r.stdout

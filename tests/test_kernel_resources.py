"""Register and local-memory budgets of every kernel, read from ptxas's resource report
(nvcc -Xptxas -v for sm_103a, compiled on the CPU): no kernel spills registers to local
memory beyond one small documented case, and each tensor-core GEMM instance fits its
384-thread CTA in one SM's 65,536 registers."""
import glob
import os
import re
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor

import pytest

from paper_2607_18582_gb300 import build

# the 32-class output-layer variant (n_classes 17..32) holds 32 accumulators per thread;
# the 10-class workloads never launch it.  The generic delta kernel (every layer kind:
# convolution, dense, depthwise, embedding) keeps a few bytes of its slot context on the
# stack; it is bound by its memory traffic
SPILL_ALLOWED = {"_ZN4mure13k_final_denseILi32EEEvNS_11FinalParamsE": 16,
                 "_ZN4mure12k_patch_valsENS_15PatchValsParamsE": 16}
TC_THREADS = 384


def _report():
    nvcc = build._nvcc()
    if shutil.which(nvcc) is None and not os.path.exists(nvcc):
        pytest.skip("nvcc not available")
    out = os.path.join(build.BUILD, "ptxas_check")
    os.makedirs(out, exist_ok=True)

    def one(src):
        obj = os.path.join(out, os.path.basename(src)[:-3] + ".o")
        r = subprocess.run([nvcc] + build.NVCC_FLAGS + ["-Xptxas", "-v", "-c", src, "-o", obj],
                           capture_output=True, text=True)
        assert r.returncode == 0, r.stderr[-2000:]
        return r.stderr

    srcs = sorted(glob.glob(os.path.join(build.CSRC, "*.cu")))
    with ThreadPoolExecutor(max_workers=min(8, len(srcs))) as ex:
        logs = list(ex.map(one, srcs))
    funcs = {}
    for log in logs:
        cur = None
        for line in log.splitlines():
            m = re.search(r"Compiling entry function '(\w+)'", line)
            if m:
                cur = m.group(1)
                funcs[cur] = {}
            m = re.search(r"(\d+) bytes spill stores, (\d+) bytes spill loads", line)
            if m and cur:
                funcs[cur]["spill"] = max(int(m.group(1)), int(m.group(2)))
            m = re.search(r"Used (\d+) registers", line)
            if m and cur:
                funcs[cur]["regs"] = int(m.group(1))
    return funcs


@pytest.fixture(scope="module")
def report():
    return _report()


def test_every_kernel_reported(report):
    names = " ".join(report)
    for k in ("k_tc_gemm", "k_stage_simt", "k_conv_small", "k_patch_vals", "k_final_dense", "k_scores", "k_expand"):
        assert k in names, k
    assert all("regs" in v for v in report.values())


def test_no_register_spills(report):
    bad = {f: v["spill"] for f, v in report.items() if v.get("spill", 0) > SPILL_ALLOWED.get(f, 0)}
    assert not bad, bad


def test_tensor_core_kernel_fits_one_cta_per_sm(report):
    tc = {f: v["regs"] for f, v in report.items() if "k_tc_gemm" in f}
    assert len(tc) >= 4
    for f, r in tc.items():
        assert r * TC_THREADS <= 65536, (f, r)

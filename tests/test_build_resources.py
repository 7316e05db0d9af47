"""Register use and spills of every kernel as ptxas reports it (nvcc -Xptxas -v for sm_103a; no
device). The batch-1 kernels (stream-K, row-resident, table lookup), the packers and the quantizer
spill nothing; the narrow row-resident instantiations fit 128 registers, so two of their CTAs share
an SM (the next call's CTAs start beside the running ones); the kernels that spill a few bytes
today (the general kernel at M = 16, one low-batch variant, the base-3 fixed-point kernel) spill no
more than that."""
import concurrent.futures as cf
import os
import re
import shutil
import subprocess
import tempfile

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_00224_gb300", "csrc")

# spill-store bytes allowed per kernel (mangled-name fragment): today's figures
KNOWN_SPILLS = {
    "qtea_gemv_generic_kernelILi16E": 8,
    "qtea_gemv_mb_kernelILi2ELb1ELb0E": 8,
    "qtea_gemv_paper_b3_kernelILi4E": 80,
    "qtea_gemv_paper_b3_kernelILi2E": 16,
    "qtea_gemv_paper_b3_kernelILi1E": 16,
}


def _ptxas_report(src, out_dir):
    cmd = ["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17", "-Xcompiler", "-fPIC",
           "-I", os.path.join(ROOT, "include"), "-I", CSRC, "-Xptxas", "-v", "-c", src,
           "-o", os.path.join(out_dir, os.path.basename(src) + ".o")]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr[-2000:]
    return r.stderr


def _kernels(report):
    """Entry functions: name -> (registers, spill-store bytes, spill-load bytes)."""
    out, name, spills = {}, None, (0, 0)
    for line in report.splitlines():
        m = re.search(r"Compiling entry function '(\S+)'", line)
        if m:
            name, spills = m.group(1), (0, 0)
            continue
        m = re.search(r"(\d+) bytes spill stores, (\d+) bytes spill loads", line)
        if m and name:
            spills = (int(m.group(1)), int(m.group(2)))
            continue
        m = re.search(r"Used (\d+) registers", line)
        if m and name:
            out[name] = (int(m.group(1)),) + spills
            name = None
    return out


@pytest.fixture(scope="module")
def kernels():
    if shutil.which("nvcc") is None:
        pytest.skip("nvcc not on PATH")
    srcs = sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cu"))
    with tempfile.TemporaryDirectory() as d, cf.ThreadPoolExecutor(max(1, min(8, os.cpu_count() or 1))) as ex:
        reports = list(ex.map(lambda s: _ptxas_report(s, d), srcs))
    k = {}
    for rep in reports:
        k.update(_kernels(rep))
    return k


def test_every_kernel_is_reported(kernels):
    for frag in ("qtea_gemv_m1_kernel", "qtea_gemv_rows_kernel", "qtea_gemv_lut_kernel", "qtea_gemv_mb_kernel",
                 "qtea_pack_2bit_kernel", "qtea_quant"):
        assert any(frag in n for n in kernels), frag


def test_no_spills_beyond_the_known_ones(kernels):
    for name, (regs, st, ld) in kernels.items():
        allowed = next((b for frag, b in KNOWN_SPILLS.items() if frag in name), 0)
        assert st <= allowed and ld <= max(allowed, st), f"{name}: {st} B spill stores, {ld} B loads"


def test_hot_kernels_spill_nothing(kernels):
    for name, (regs, st, ld) in kernels.items():
        if any(f in name for f in ("qtea_gemv_m1_kernel", "qtea_gemv_rows_kernel", "qtea_gemv_lut_kernel",
                                   "qtea_pack_", "qtea_quant")):
            assert st == 0 and ld == 0, name


def test_narrow_row_resident_instantiations_fit_two_ctas_per_sm(kernels):
    narrow = {n: v for n, v in kernels.items() if "qtea_gemv_rows_kernel" in n and "Lb0E" in n}
    wide = {n: v for n, v in kernels.items() if "qtea_gemv_rows_kernel" in n and "Lb1E" in n}
    assert len(narrow) == 4 and len(wide) == 2
    assert all(regs <= 128 for regs, _, _ in narrow.values())  # 2 x 256 threads x 128 = 65,536
    assert all(regs <= 255 for regs, _, _ in wide.values())

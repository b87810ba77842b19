"""Host-side checks of the C-ABI boundary (no GPU needed)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "esspt.h")


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(esspt_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def libpath():
    from paper_1410_8043_gb300 import build

    return build.build()


def test_library_exports_every_declared_symbol(libpath):
    import torch  # noqa: F401  (loads the CUDA runtime the library links against)

    lib = ctypes.CDLL(libpath)
    names = _declared()
    assert len(names) >= 20
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_covers_the_header():
    from paper_1410_8043_gb300 import esspt

    assert sorted(esspt.EXPORTS) == _declared()


def test_config_struct_layout_matches_c(tmp_path):
    """The ctypes Config mirrors esspt_config byte for byte."""
    from paper_1410_8043_gb300 import esspt

    probe = tmp_path / "probe.c"
    probe.write_text(
        '#include <stdio.h>\n#include <stddef.h>\n#include "esspt.h"\n'
        "int main(void){printf(\"%zu %zu %zu %zu %zu %zu\\n\", sizeof(esspt_config),"
        " offsetof(esspt_config, essp_p), offsetof(esspt_config, seed), offsetof(esspt_config, stream),"
        " offsetof(esspt_config, essp_max_delay), offsetof(esspt_config, vap_v0));return 0;}\n"
    )
    exe = tmp_path / "probe"
    subprocess.check_call(["gcc", "-I", os.path.join(ROOT, "include"), str(probe), "-o", str(exe)])
    size, o_p, o_seed, o_stream, o_md, o_v0 = map(int, subprocess.check_output([str(exe)]).split())
    C = esspt.Config
    assert ctypes.sizeof(C) == size
    assert C.essp_p.offset == o_p and C.seed.offset == o_seed and C.stream.offset == o_stream
    assert C.essp_max_delay.offset == o_md and C.vap_v0.offset == o_v0


def test_status_codes_match_header():
    from paper_1410_8043_gb300 import esspt

    src = open(HEADER).read()
    for name, val in [("ESSPT_OK", esspt.OK), ("ESSPT_EINVAL", esspt.EINVAL), ("ESSPT_ESTATE", esspt.ESTATE),
                      ("ESSPT_ENOSPC", esspt.ENOSPC), ("ESSPT_ESTALE", esspt.ESTALE), ("ESSPT_ECUDA", esspt.ECUDA)]:
        assert re.search(rf"\b{name}\s*=\s*{val}\b", src)
    for name, val in esspt.MODELS.items():
        cname = {"ssp": "ESSPT_SSP_LAZY", "essp": "ESSPT_ESSP_EAGER", "external": "ESSPT_EXTERNAL",
                 "vap": "ESSPT_VAP", "ssp_row": "ESSPT_SSP_ROW"}[name]
        assert re.search(rf"\b{cname}\s*=\s*{val}\b", src)


def test_product_path_never_touches_the_oracle():
    """Neither the package nor bench.py's GPU leg imports or loads oracle/."""
    pkg = os.path.join(ROOT, "paper_1410_8043_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                text = open(os.path.join(dirpath, f)).read()
                assert "oracle" not in text.lower(), f
    bench = open(os.path.join(ROOT, "bench.py")).read()
    gpu_leg = bench[bench.index("def run_gpu("):bench.index("def cpu_baseline(")]
    assert "import oracle" not in gpu_leg and "from oracle" not in gpu_leg


def test_no_gpu_means_no_table():
    """Without a CUDA device the binding refuses to run (no CPU fallback)."""
    import torch

    from paper_1410_8043_gb300 import esspt

    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(RuntimeError):
        esspt.Table(10, 4, 1, 0)


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    from paper_1410_8043_gb300 import esspt

    monkeypatch.setattr(esspt, "_lib", None)
    monkeypatch.setattr(esspt, "LIB_PATH", str(tmp_path / "nope.so"))
    with pytest.raises(RuntimeError):
        esspt.lib()


def test_report_module_imports_without_gpu():
    """The staleness/convergence report is part of the package and imports on a CPU host."""
    from paper_1410_8043_gb300 import report

    assert callable(report.main) and callable(report.run_workload)

"""The C-ABI library loads and exports every entry point include/wdc.h declares
(no compute call: this runs without a GPU)."""
import ctypes
import os
import re

import pytest

from paper_2608_01845_gb300 import wdc

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "wdc.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(wdc_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for required in ["wdc_dit_forward", "wdc_scheduler_step", "wdc_surrogate_step", "wdc_risk_update", "wdc_rollout"]:
        assert required in names


def test_library_exports_every_declared_symbol():
    lib = ctypes.CDLL(wdc.LIB_PATH)
    missing = [n for n in _declared() if not hasattr(lib, n)]
    assert missing == []


def test_default_params_and_status_strings():
    p = wdc.default_params()
    assert p.bank_capacity == 4 and p.max_age == 6 and p.flags == 0
    assert wdc.LIB.wdc_status_string(0) == b"ok"
    assert wdc.LIB.wdc_status_string(6) == b"call out of order"


def test_struct_sizes_match_the_header_layout():
    # wdc_step_info: 7 ints, pad to 8-byte alignment, 12 doubles, 2 x 8 doubles
    assert ctypes.sizeof(wdc.StepInfo) == 8 * 4 + 12 * 8 + 16 * 8
    assert ctypes.sizeof(wdc.Cond) == 8 + 8 * 8


def test_ablation_flags_and_defaults_match_the_header():
    src = open(os.path.join(ROOT, "include", "wdc.h")).read()
    hdr = {m.group(1): int(m.group(2), 16) for m in re.finditer(r"#define WDC_ABL_([A-Z_]+)\s+0x([0-9A-Fa-f]+)", src)}
    names = ["PERIODIC", "SECANT", "INSTANT_RISK", "NO_IMPACT", "NO_CALIB", "NO_SUPPORT", "LINEAR_OBS", "NO_COND"]
    for n in names:
        assert getattr(wdc, "ABL_" + n) == hdr[n]
    assert hdr["ALL"] == sum(hdr[n] for n in names)
    m = re.search(r"#define WDC_OBS_RESIDUAL\s+0x([0-9A-Fa-f]+)", src)
    assert int(m.group(1), 16) == wdc.OBS_RESIDUAL and not (wdc.OBS_RESIDUAL & hdr["ALL"])
    p = wdc.default_params()
    assert p.period == 8 and p.ridge == 1e-6


@pytest.mark.parametrize("cname,pystruct", [("wdc_cache_params", "CacheParams"), ("wdc_dit_config", "DitConfig"),
                                             ("wdc_schedule", "Schedule"), ("wdc_cond", "Cond"),
                                             ("wdc_step_info", "StepInfo")])
def test_struct_layout_matches_a_c_compiler(tmp_path, cname, pystruct):
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    st = getattr(wdc, pystruct)
    fields = [f for f, _ in st._fields_]
    prog = tmp_path / "layout.c"
    prog.write_text('#include <stdio.h>\n#include <stddef.h>\n#include "wdc.h"\nint main(void) {\n'
                    f'  printf("%zu\\n", sizeof({cname}));\n'
                    + "".join(f'  printf("%zu\\n", offsetof({cname}, {f}));\n' for f in fields)
                    + "  return 0;\n}\n")
    exe = tmp_path / "layout"
    subprocess.run([cc, "-I", os.path.join(ROOT, "include"), "-I", "/usr/local/cuda/include", str(prog), "-o", str(exe)],
                   check=True)
    out = [int(x) for x in subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split()]
    assert out[0] == ctypes.sizeof(st)
    assert out[1:] == [getattr(st, f).offset for f in fields]


def test_batch_limit_matches_the_header():
    src = open(os.path.join(ROOT, "include", "wdc.h")).read()
    assert int(re.search(r"#define WDC_MAX_BATCH\s+(\d+)", src).group(1)) == wdc.MAX_BATCH


def test_observe_noalloc_binding_checks_sizes_before_the_call():
    """wdc_observe_noalloc has no context that knows the latent size, so the
    binding checks every tensor before calling in: a short statistics buffer
    (120 of the 123 values) or a weight count that differs from the latent
    count raises ValueError without reaching the library."""
    import torch
    z = torch.zeros(256, dtype=torch.float32)
    with pytest.raises(ValueError, match="stats"):
        wdc.observe_noalloc([z], [1.0], z, torch.zeros_like(z), torch.zeros(120, dtype=torch.float64))
    with pytest.raises(ValueError, match="weights"):
        wdc.observe_noalloc([z, z], [1.0], z, torch.zeros_like(z), torch.zeros(123, dtype=torch.float64))
    with pytest.raises(ValueError, match="z_out"):
        wdc.observe_noalloc([z[:128]], [1.0], z, torch.zeros_like(z), torch.zeros(123, dtype=torch.float64))
    with pytest.raises(ValueError, match="device"):
        wdc.observe_noalloc([z], [1.0], z, torch.zeros_like(z), torch.zeros(123, dtype=torch.float64))

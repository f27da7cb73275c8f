"""Host-side checks of the C ABI: the library builds and loads, exports every
symbol include/fva.h declares, and rejects bad arguments before touching a GPU."""
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

import workloads as WL

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="session")
def fva():
    import paper_2608_27384_gb300 as pkg
    from paper_2608_27384_gb300.build import build
    build()
    pkg.lib()
    return pkg


def header_functions():
    text = open(os.path.join(ROOT, "include", "fva.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(fva_[a-z0-9_]+)\s*\(", text)))


def test_exports_every_declared_symbol(fva):
    declared = header_functions()
    assert len(declared) >= 13
    out = subprocess.run(["nm", "-D", "--defined-only", fva.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (fva_\w+)", out))
    missing = [f for f in declared if f not in exported]
    assert not missing, missing
    assert set(declared) == set(fva.EXPORTS)
    for name in declared:
        getattr(fva.lib(), name)


def test_header_constants_match_binding(fva):
    """Every integer #define of include/fva.h (flags, ring size, ABI version) has the
    same value in the Python binding, and every enumerator the binding names exists
    in the header with that value."""
    text = open(os.path.join(ROOT, "include", "fva.h")).read()
    defines = dict((m.group(1), int(m.group(2)))
                   for m in re.finditer(r"#define (FVA_[A-Z0-9_]+) (\d+)u?\b", text))
    assert {"FVA_FLAG_NO_GRAPH", "FVA_STEP_REUSE_FILM", "FVA_STEP_SERIAL_FILM",
            "FVA_PARAM_RING", "FVA_ABI_VERSION"} <= set(defines)
    for name, value in defines.items():
        assert getattr(fva, name) == value, name
    enums = dict((m.group(1), int(m.group(2)))
                 for m in re.finditer(r"\b(FVA_[A-Z0-9_]+)\s*=\s*(\d+)", text))
    for name in ("FVA_FP32", "FVA_BF16"):
        assert getattr(fva, name) == enums[name], name


def _cfg(fva, **over):
    wl = WL.standard_workloads()["pi05_2view"]
    from paper_2608_27384_gb300.harness import config_for
    c = config_for(wl)
    for k, v in over.items():
        setattr(c, k, v)
    return c


def test_config_struct_layout(fva, tmp_path):
    """The binding's ctypes structs have the C header's layout (compiled with gcc)."""
    import shutil
    import subprocess
    assert ctypes.sizeof(fva.fva_config) == 80
    assert fva.fva_config.noise_seed.offset == 72
    assert ctypes.sizeof(fva.fva_step_opts) == 40
    assert fva.fva_step_opts.n_valid.offset == 32
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "layout.c"
    src.write_text(
        "#include <stdio.h>\n#include <stddef.h>\n#include \"fva.h\"\n"
        "int main(void) { printf(\"%zu %zu %zu %zu %zu\\n\", sizeof(fva_config),"
        " offsetof(fva_config, noise_seed), sizeof(fva_step_opts),"
        " offsetof(fva_step_opts, trace_out), offsetof(fva_step_opts, n_valid)); return 0; }\n")
    exe = tmp_path / "layout"
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    subprocess.run([cc, "-I", inc, str(src), "-o", str(exe)], check=True)
    got = [int(v) for v in subprocess.run([str(exe)], capture_output=True, text=True,
                                          check=True).stdout.split()]
    assert got == [ctypes.sizeof(fva.fva_config), fva.fva_config.noise_seed.offset,
                   ctypes.sizeof(fva.fva_step_opts), fva.fva_step_opts.trace_out.offset,
                   fva.fva_step_opts.n_valid.offset]


@pytest.mark.parametrize("field,value,status", [
    ("abi_version", 99, "FVA_ERR_INVALID_ARG"),
    ("dtype", 7, "FVA_ERR_INVALID_ARG"),
    ("n_layers", 0, "FVA_ERR_INVALID_ARG"),
    ("n_kv_heads", 2, "FVA_ERR_UNSUPPORTED"),
    ("head_dim", 128, "FVA_ERR_UNSUPPORTED"),
    ("n_q_heads", 3, "FVA_ERR_UNSUPPORTED"),
    ("width", 1000, "FVA_ERR_UNSUPPORTED"),
    ("rms_eps", 0.0, "FVA_ERR_INVALID_ARG"),
    ("t_max_period", 1e-3, "FVA_ERR_INVALID_ARG"),
    ("action_dim", 200, "FVA_ERR_UNSUPPORTED"),
    ("max_prefix", 9000, "FVA_ERR_UNSUPPORTED"),
])
def test_create_rejects_bad_config(fva, field, value, status):
    with pytest.raises(fva.FvaError) as e:
        fva.fva_create(_cfg(fva, **{field: value}))
    assert e.value.name == status
    assert fva.fva_last_error()


def test_weight_count_and_shapes(fva):
    for name, wl in WL.standard_workloads().items():
        from paper_2608_27384_gb300.harness import config_for
        c = config_for(wl)
        names = WL.weight_names(wl.n_layers)
        assert fva.fva_num_weights(c) == len(names)
        shapes = WL.tensor_shapes(wl)
        for i, n in enumerate(names):
            r, k = fva.fva_weight_shape(c, i)
            s = shapes[n.split(".")[-1]]
            assert (r, k) == ((1, s[0]) if len(s) == 1 else s), (name, n)
        with pytest.raises(fva.FvaError):
            fva.fva_weight_shape(c, len(names))


def test_null_arguments(fva):
    L = fva.lib()
    assert L.fva_step(None, None, None, None, 1, None) == 1
    assert L.fva_step_ex(None, None, None, None, 1, None, None) == 1
    assert L.fva_load_weights(None, None, 0, 0) == 1
    assert L.fva_set_prefix_kv(None, 0, 0, None, None, 0, 0, None) == 1
    assert L.fva_mask_table(None, 1, None, None) == 1
    assert L.fva_create(None, None) == 1
    L.fva_destroy(None)
    assert L.fva_trace_floats(None, 1) == 0
    assert "NULL" in fva.fva_last_error()


def test_create_without_gpu_reports_cuda_error(fva):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(fva.FvaError) as e:
        fva.fva_create(_cfg(fva))
    assert e.value.name == "FVA_ERR_CUDA"

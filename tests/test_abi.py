"""The C-ABI library loads and exports every symbol include/crf.h declares; the ctypes
mirror has the C compiler's struct layouts. No compute calls (runs without a GPU)."""
import ctypes
import os
import re
import shutil
import subprocess

import pytest

from paper_2609_30884_gb300 import abi, build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "crf.h")


@pytest.fixture(scope="module")
def lib():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        if not os.path.exists(abi.LIB_PATH):
            pytest.skip("no nvcc and no prebuilt library")
    else:
        build.build()
    return abi.load()


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"CRF_API\s+[\w\s\*]*?\b(crf_\w+)\s*\(", text)))


def test_header_declares_the_binding_exports():
    assert declared_functions() == sorted(abi.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
    # the binding's signatures are installed
    assert lib.crf_last_error.restype is ctypes.c_char_p


def test_last_error_is_empty_before_any_call(lib):
    assert lib.crf_last_error() in (b"", None)


STRUCTS = {
    "crf_model_dims": (abi.ModelDims, ["n_layers", "hidden", "n_q_heads", "n_kv_heads", "head_dim",
                                       "ffn", "vocab", "rms_eps", "rope_theta", "qkv_bias"]),
    "crf_lora_dims": (abi.LoraDims, ["rank", "alpha", "module_mask"]),
    "crf_layer_weights": (abi.LayerWeights, ["W", "bias", "ln1", "ln2"]),
    "crf_model": (abi.Model, ["dims", "layers", "embed", "final_norm", "lm_head"]),
    "crf_adapter": (abi.Adapter, ["dims", "A", "B"]),
    "crf_kv_pool": (abi.KVPool, ["k_pages", "v_pages", "num_pages"]),
    "crf_request": (abi.Request, ["n_tokens", "s", "e", "page_table", "tokens", "hidden_in",
                                  "hidden_out", "final_hidden_out"]),
    "crf_decode_row": (abi.DecodeRow, ["pos", "page_table", "token"]),
}


def test_struct_layouts_match_c(tmp_path):
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    lines = ['#include <stdio.h>', '#include <stddef.h>', f'#include "{HEADER}"', "int main(void){"]
    for sname, (_, fields) in STRUCTS.items():
        lines.append(f'printf("{sname} size %zu\\n", sizeof({sname}));')
        for f in fields:
            lines.append(f'printf("{sname}.{f} %zu\\n", offsetof({sname}, {f}));')
    lines.append('printf("enum %d %d %d\\n", CRF_MOD_DOWN, CRF_PAGE_SIZE, CRF_MAX_REQUESTS);')
    lines.append("return 0;}")
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    subprocess.run([cc, str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n")
    got = dict(l.rsplit(" ", 1) for l in out if l)
    for sname, (cls, fields) in STRUCTS.items():
        assert int(got[f"{sname} size"]) == ctypes.sizeof(cls), sname
        for f in fields:
            assert int(got[f"{sname}.{f}"]) == getattr(cls, f).offset, f"{sname}.{f}"
    assert got["enum 6 16"] == str(abi.MAX_REQUESTS)
    assert abi.PAGE_SIZE == 16 and abi.NUM_MODULES == 7


def test_debug_build_exports_every_declared_symbol():
    """The CRF_DEBUG variant (device-side page-id checks) builds from the same sources."""
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("no nvcc")
    path = build.build(debug=True)
    assert os.path.basename(path) == "libcrf_debug.so"
    dbg = ctypes.CDLL(path)
    for name in declared_functions():
        assert hasattr(dbg, name), name

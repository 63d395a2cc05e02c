"""Host-side checks of the C ABI (CPU only: no kernel is launched).

The library must build for sm_103a, load, export every entry point that
include/hscale.h declares, and reject bad arguments with a status code before it
enqueues anything.
"""
import ctypes
import pathlib
import re

import pytest

import paper_2608_28113_gb300 as hs
from paper_2608_28113_gb300 import build

HEADER = pathlib.Path(__file__).resolve().parent.parent / "include" / "hscale.h"

OK, ERR_NULL, ERR_SHAPE, ERR_ALIGN, ERR_ARG, ERR_CUDA, ERR_WS = range(7)


@pytest.fixture(scope="module")
def lib():
    build.build()
    return hs.load()


def declared_functions():
    text = HEADER.read_text()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\*?\s+\*?(hscale_\w+)\s*\(", text, flags=re.M)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("hscale_hessian_diag_accumulate", "hscale_rtn_scales",
                     "hscale_refine_scales", "hscale_pack_nvfp4"):
        assert required in names
    assert set(names) == set(hs.EXPORTED_SYMBOLS)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert hs.hscale_abi_version() == 4
    assert hs.library_path().exists()


def test_header_is_plain_c_and_every_symbol_links(lib, tmp_path):
    """include/hscale.h compiles as strict C99, and a C program that takes the address of
    every declared entry point links against the in-tree library and runs (host-only
    calls: the ABI version, a status string, an argument error)."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    names = declared_functions()
    src = tmp_path / "abi_check.c"
    src.write_text(
        "#include <stdio.h>\n#include \"hscale.h\"\n"
        "typedef void (*fn_t)(void);\n"
        "static const fn_t every[] = {\n" + "".join(f"  (fn_t)&{n},\n" for n in names) + "};\n"
        "int main(void) {\n"
        "  if (sizeof every / sizeof every[0] != %d) return 2;\n" % len(names) +
        "  printf(\"%d %s\\n\", hscale_abi_version(), hscale_status_string(HSCALE_ERR_SHAPE));\n"
        "  return hscale_refine_scales(0, 0, 4, 40, 0, 0, 4, 4, 0, 0, 0) == HSCALE_ERR_SHAPE ? 0 : 1;\n"
        "}\n")
    build_dir = hs.library_path().parent
    exe = tmp_path / "abi_check"
    cmd = [cc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", f"-I{HEADER.parent}", str(src),
           f"-L{build_dir}", "-lhscale", f"-Wl,-rpath,{build_dir}", "-o", str(exe)]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True)
    assert r.returncode == 0, (r.stdout, r.stderr)
    assert r.stdout.split()[0] == str(hs.hscale_abi_version())


def test_status_strings(lib):
    for s in range(7):
        assert hs.hscale_status_string(s)
    assert hs.hscale_status_string(99) == "unknown status"


FAKE = ctypes.c_void_p(0x10000)  # 64 KiB-aligned; never dereferenced: checks fail or no-op first
MIS = ctypes.c_void_p(0x10002)


def test_hessian_argument_errors(lib):
    f = lib.hscale_hessian_diag_accumulate
    assert f(None, 4, 64, 64, FAKE, None) == ERR_NULL
    assert f(FAKE, 4, 64, 64, None, None) == ERR_NULL
    assert f(FAKE, -1, 64, 64, FAKE, None) == ERR_SHAPE
    assert f(FAKE, 4, 60, 64, FAKE, None) == ERR_SHAPE        # n % 8
    assert f(FAKE, 4, 64, 32, FAKE, None) == ERR_SHAPE        # ld < n
    assert f(FAKE, 4, 64, 68, FAKE, None) == ERR_ALIGN        # ld % 8
    assert f(MIS, 4, 64, 64, FAKE, None) == ERR_ALIGN
    assert f(FAKE, 0, 64, 64, FAKE, None) == OK               # empty chunk: no-op
    assert f(None, 0, 0, 0, None, None) == OK
    fx = lib.hscale_hessian_diag_accumulate_ex
    assert fx(FAKE, 4, 64, 64, FAKE, 2, None) == ERR_ARG     # unknown flag bit
    assert fx(FAKE, 4, 64, 64, FAKE, 0xFFFFFFFF, None) == ERR_ARG
    assert fx(None, 4, 64, 64, FAKE, hs.HSCALE_HESSIAN_X_READY, None) == ERR_NULL
    assert fx(FAKE, 4, 60, 64, FAKE, hs.HSCALE_HESSIAN_X_READY, None) == ERR_SHAPE
    assert fx(FAKE, 0, 64, 64, FAKE, hs.HSCALE_HESSIAN_X_READY, None) == OK


def test_sharding_entry_point_argument_errors(lib):
    f = lib.hscale_hessian_sum_partials
    assert f(FAKE, 2, 64, 32, FAKE, None) == ERR_SHAPE        # ld < n
    assert f(FAKE, -1, 64, 64, FAKE, None) == ERR_SHAPE
    assert f(None, 2, 64, 64, FAKE, None) == ERR_NULL
    assert f(FAKE, 2, 64, 64, None, None) == ERR_NULL
    assert f(MIS, 2, 64, 64, FAKE, None) == ERR_ALIGN
    assert f(None, 0, 64, 64, None, None) == OK               # no parts: no-op
    g = lib.hscale_amax_bits
    assert g(FAKE, 4, 24, FAKE, None) == ERR_SHAPE            # n % 16
    assert g(FAKE, 4, 32, None, None) == ERR_NULL
    assert g(MIS, 4, 32, FAKE, None) == ERR_ALIGN
    assert g(FAKE, 4, 32, MIS, None) == ERR_ALIGN
    q = lib.hscale_global_scale_from_amax
    assert q(None, FAKE, None) == ERR_NULL and q(FAKE, None, None) == ERR_NULL
    assert q(MIS, FAKE, None) == ERR_ALIGN


def test_rtn_argument_errors(lib):
    f = lib.hscale_rtn_scales
    ws = hs.hscale_rtn_workspace_bytes()
    assert ws >= 4
    assert f(FAKE, 4, 24, FAKE, FAKE, FAKE, ws, None) == ERR_SHAPE   # n % 16
    assert f(None, 4, 32, FAKE, FAKE, FAKE, ws, None) == ERR_NULL
    assert f(FAKE, 4, 32, None, FAKE, FAKE, ws, None) == ERR_NULL
    assert f(FAKE, 4, 32, FAKE, FAKE, None, ws, None) == ERR_WS
    assert f(FAKE, 4, 32, FAKE, FAKE, FAKE, 2, None) == ERR_WS
    assert f(MIS, 4, 32, FAKE, FAKE, FAKE, ws, None) == ERR_ALIGN
    assert f(FAKE, -4, 32, FAKE, FAKE, FAKE, ws, None) == ERR_SHAPE
    assert f(None, 0, 32, None, None, None, 0, None) == OK


def test_refine_argument_errors(lib):
    f = lib.hscale_refine_scales
    assert f(FAKE, FAKE, 4, 32, FAKE, None, -1, 4, FAKE, FAKE, None) == ERR_ARG
    assert f(FAKE, FAKE, 4, 32, FAKE, None, 4, 126, FAKE, FAKE, None) == ERR_ARG
    assert f(FAKE, FAKE, 4, 40, FAKE, None, 4, 4, FAKE, FAKE, None) == ERR_SHAPE
    assert f(FAKE, FAKE, 4, 32, None, None, 4, 4, FAKE, FAKE, None) == ERR_NULL
    assert f(FAKE, FAKE, 4, 32, FAKE, None, 4, 4, None, FAKE, None) == ERR_NULL
    assert f(FAKE, MIS, 4, 32, FAKE, None, 4, 4, FAKE, FAKE, None) == ERR_ALIGN   # h 16-B
    assert f(FAKE, FAKE, 4, 32, FAKE, None, 4, 4, FAKE, ctypes.c_void_p(0x10004), None) == ERR_ALIGN
    assert f(None, None, 0, 32, None, None, 4, 4, None, None, None) == OK


def test_refine_ex_argument_errors(lib):
    f = lib.hscale_refine_scales_ex
    assert f(FAKE, FAKE, 4, 32, FAKE, None, 4, 4, FAKE, FAKE, -1, None) == ERR_ARG
    assert f(FAKE, FAKE, 4, 32, FAKE, None, -1, 4, FAKE, FAKE, 0, None) == ERR_ARG
    assert f(FAKE, FAKE, 4, 40, FAKE, None, 4, 4, FAKE, FAKE, 5, None) == ERR_SHAPE
    assert f(FAKE, FAKE, 4, 32, None, None, 4, 4, FAKE, FAKE, 5, None) == ERR_NULL
    assert f(None, None, 0, 32, None, None, 4, 4, None, None, 5, None) == OK


def test_refine_strided_argument_errors(lib):
    f = lib.hscale_refine_scales_strided
    ok = (FAKE, 64, FAKE, 4, 32, FAKE, None, 0, 0, 4, 4, FAKE, 4, FAKE, 32, 0, None)

    def call(**kw):
        names = ["w", "ld_w", "h", "m", "n", "sg", "init", "ld_i", "f46", "down", "up", "codes", "ld_c",
                 "packed", "ld_p", "ctas", "stream"]
        args = dict(zip(names, ok))
        args.update(kw)
        return f(*[args[k] for k in names])

    assert call(ld_w=16) == ERR_SHAPE                 # ld_w < n
    assert call(ld_w=36) == ERR_ALIGN                 # rows not 16-byte aligned
    assert call(ld_c=1) == ERR_SHAPE                  # ld_codes < n/16
    assert call(ld_p=8) == ERR_SHAPE                  # ld_packed < n/2
    assert call(ld_p=20) == ERR_ALIGN                 # ld_packed % 8
    assert call(init=FAKE, ld_i=1) == ERR_SHAPE       # ld_init < n/16
    assert call(f46=2) == ERR_ARG
    assert call(f46=1, init=FAKE) == ERR_ARG          # 4over6 decides the codes itself
    assert call(ctas=-1) == ERR_ARG
    assert call(down=126) == ERR_ARG
    assert call(codes=None) == ERR_NULL
    assert call(sg=None) == ERR_NULL
    assert call(w=MIS) == ERR_ALIGN
    assert call(h=MIS) == ERR_ALIGN
    assert call(n=40) == ERR_SHAPE
    assert call(m=0, w=None, codes=None) == OK        # empty view: no-op


def test_refine_ws_argument_errors(lib):
    assert lib.hscale_refine_workspace_bytes() == 16
    f = lib.hscale_refine_scales_ws
    ok = (FAKE, FAKE, 4, 32, FAKE, None, 0, 4, 4, FAKE, FAKE, 0, FAKE, 16, None)

    def call(**kw):
        names = ["w", "h", "m", "n", "sg", "init", "f46", "down", "up", "codes", "packed", "ctas", "ws", "wsb",
                 "stream"]
        args = dict(zip(names, ok))
        args.update(kw)
        return f(*[args[k] for k in names])

    assert call(wsb=15) == ERR_WS                     # smaller than the query
    assert call(ws=ctypes.c_void_p(0x10008)) == ERR_ALIGN
    assert call(f46=2) == ERR_ARG
    assert call(f46=1, init=FAKE) == ERR_ARG          # 4over6 decides the codes itself
    assert call(ctas=-1) == ERR_ARG
    assert call(down=126) == ERR_ARG
    assert call(n=40) == ERR_SHAPE
    assert call(codes=None) == ERR_NULL
    assert call(sg=None) == ERR_NULL
    assert call(h=MIS) == ERR_ALIGN
    assert call(m=0, w=None, codes=None) == OK        # empty: no-op
    assert call(m=0, w=None, codes=None, ws=None, wsb=0) == OK


def test_refine_4over6_argument_errors(lib):
    f = lib.hscale_refine_scales_4over6
    assert f(FAKE, FAKE, 4, 32, FAKE, 4, 4, FAKE, FAKE, -1, None) == ERR_ARG
    assert f(FAKE, FAKE, 4, 32, FAKE, -1, 4, FAKE, FAKE, 0, None) == ERR_ARG
    assert f(FAKE, FAKE, 4, 32, FAKE, 4, 126, FAKE, FAKE, 0, None) == ERR_ARG
    assert f(FAKE, FAKE, 4, 40, FAKE, 4, 4, FAKE, FAKE, 0, None) == ERR_SHAPE
    assert f(None, FAKE, 4, 32, FAKE, 4, 4, FAKE, FAKE, 0, None) == ERR_NULL
    assert f(FAKE, FAKE, 4, 32, None, 4, 4, FAKE, FAKE, 0, None) == ERR_NULL
    assert f(FAKE, FAKE, 4, 32, FAKE, 4, 4, None, FAKE, 0, None) == ERR_NULL
    assert f(FAKE, MIS, 4, 32, FAKE, 4, 4, FAKE, FAKE, 0, None) == ERR_ALIGN      # h 16-B
    assert f(FAKE, FAKE, 4, 32, FAKE, 4, 4, FAKE, ctypes.c_void_p(0x10004), 0, None) == ERR_ALIGN
    assert f(MIS, FAKE, 4, 32, FAKE, 4, 4, FAKE, FAKE, 0, None) == ERR_ALIGN
    assert f(None, None, 0, 32, None, 4, 4, None, None, 0, None) == OK


def test_residual_and_output_error_argument_errors(lib):
    r = lib.hscale_dequant_residual
    assert r(FAKE, 4, 24, FAKE, FAKE, FAKE, FAKE, 128, None) == ERR_SHAPE       # n % 16
    assert r(FAKE, 4, 80, FAKE, FAKE, FAKE, FAKE, 200, None) == ERR_SHAPE       # ld < 2 * 128
    assert r(FAKE, 4, 64, FAKE, None, FAKE, FAKE, 128, None) == ERR_NULL
    assert r(FAKE, 4, 64, FAKE, FAKE, FAKE, MIS, 128, None) == ERR_ALIGN
    assert r(FAKE, 4, 64, FAKE, FAKE, FAKE, FAKE, 132, None) == ERR_ALIGN       # ld % 8
    assert r(None, 0, 64, None, None, None, None, 0, None) == OK
    ws = lib.hscale_output_error_workspace_bytes
    assert ws(0, 256) == 0 and ws(128, 256) == 256 and ws(129, 257) == 256 and ws(128 * 64, 256 * 40) == 20480
    f = lib.hscale_output_error
    assert f(FAKE, 128, 64, 64, FAKE, 100, 256, FAKE, FAKE, 256, None) == ERR_SHAPE   # ld_dw2 < 128
    assert f(FAKE, 128, 40, 40, FAKE, 128, 256, FAKE, FAKE, 256, None) == ERR_SHAPE   # n % 16
    assert f(FAKE, 128, 64, 64, FAKE, 128, 256, None, FAKE, 256, None) == ERR_NULL
    assert f(FAKE, 128, 64, 64, FAKE, 128, 256, FAKE, FAKE, 8, None) == ERR_WS
    assert f(FAKE, 128, 64, 64, FAKE, 128, 256, FAKE, None, 256, None) == ERR_WS
    assert f(MIS, 128, 64, 64, FAKE, 128, 256, FAKE, FAKE, 256, None) == ERR_ALIGN
    assert f(None, 0, 64, 64, None, 128, 256, None, None, 0, None) == OK


def test_gptq_argument_errors(lib):
    ws = lib.hscale_hessian_full_workspace_bytes
    assert ws(0, 64) == 0 and ws(100, 64) == 13312    # 64 rows of 104 bf16, rounded to 256 B
    f = lib.hscale_hessian_full_accumulate
    assert f(FAKE, 100, 64, 32, FAKE, 64, FAKE, 1 << 20, None) == ERR_SHAPE      # ld_x < n
    assert f(FAKE, 100, 64, 64, None, 64, FAKE, 1 << 20, None) == ERR_NULL
    # X whose rows are not 16-byte aligned (ld_x % 8 != 0) is transposed: a workspace is needed
    assert f(FAKE, 100, 64, 66, FAKE, 64, FAKE, 16, None) == ERR_WS
    assert f(FAKE, 100, 64, 66, FAKE, 64, None, 0, None) == ERR_WS
    assert f(None, 0, 64, 64, None, 64, None, 0, None) == OK
    g = lib.hscale_gptq_factor
    assert g(FAKE, 64, 32, 0.01, FAKE, None, FAKE, FAKE, 1 << 20, None) == ERR_SHAPE   # ld < n
    assert g(FAKE, 64, 64, -1.0, FAKE, None, FAKE, FAKE, 1 << 20, None) == ERR_ARG
    assert g(FAKE, 64, 64, 0.01, None, None, FAKE, FAKE, 1 << 20, None) == ERR_NULL
    assert g(None, 0, 0, 0.01, None, None, None, None, 0, None) == OK
    # the factor's workspace: the 128 x 256 fp32 pair [B | X] (n = 64 pads to one block), the
    # 128 x 128 panel and two 128 x 768 bf16 split operands
    wsf = lib.hscale_gptq_factor_workspace_bytes
    assert wsf(64) == 131072 + 65536 + 2 * 196608
    assert wsf(0) == 0 and wsf(65537) == 0
    assert g(FAKE, 64, 64, 0.01, FAKE, None, FAKE, FAKE, wsf(64) - 256, None) == ERR_WS
    assert g(FAKE, 64, 64, 0.01, FAKE, None, FAKE, None, wsf(64), None) == ERR_WS
    assert g(FAKE, 65537, 65537, 0.01, FAKE, None, FAKE, FAKE, 1 << 20, None) == ERR_SHAPE
    # 4x64 fp32 weights + 4x32 fp32 E + 4x192 and 64x192 bf16 split operands, each rounded to 256 B
    assert lib.hscale_gptq_workspace_bytes(4, 64, 32) == 1024 + 2 * 1536 + 2 * 24576
    q = lib.hscale_gptq_hscale
    assert q(FAKE, 4, 64, FAKE, FAKE, FAKE, None, 24, 4, 4, FAKE, FAKE, FAKE, 1 << 20, None) == ERR_SHAPE
    assert q(FAKE, 4, 64, FAKE, FAKE, FAKE, None, 48, 4, 4, FAKE, FAKE, FAKE, 1 << 20, None) == ERR_SHAPE
    assert q(FAKE, 4, 64, FAKE, FAKE, FAKE, None, 32, -1, 4, FAKE, FAKE, FAKE, 1 << 20, None) == ERR_ARG
    assert q(FAKE, 4, 64, None, FAKE, FAKE, None, 32, 4, 4, FAKE, FAKE, FAKE, 1 << 20, None) == ERR_NULL
    assert q(FAKE, 4, 64, FAKE, FAKE, FAKE, None, 32, 4, 4, FAKE, FAKE, FAKE, 64, None) == ERR_WS
    assert q(None, 0, 64, None, None, None, None, 32, 4, 4, None, None, None, 0, None) == OK


def test_library_sources_load_no_other_library_at_run_time():
    """Every kernel of the path is the library's own: nothing is looked up with dlopen (the
    factor of Algorithm 3 no longer calls a solver library)."""
    csrc = pathlib.Path(hs.__file__).resolve().parent / "csrc"
    for src in csrc.iterdir():
        text = src.read_text()
        for word in ("dlopen", "cusolver", "cublas"):
            assert word not in text.lower(), (src.name, word)


def test_pack_argument_errors(lib):
    f = lib.hscale_pack_nvfp4
    assert f(FAKE, 4, 32, FAKE, None, FAKE, None) == ERR_NULL
    assert f(FAKE, 4, 32, FAKE, FAKE, None, None) == ERR_NULL
    assert f(FAKE, 4, 33, FAKE, FAKE, FAKE, None) == ERR_SHAPE
    assert f(FAKE, 4, 32, FAKE, FAKE, ctypes.c_void_p(0x10004), None) == ERR_ALIGN
    assert f(None, 4, 0, None, None, None, None) == OK


def test_binding_refuses_cpu_tensors(lib):
    import torch
    x = torch.zeros(4, 16, dtype=torch.bfloat16)
    h = torch.zeros(16)
    with pytest.raises(TypeError):
        hs.hscale_hessian_diag_accumulate(x, h)
    w = torch.zeros(4, 512, dtype=torch.bfloat16)
    sg = torch.ones(1)
    codes = torch.zeros(4 * 32, dtype=torch.uint8)
    with pytest.raises(TypeError):   # host tensors, before any call into the library
        hs.hscale_refine_scales_ws(w, None, sg, None, 0, 4, 4, codes, None, 0, torch.zeros(16, dtype=torch.uint8))


def test_build_flags_target_sm103a_only():
    assert build.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]
    assert not any("fast_math" in f or "ftz=true" in f for f in build.NVCC_FLAGS)

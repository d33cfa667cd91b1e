"""C-ABI checks that need no GPU: the library builds and loads, exports every
function include/rowop.h declares, applies the row-length dispatch rule
exactly as the oracle states it, and rejects bad arguments synchronously
(before touching the device)."""
import ctypes
import os
import re

import pytest

from oracle import rowop_oracle as orc

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "rowop.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2607_23089_gb300 import build, rowop
    build.build()
    return rowop


def declared_functions():
    text = open(HEADER).read()
    return re.findall(r"ROWOP_API\s+[\w\s\*]+?\b(rowop_\w+)\s*\(", text)


def test_header_declares_the_abi():
    names = declared_functions()
    for n in ("rowop_softmax", "rowop_logsoftmax", "rowop_layernorm", "rowop_rmsnorm",
              "rowop_softmax_ragged", "rowop_logsoftmax_ragged", "rowop_layernorm_ragged",
              "rowop_rmsnorm_ragged", "rowop_ragged_workspace_size",
              "rowop_select_bucket", "rowop_status_string", "rowop_check_status",
              "rowop_last_cuda_error"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    raw = ctypes.CDLL(lib.LIB_PATH)
    names = declared_functions()
    assert names
    for n in names:
        assert hasattr(raw, n), n
        assert n in lib.SIGNATURES, n


def test_select_bucket_matches_the_rule(lib):
    for dtype, es in ((lib.ROWOP_F32, 4), (lib.ROWOP_BF16, 2)):
        lens = set(range(0, 70)) | {1023, 1024, 1025, 2047, 2048, 2049, 8191, 8192,
                                    8193, 16383, 16384, 16385, 262144, 1 << 22}
        for n in sorted(lens):
            assert lib.rowop_select_bucket(n, dtype) == orc.bucket(n, es), (n, es)
    assert lib.rowop_select_bucket(-1, lib.ROWOP_F32) == -1
    assert lib.rowop_select_bucket(10, 9) == -1


def test_limits_and_strings(lib):
    assert lib.rowop_max_row_len(lib.ROWOP_F32) >= 262144
    assert lib.rowop_max_row_len(lib.ROWOP_BF16) >= 2 * 262144 - 8
    assert lib.rowop_max_row_len(5) == 0
    for code in range(8):
        s = lib.rowop_status_string(code).decode()
        assert s.startswith(lib.STATUS[code])
    assert b"unknown" in lib.rowop_status_string(99)
    assert lib.rowop_ragged_workspace_size(0) >= 256
    n = 16384
    ws = lib.rowop_ragged_workspace_size(n)
    assert ws >= 256 + n + 3 * 4 * n


def test_get_config(lib):
    """rowop_get_config reports the rule rowop_select_bucket applies and the
    limits the entry points enforce."""
    import ctypes as _ct
    cfg = lib.get_config()
    assert cfg["size"] == _ct.sizeof(lib.RowopConfig)
    assert cfg["chunk_bytes"] == 16 and cfg["tile_bytes"] == 1024
    for dtype, es in ((lib.ROWOP_F32, 4), (lib.ROWOP_BF16, 2), (lib.ROWOP_F16, 2)):
        s_el = cfg["small_max_bytes"] // es
        m_el = cfg["medium_max_bytes"] // es
        assert lib.rowop_select_bucket(s_el, dtype) == 0
        assert lib.rowop_select_bucket(s_el + 1, dtype) == 1
        assert lib.rowop_select_bucket(m_el, dtype) == 1
        assert lib.rowop_select_bucket(m_el + 1, dtype) == 2
        assert cfg["max_row_len"][dtype] == lib.rowop_max_row_len(dtype)
    assert cfg["small_max_bytes"] == 4096 and cfg["medium_max_bytes"] == 32768
    assert cfg["max_cluster"] == 16
    assert cfg["resident_max_tiles"] == [64, 32]
    assert cfg["wait_limit_ns"] == 2 * 10**9
    text = open(HEADER).read()
    assert cfg["static_max_rows"] == int(
        re.search(r"#define\s+ROWOP_STATIC_MAX_ROWS\s+(\d+)", text).group(1))
    assert lib.rowop_get_config(None) == lib.ROWOP_ERR_INVALID_ARG


FAKE = 1 << 20  # a non-NULL, 16-byte aligned address that is never touched


def test_dense_validation(lib):
    F32, BF16 = lib.ROWOP_F32, lib.ROWOP_BF16
    sm = lib.rowop_softmax
    assert sm(FAKE, FAKE, 4, 8, 8, 7, None) == lib.ROWOP_ERR_UNSUPPORTED_DTYPE
    assert sm(FAKE, FAKE, -1, 8, 8, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert sm(None, None, 0, 8, 8, F32, None) == lib.ROWOP_OK  # empty batch: no-op
    assert sm(FAKE, FAKE, 4, 0, 8, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert sm(FAKE, FAKE, 4, 8, 7, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert sm(None, FAKE, 4, 8, 8, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert sm(FAKE, None, 4, 8, 8, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert sm(FAKE + 2, FAKE, 4, 8, 8, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert sm(FAKE + 1, FAKE, 4, 8, 8, BF16, None) == lib.ROWOP_ERR_INVALID_ARG
    too_long = lib.rowop_max_row_len(F32) + 1
    assert sm(FAKE, FAKE, 1, too_long, too_long, F32, None) == lib.ROWOP_ERR_TOO_LONG
    assert sm(FAKE, FAKE, 1 << 40, 1 << 30, 1 << 30, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    ln = lib.rowop_layernorm
    assert ln(FAKE, FAKE, None, None, 4, 8, 8, F32, -1.0, None) == lib.ROWOP_ERR_INVALID_ARG
    assert ln(FAKE, FAKE, None, None, 4, 8, 8, F32, float("nan"), None) == lib.ROWOP_ERR_INVALID_ARG
    assert ln(FAKE, FAKE, FAKE + 2, None, 4, 8, 8, F32, 1e-5, None) == lib.ROWOP_ERR_INVALID_ARG
    rms = lib.rowop_rmsnorm
    assert rms(FAKE, FAKE, None, 4, 8, 8, F32, float("inf"), None) == lib.ROWOP_ERR_INVALID_ARG
    assert rms(FAKE, FAKE, None, 0, 8, 8, F32, 1e-6, None) == lib.ROWOP_OK


def test_ragged_validation(lib):
    F32 = lib.ROWOP_F32
    ws_need = lib.rowop_ragged_workspace_size(10)
    r = lib.rowop_softmax_ragged
    assert r(FAKE, FAKE, FAKE, 10, 64, 3, FAKE, ws_need, None) == lib.ROWOP_ERR_UNSUPPORTED_DTYPE
    assert r(FAKE, FAKE, FAKE, -1, 64, F32, FAKE, ws_need, None) == lib.ROWOP_ERR_INVALID_ARG
    assert r(FAKE, FAKE, FAKE, 0, 64, F32, None, 0, None) == lib.ROWOP_OK
    assert r(FAKE, FAKE, FAKE, 10, -1, F32, FAKE, ws_need, None) == lib.ROWOP_ERR_INVALID_ARG
    assert r(FAKE, FAKE, None, 10, 64, F32, FAKE, ws_need, None) == lib.ROWOP_ERR_INVALID_ARG
    assert r(FAKE, FAKE, FAKE + 4, 10, 64, F32, FAKE, ws_need, None) == lib.ROWOP_ERR_INVALID_ARG
    assert r(FAKE, FAKE, FAKE, 10, 64, F32, None, ws_need, None) == lib.ROWOP_ERR_WORKSPACE
    assert r(FAKE, FAKE, FAKE, 10, 64, F32, FAKE + 16, ws_need, None) == lib.ROWOP_ERR_WORKSPACE
    assert r(FAKE, FAKE, FAKE, 10, 64, F32, FAKE, ws_need - 1, None) == lib.ROWOP_ERR_WORKSPACE
    assert r(FAKE, FAKE, FAKE, 1 << 31, 64, F32, FAKE, 1 << 40, None) == lib.ROWOP_ERR_INVALID_ARG
    too_long = lib.rowop_max_row_len(F32) + 1
    assert r(FAKE, FAKE, FAKE, 10, too_long, F32, FAKE, ws_need, None) == lib.ROWOP_ERR_TOO_LONG
    ln = lib.rowop_layernorm_ragged
    assert ln(FAKE, FAKE, None, None, FAKE, 10, 64, F32, -0.5, FAKE, ws_need,
              None) == lib.ROWOP_ERR_INVALID_ARG


def test_static_ragged_validation_order(lib):
    """The library-workspace ragged LayerNorm reports argument errors exactly
    as the caller-workspace call does, before its row limit: only an
    otherwise valid call is refused for having too many rows."""
    import re as _re
    text = open(HEADER).read()
    nmax = int(_re.search(r"#define\s+ROWOP_STATIC_MAX_ROWS\s+(\d+)", text).group(1))
    F32 = lib.ROWOP_F32
    st = lib.rowop_layernorm_ragged_static
    big = nmax + 1
    assert st(FAKE, FAKE, None, None, FAKE, big, 64, 9, 1e-5, None) == \
        lib.ROWOP_ERR_UNSUPPORTED_DTYPE
    assert st(FAKE, FAKE, None, None, None, big, 64, F32, 1e-5, None) == lib.ROWOP_ERR_INVALID_ARG
    assert st(FAKE, FAKE, None, None, FAKE, big, 64, F32, -1.0, None) == lib.ROWOP_ERR_INVALID_ARG
    assert st(FAKE, None, None, None, FAKE, big, 64, F32, 1e-5, None) == lib.ROWOP_ERR_INVALID_ARG
    too_long = lib.rowop_max_row_len(F32) + 1
    assert st(FAKE, FAKE, None, None, FAKE, big, too_long, F32, 1e-5, None) == \
        lib.ROWOP_ERR_TOO_LONG
    assert st(FAKE, FAKE, None, None, FAKE, big, 64, F32, 1e-5, None) == lib.ROWOP_ERR_WORKSPACE
    assert st(None, None, None, None, None, 0, 64, F32, 1e-5, None) == lib.ROWOP_OK


def test_debug_timeout_rejects_bad_limits(lib):
    assert lib.rowop_debug_wait_timeout(0, None) == lib.ROWOP_ERR_INVALID_ARG
    assert lib.rowop_debug_wait_timeout(2 * 10**9, None) == lib.ROWOP_ERR_INVALID_ARG


def test_binding_refuses_cpu_tensors(lib):
    import torch
    with pytest.raises(ValueError):
        lib.softmax(torch.zeros(4, 8))


def test_pad_and_moe_validation(lib):
    """Bad shapes are refused before anything touches the device."""
    F32 = lib.ROWOP_F32
    assert lib.rowop_pad_scale(None, None, 0, 4, 8, 4, 8, 1.0, F32, None) == lib.ROWOP_OK
    assert lib.rowop_pad_scale(None, None, 4, 9, 8, 9, 8, 1.0, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert lib.rowop_pad_scale(None, None, 4, 4, 8, 4, 8, 1.0, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert lib.rowop_pad_scale(16, 16, 4, 4, 8, 3, 8, 1.0, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert lib.rowop_pad_scale(16, 16, 4, 4, 8, 4, 8, float("nan"), F32, None) == \
        lib.ROWOP_ERR_INVALID_ARG
    assert lib.rowop_pad_scale(16, 16, 4, 4, 8, 4, 8, 1.0, 7, None) == \
        lib.ROWOP_ERR_UNSUPPORTED_DTYPE
    assert lib.rowop_moe_group_top2(16, 16, 0, 64, 64, F32, None) == lib.ROWOP_OK
    assert lib.rowop_moe_group_top2(16, 16, 4, 48, 48, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert lib.rowop_moe_group_top2(16, 16, 4, 64, 32, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert lib.rowop_moe_group_top2(None, 16, 4, 64, 64, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert lib.rowop_moe_group_top2(16, 18, 4, 64, 64, F32, None) == lib.ROWOP_ERR_INVALID_ARG


def test_backward_validation(lib):
    """Backward entry points: bad arguments are refused before the device is
    touched (the workspace size needs the device, so it is not checked
    here)."""
    F32, BF16 = lib.ROWOP_F32, lib.ROWOP_BF16
    sb = lib.rowop_softmax_backward
    assert sb(FAKE, FAKE, FAKE, 4, 8, 8, 7, None) == lib.ROWOP_ERR_UNSUPPORTED_DTYPE
    assert sb(FAKE, FAKE, FAKE, -1, 8, 8, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert sb(None, None, None, 0, 8, 8, F32, None) == lib.ROWOP_OK
    assert sb(FAKE, FAKE, FAKE, 4, 0, 8, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert sb(FAKE, FAKE, FAKE, 4, 8, 7, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert sb(FAKE, None, FAKE, 4, 8, 8, F32, None) == lib.ROWOP_ERR_INVALID_ARG
    assert sb(FAKE, FAKE, FAKE + 1, 4, 8, 8, BF16, None) == lib.ROWOP_ERR_INVALID_ARG
    assert sb(FAKE, FAKE, FAKE, 1, 262145, 262145, F32, None) == lib.ROWOP_ERR_TOO_LONG
    ls = lib.rowop_logsoftmax_backward
    assert ls(FAKE, FAKE, FAKE, 2, 8, 8, F32 + 9, None) == lib.ROWOP_ERR_UNSUPPORTED_DTYPE
    ln = lib.rowop_layernorm_backward
    assert ln(FAKE, FAKE, None, FAKE, None, None, 4, 8, 8, F32, -1.0, None, 0,
              None) == lib.ROWOP_ERR_INVALID_ARG
    assert ln(FAKE, FAKE, FAKE + 2, FAKE, None, None, 4, 8, 8, F32, 1e-5, None, 0,
              None) == lib.ROWOP_ERR_INVALID_ARG
    assert ln(FAKE, FAKE, None, FAKE, FAKE + 1, None, 4, 8, 8, BF16, 1e-5, None, 0,
              None) == lib.ROWOP_ERR_INVALID_ARG
    assert ln(None, None, None, None, None, None, 0, 0, 0, F32, 1e-5, None, 0,
              None) == lib.ROWOP_OK  # no rows, no parameter gradients: a no-op
    assert ln(None, None, None, None, FAKE, None, 0, 0, 0, F32, 1e-5, None, 0,
              None) == lib.ROWOP_ERR_INVALID_ARG  # zeros of dgamma need cols
    assert ln(FAKE, FAKE, None, FAKE, None, None, 1, 262145, 262145, F32, 1e-5, None, 0,
              None) == lib.ROWOP_ERR_TOO_LONG
    rms = lib.rowop_rmsnorm_backward
    assert rms(FAKE, FAKE, None, FAKE, None, 4, 8, 8, F32, float("nan"), None, 0,
               None) == lib.ROWOP_ERR_INVALID_ARG
    assert rms(FAKE, FAKE, None, None, None, 4, 8, 8, F32, 1e-6, None, 0,
               None) == lib.ROWOP_ERR_INVALID_ARG
    assert lib.rowop_layernorm_backward_workspace_size(0) == 0
    assert lib.rowop_rmsnorm_backward_workspace_size(-5) == 0


def test_backward_ragged_norm_validation(lib):
    """Argument checks of the ragged norm backward calls that come before any
    device query (this host has no GPU)."""
    F32, BF16 = lib.ROWOP_F32, lib.ROWOP_BF16
    ln = lib.rowop_layernorm_backward_ragged
    rms = lib.rowop_rmsnorm_backward_ragged
    plan = lib.rowop_ragged_workspace_size(10)
    # x, dy, gamma, dx, dgamma, dbeta, offsets, rows, max_len, dtype, eps, ws, ws_bytes, stream
    assert ln(FAKE, FAKE, None, FAKE, FAKE, FAKE, FAKE, 10, 64, 7, 1e-5, FAKE, plan,
              None) == lib.ROWOP_ERR_UNSUPPORTED_DTYPE
    assert ln(FAKE, FAKE, None, FAKE, FAKE, FAKE, FAKE, -1, 64, F32, 1e-5, FAKE, plan,
              None) == lib.ROWOP_ERR_INVALID_ARG
    assert ln(FAKE, FAKE, None, FAKE, FAKE, FAKE, FAKE, 10, -1, F32, 1e-5, FAKE, plan,
              None) == lib.ROWOP_ERR_INVALID_ARG
    assert ln(FAKE, FAKE, None, FAKE, FAKE, FAKE, FAKE, 10, 64, F32, -1.0, FAKE, plan,
              None) == lib.ROWOP_ERR_INVALID_ARG
    # nothing to do: no rows and no parameter gradients (or none of any length)
    assert ln(None, None, None, None, None, None, None, 0, 64, F32, 1e-5, None, 0,
              None) == lib.ROWOP_OK
    assert ln(None, None, None, None, FAKE, FAKE, None, 0, 0, F32, 1e-5, None, 0,
              None) == lib.ROWOP_OK
    # rows, or dgamma / dbeta to zero, need their pointers and a workspace
    assert ln(FAKE, FAKE, None, FAKE, FAKE, FAKE, None, 10, 64, F32, 1e-5, FAKE, plan,
              None) == lib.ROWOP_ERR_INVALID_ARG
    assert ln(FAKE, None, None, FAKE, None, None, FAKE, 10, 64, F32, 1e-5, FAKE, plan,
              None) == lib.ROWOP_ERR_INVALID_ARG
    assert ln(FAKE + 1, FAKE, None, FAKE, None, None, FAKE, 10, 64, BF16, 1e-5, FAKE, plan,
              None) == lib.ROWOP_ERR_INVALID_ARG
    assert ln(FAKE, FAKE, FAKE + 2, FAKE, None, None, FAKE, 10, 64, F32, 1e-5, FAKE, plan,
              None) == lib.ROWOP_ERR_INVALID_ARG
    assert ln(FAKE, FAKE, None, FAKE, FAKE + 1, None, FAKE, 10, 64, BF16, 1e-5, FAKE, plan,
              None) == lib.ROWOP_ERR_INVALID_ARG
    assert ln(FAKE, FAKE, None, FAKE, FAKE, FAKE, FAKE, 10, 262145, F32, 1e-5, FAKE, plan,
              None) == lib.ROWOP_ERR_TOO_LONG
    assert ln(FAKE, FAKE, None, FAKE, FAKE, FAKE, FAKE, 10, 64, F32, 1e-5, FAKE, plan - 1,
              None) == lib.ROWOP_ERR_WORKSPACE
    assert ln(FAKE, FAKE, None, FAKE, FAKE, FAKE, FAKE, 10, 64, F32, 1e-5, FAKE + 16, plan,
              None) == lib.ROWOP_ERR_WORKSPACE
    assert ln(None, None, None, None, FAKE, FAKE, None, 0, 64, F32, 1e-5, None, 0,
              None) == lib.ROWOP_ERR_WORKSPACE
    # x, dy, gamma, dx, dgamma, offsets, rows, max_len, dtype, eps, ws, ws_bytes, stream
    assert rms(FAKE, FAKE, None, FAKE, FAKE, FAKE, 10, 64, 9, 1e-6, FAKE, plan,
               None) == lib.ROWOP_ERR_UNSUPPORTED_DTYPE
    assert rms(FAKE, FAKE, None, FAKE, FAKE, None, 10, 64, F32, 1e-6, FAKE, plan,
               None) == lib.ROWOP_ERR_INVALID_ARG
    assert rms(FAKE, FAKE, None, FAKE, FAKE, FAKE, 10, 300000, F32, 1e-6, FAKE, plan,
               None) == lib.ROWOP_ERR_TOO_LONG
    # one team holds at most 131072 elements of a ragged norm row
    for dtype in (F32, BF16):
        assert ln(FAKE, FAKE, None, FAKE, FAKE, FAKE, FAKE, 10, 131073, dtype, 1e-5, FAKE, plan,
                  None) == lib.ROWOP_ERR_TOO_LONG
        assert ln(FAKE, FAKE, None, FAKE, FAKE, FAKE, FAKE, 10, 131072, dtype, 1e-5, FAKE,
                  plan - 1, None) == lib.ROWOP_ERR_WORKSPACE
    assert rms(FAKE, FAKE, None, FAKE, FAKE, FAKE, 10, 64, F32, 1e-6, None, plan,
               None) == lib.ROWOP_ERR_WORKSPACE
    # the size queries reject bad arguments without a device
    assert lib.rowop_layernorm_backward_ragged_workspace_size(-1, 64, F32) == 0
    assert lib.rowop_rmsnorm_backward_ragged_workspace_size(10, -1, F32) == 0
    assert lib.rowop_rmsnorm_backward_ragged_workspace_size(10, 64, 7) == 0


def test_backward_ragged_validation(lib):
    F32 = lib.ROWOP_F32
    f = lib.rowop_softmax_backward_ragged
    ws_need = lib.rowop_ragged_workspace_size(10)
    assert f(FAKE, FAKE, FAKE, FAKE, 10, 64, 7, FAKE, ws_need, None) == lib.ROWOP_ERR_UNSUPPORTED_DTYPE
    assert f(FAKE, FAKE, FAKE, FAKE, -1, 64, F32, FAKE, ws_need, None) == lib.ROWOP_ERR_INVALID_ARG
    assert f(None, None, None, None, 0, 64, F32, None, 0, None) == lib.ROWOP_OK
    assert f(FAKE, FAKE, FAKE, None, 10, 64, F32, FAKE, ws_need, None) == lib.ROWOP_ERR_INVALID_ARG
    assert f(FAKE, None, FAKE, FAKE, 10, 64, F32, FAKE, ws_need, None) == lib.ROWOP_ERR_INVALID_ARG
    assert f(FAKE, FAKE, FAKE, FAKE, 10, 262145, F32, FAKE, ws_need, None) == lib.ROWOP_ERR_TOO_LONG
    assert f(FAKE, FAKE, FAKE, FAKE, 10, 64, F32, FAKE, ws_need - 1, None) == lib.ROWOP_ERR_WORKSPACE
    g = lib.rowop_logsoftmax_backward_ragged
    assert g(FAKE, FAKE, FAKE, FAKE, 10, -1, F32, FAKE, ws_need, None) == lib.ROWOP_ERR_INVALID_ARG


C_CLIENT = r"""
#include <stdio.h>
#include <string.h>
#include "rowop.h"

/* A plain C99 client of the ABI: only calls that need no device. */
int main(void) {
    if (rowop_select_bucket(1024, ROWOP_F32) != ROWOP_SMALL) return 1;
    if (rowop_select_bucket(1025, ROWOP_F32) != ROWOP_MEDIUM) return 2;
    if (rowop_select_bucket(16385, ROWOP_BF16) != ROWOP_LARGE) return 3;
    if (rowop_max_row_len(ROWOP_BF16) < 2 * (int64_t)262144 - 8) return 4;
    if (strlen(rowop_status_string(ROWOP_ERR_TOO_LONG)) == 0) return 5;
    if (rowop_softmax(NULL, NULL, -1, 8, 8, ROWOP_F32, NULL) != ROWOP_ERR_INVALID_ARG) return 6;
    if (rowop_layernorm(NULL, NULL, NULL, NULL, 4, 8, 8, (rowop_dtype_t)9, 1e-5f, NULL) !=
        ROWOP_ERR_UNSUPPORTED_DTYPE)
        return 7;
    if (rowop_softmax(NULL, NULL, 0, 8, 8, ROWOP_F32, NULL) != ROWOP_OK) return 8;
    puts("ok");
    return 0;
}
"""


def test_plain_c_client(tmp_path, lib):
    """include/rowop.h compiles as strict C99 and a C program links
    librowop.so and gets the documented answers from the device-free calls."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "client.c"
    src.write_text(C_CLIENT)
    exe = tmp_path / "client"
    libdir = os.path.dirname(lib.LIB_PATH)
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I", inc,
                    str(src), "-o", str(exe), "-L", libdir, "-l:librowop.so",
                    f"-Wl,-rpath,{libdir}"], check=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0 and r.stdout.strip() == "ok", (r.returncode, r.stdout, r.stderr)

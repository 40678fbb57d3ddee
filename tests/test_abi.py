"""The C ABI library builds, loads and exports every symbol include/*.h declares.

CPU only: no call here launches GPU work.  Struct layouts of the ctypes binding are
checked against a C compiler's view of include/dkv.h.
"""
import ctypes
import glob
import os
import re
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = sorted(glob.glob(os.path.join(ROOT, "include", "*.h")))


def _built_lib():
    from paper_2608_27922_gb300 import build as B
    if not os.path.exists(B.LIB):
        if not (shutil.which("nvcc") or os.path.exists("/usr/local/cuda/bin/nvcc")):
            pytest.skip("nvcc unavailable and the library is not built")
        B.build()
    from paper_2608_27922_gb300 import dkv
    return dkv


def _declared_functions():
    names = set()
    for h in HEADERS:
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"^[A-Za-z_][\w\s\*]*?\b(dkv_\w+)\s*\(", text, flags=re.M):
            names.add(m.group(1))
    return names


def test_header_declares_the_hot_path():
    names = _declared_functions()
    for required in ("dkv_bank_create", "dkv_bank_admit", "dkv_bank_compress", "dkv_bank_evict",
                     "dkv_bank_commit", "dkv_bank_attend", "dkv_bank_destroy", "dkv_bank_workspace_size"):
        assert required in names


def test_every_declared_symbol_is_exported():
    dkv = _built_lib()
    L = dkv.lib()
    declared = _declared_functions()
    missing = [n for n in sorted(declared) if not hasattr(L, n)]
    assert not missing, missing
    bound = {n for n, _, _ in dkv.SIGNATURES}
    assert declared <= bound, sorted(declared - bound)


def test_struct_layouts_match_c():
    dkv = _built_lib()
    if not shutil.which("gcc"):
        pytest.skip("gcc unavailable")
    src = r"""
#include <stdio.h>
#include <stddef.h>
#include "dkv.h"
int main(void) {
  printf("%zu %zu %zu %zu %zu %zu %zu %zu %zu %zu %zu\n", sizeof(dkv_params_t), sizeof(dkv_buffers_t),
         sizeof(dkv_layer_stats_t), sizeof(dkv_head_stats_t), sizeof(dkv_intermediates_t),
         offsetof(dkv_buffers_t, workspace_bytes), offsetof(dkv_params_t, order), offsetof(dkv_params_t, eviction),
         offsetof(dkv_params_t, refresh_baselines), offsetof(dkv_params_t, layer_heads),
         offsetof(dkv_params_t, descriptor));
  return 0;
}
"""
    tmp = os.path.join(ROOT, "tests", "_abi_layout_probe")
    with open(tmp + ".c", "w") as f:
        f.write(src)
    try:
        subprocess.check_call(["gcc", "-I", os.path.join(ROOT, "include"), tmp + ".c", "-o", tmp])
        out = subprocess.check_output([tmp]).decode().split()
    finally:
        for p in (tmp + ".c", tmp):
            if os.path.exists(p):
                os.remove(p)
    sizes = [int(x) for x in out]
    assert sizes == [ctypes.sizeof(dkv.dkv_params_t), ctypes.sizeof(dkv.dkv_buffers_t),
                     ctypes.sizeof(dkv.dkv_layer_stats_t), ctypes.sizeof(dkv.dkv_head_stats_t),
                     ctypes.sizeof(dkv.dkv_intermediates_t), dkv.dkv_buffers_t.workspace_bytes.offset,
                     dkv.dkv_params_t.order.offset, dkv.dkv_params_t.eviction.offset,
                     dkv.dkv_params_t.refresh_baselines.offset, dkv.dkv_params_t.layer_heads.offset,
                     dkv.dkv_params_t.descriptor.offset]


def test_host_only_entry_points():
    dkv = _built_lib()
    L = dkv.lib()
    for s in range(9):
        assert L.dkv_status_str(s)
    assert dkv.dkv_version() >= 100
    p = dkv.dkv_params_default(128)
    assert (p.tau, p.sigma, p.p, p.eps, p.sync_heads) == (2.0, 8.0, 2.0, 1.0, 1)
    assert abs(p.delta - 1e-6) < 1e-12
    assert dkv.dkv_params_default(64).sigma == pytest.approx(32 ** 0.5)
    # workspace size: positive for valid shapes, zero for invalid ones
    assert dkv.dkv_bank_workspace_size(12, 128, [9360] * 12, 4680, dkv.DKV_DTYPE_BF16) > 0
    assert dkv.dkv_bank_workspace_size(12, 96, [9360] * 12, 4680, dkv.DKV_DTYPE_BF16) == 0
    assert dkv.dkv_bank_workspace_size(2, 64, [0, 5], 16, dkv.DKV_DTYPE_FP32) == 0
    assert dkv.dkv_bank_workspace_size(2, 64, [5, 5], 1 << 20, dkv.DKV_DTYPE_FP32) == 0
    # the [K; V] descriptor adds the value copies: H (n_max + M_max + n_max) d elements
    p = dkv.dkv_params_default(128)
    base = dkv.dkv_bank_workspace_size(12, 128, [9360] * 12, 4680, dkv.DKV_DTYPE_BF16, p)
    assert base == dkv.dkv_bank_workspace_size(12, 128, [9360] * 12, 4680, dkv.DKV_DTYPE_BF16)
    p.descriptor = dkv.DKV_DESC_KV
    kv = dkv.dkv_bank_workspace_size(12, 128, [9360] * 12, 4680, dkv.DKV_DTYPE_BF16, p)
    assert 0 <= kv - base - 12 * (4680 + 9360 + 4680) * 128 * 2 < 3 * 256
    p.descriptor = 2
    assert dkv.dkv_bank_workspace_size(12, 128, [9360] * 12, 4680, dkv.DKV_DTYPE_BF16, p) == 0
    # argument errors are reported before any CUDA call
    h = ctypes.c_void_p()
    assert L.dkv_bank_create(ctypes.byref(h), 2, 64, None, 16, 1, None, None) == 1
    assert L.dkv_bank_admit(None, None, None, 1, 0, None) == 1
    assert L.dkv_bank_admit_rope(None, None, None, 1, 0, None, None, 0, None) == 1
    assert L.dkv_bank_compress(None, None) == 1
    assert L.dkv_bank_evict(None, None) == 1
    assert L.dkv_bank_commit(None, None) == 1
    assert L.dkv_bank_attend(None, None, 1, None, None, 0, None, None) == 1
    assert L.dkv_bank_sync(None) == 1
    L.dkv_bank_destroy(None)


def test_every_entry_point_rejects_a_missing_handle():
    """Argument errors come back as DKV_ERR_ARG before any CUDA call, so they need no GPU:
    every call that takes a handle, with none."""
    L = _built_lib().lib()
    for name, args in [("export", (None, None)), ("import", (None, None, None)), ("stats", (None, None, None)),
                       ("occupancy", (None, None)), ("intermediates", (None, None)), ("set_timing", (None, 1)),
                       ("kernel_times", (None, 0, None, None, None, None)), ("reset", (None, None)),
                       ("update_sequential", (None, None, None, 1, 0, None, 0, None))]:
        assert getattr(L, "dkv_bank_" + name)(*args) == 1, name
    assert L.dkv_params_default(None, 128) == 1
    assert L.dkv_candidate_order_noalloc(None, None, 1, None, 1, 128, 0, None, None, None, None) == 1
    # scratch of the sequential update: zero for an unsupported head size
    assert L.dkv_sequential_scratch_size(2, 96, 16, 0) == 0
    assert L.dkv_sequential_scratch_size(2, 128, 16, 0) > 0


def test_binding_has_no_fallback(monkeypatch):
    from paper_2608_27922_gb300 import dkv
    monkeypatch.setattr(dkv, "LIB_PATH", "/nonexistent/libdkv.so")
    monkeypatch.setattr(dkv, "_LIB", None)
    with pytest.raises(RuntimeError):
        dkv.lib()


def test_plain_c_program_links_and_calls_the_library():
    """A C program that includes dkv.h and links libdkv.so: the host-only calls and the
    argument errors behave as documented, with no Python in between."""
    dkv = _built_lib()
    if not shutil.which("gcc"):
        pytest.skip("gcc unavailable")
    from paper_2608_27922_gb300 import build as B
    src = r"""
#include <stdio.h>
#include <string.h>
#include "dkv.h"
int main(void) {
  dkv_params_t p;
  if (dkv_params_default(&p, 128) != DKV_OK || p.tau != 2.0f || p.sigma != 8.0f || p.descriptor != DKV_DESC_K)
    return 1;
  int32_t budgets[12];
  for (int h = 0; h < 12; ++h) budgets[h] = 9360;
  size_t a = dkv_bank_workspace_size(12, 128, budgets, 4680, DKV_DTYPE_BF16);
  size_t b = dkv_bank_workspace_size_ex(12, 128, budgets, 4680, DKV_DTYPE_BF16, &p);
  p.descriptor = DKV_DESC_KV;
  size_t c = dkv_bank_workspace_size_ex(12, 128, budgets, 4680, DKV_DTYPE_BF16, &p);
  if (a == 0 || a != b || c <= a) return 2;
  if (dkv_bank_workspace_size(12, 96, budgets, 4680, DKV_DTYPE_BF16) != 0) return 3;
  if (dkv_bank_admit(NULL, NULL, NULL, 1, 0, NULL) != DKV_ERR_ARG) return 4;
  if (dkv_bank_admit_rope(NULL, NULL, NULL, 1, 0, NULL, NULL, DKV_ROPE_HALF, NULL) != DKV_ERR_ARG) return 5;
  if (dkv_bank_compress(NULL, NULL) != DKV_ERR_ARG || dkv_bank_sync(NULL) != DKV_ERR_ARG) return 6;
  if (strlen(dkv_status_str(DKV_ERR_TIMEOUT)) == 0 || dkv_version() < 100) return 7;
  dkv_bank_destroy(NULL);
  printf("%d %zu\n", dkv_version(), a);
  return 0;
}
"""
    tmp = os.path.join(ROOT, "tests", "_abi_c_probe")
    with open(tmp + ".c", "w") as f:
        f.write(src)
    try:
        subprocess.check_call(["gcc", "-I", os.path.join(ROOT, "include"), tmp + ".c", "-o", tmp,
                               "-L", B.LIBDIR, "-ldkv", "-Wl,-rpath," + B.LIBDIR])
        out = subprocess.run([tmp], capture_output=True, text=True)
    finally:
        for p in (tmp + ".c", tmp):
            if os.path.exists(p):
                os.remove(p)
    assert out.returncode == 0, (out.returncode, out.stderr)
    ver, ws = out.stdout.split()
    assert int(ver) == dkv.dkv_version() and int(ws) == dkv.dkv_bank_workspace_size(12, 128, [9360] * 12, 4680,
                                                                                       dkv.DKV_DTYPE_BF16)

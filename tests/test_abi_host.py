"""Host-side checks of the C ABI: the library builds and loads without a GPU,
exports every symbol include/saki.h declares, the ctypes structs match the C
layout, and invalid arguments are rejected before any device work."""
import ctypes
import os
import re
import subprocess
import tempfile

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "saki.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2608_03228_gb300 import _build
    if not os.path.exists(_build.LIB):
        _build.build()
    from paper_2608_03228_gb300 import saki
    return saki


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"SAKI_API\s+[\w\s\*]+?\b(saki_\w+)\s*\(", text)))


def test_header_declares_the_four_path_calls():
    syms = declared_symbols()
    for s in ("saki_fit", "saki_build_index", "saki_score_topk", "saki_recall"):
        assert s in syms


def test_every_declared_symbol_is_exported(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", lib.library_path()], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (saki_\w+)", out))
    missing = [s for s in declared_symbols() if s not in exported]
    assert not missing, missing
    for s in declared_symbols():
        assert hasattr(lib._lib, s)


def test_ctypes_layout_matches_c(lib, tmp_path):
    src = tmp_path / "layout.c"
    src.write_text('#include <stdio.h>\n#include <stddef.h>\n#include "saki.h"\nint main(void){'
                   'printf("%zu %zu %zu %zu %zu\\n", sizeof(saki_config), offsetof(saki_config, eig_floor_rel),'
                   ' offsetof(saki_config, flags), sizeof(saki_layout), offsetof(saki_layout, q_visible));'
                   'printf("%zu\\n", offsetof(saki_config, method));return 0;}')
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    vals = [int(v) for v in subprocess.run([str(exe)], capture_output=True, text=True).stdout.split()]
    assert vals == [ctypes.sizeof(lib.Config), lib.Config.eig_floor_rel.offset, lib.Config.flags.offset,
                    ctypes.sizeof(lib.Layout), lib.Layout.q_visible.offset, lib.Config.method.offset]


def test_status_and_stall_hook_argument_checks(lib):
    assert lib._lib.saki_workspace_status(None, None) == 1      # no workspace: rejected before any CUDA call
    for kind in (4, 6, 99, -1):                                # only the tensor-core kernels with a producer
        assert lib._lib.saki_debug_inject_stall(kind) == 1
    assert lib._lib.saki_debug_inject_stall(0) == 0            # disarm


def test_status_strings(lib):
    for code in range(8):
        assert lib.saki_status_string(code)
    assert lib.saki_version().count(".") == 2


FAKE = 1 << 20   # aligned, never dereferenced: every call below fails before any device work


def _cfg(lib, **kw):
    base = dict(num_q_heads=8, num_kv_heads=2, rank=32, topk=64, dtype="bf16")
    base.update(kw)
    return lib.make_config(**base)


@pytest.mark.parametrize("kw,code", [
    (dict(num_kv_heads=3), 1), (dict(rank=0), 1), (dict(rank=129), 1), (dict(topk=0), 1), (dict(topk=129), 2),
    (dict(head_dim=64), 2), (dict(dtype=7), 1), (dict(center=2), 1), (dict(eig_floor_rel=-1.0), 1),
    (dict(max_sweeps=-1), 1), (dict(flags=64), 1), (dict(flags=8), 1), (dict(method=5), 1), (dict(method=-1), 1),
])
def test_config_validation(lib, kw, code):
    cfg = _cfg(lib, **kw)
    st = lib._lib.saki_fit(ctypes.byref(cfg), 16, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None, None, None, FAKE,
                           1 << 40, None)
    assert st == code
    assert lib.saki_workspace_size(cfg, lib.SAKI_OP_FIT, n_calib=16) == 0


def test_fit_argument_checks(lib):
    cfg = _cfg(lib)
    call = lambda *p: lib._lib.saki_fit(ctypes.byref(cfg), *p)
    assert call(16, None, FAKE, FAKE, FAKE, FAKE, None, None, None, None, FAKE, 1 << 40, None) == 1
    assert call(0, FAKE, FAKE, FAKE, FAKE, FAKE, None, None, None, None, FAKE, 1 << 40, None) == 1
    assert call(16, FAKE + 2, FAKE, FAKE, FAKE, FAKE, None, None, None, None, FAKE, 1 << 40, None) == 1
    need = lib.saki_workspace_size(cfg, lib.SAKI_OP_FIT, n_calib=16)
    assert need >= 10 * 128 * 128 * 4 * 3
    assert call(16, FAKE, FAKE, FAKE, FAKE, FAKE, None, None, None, None, FAKE, need - 1, None) == 6
    cfg.center = 1   # centered keys need the mu output
    assert call(16, FAKE, FAKE, FAKE, FAKE, FAKE, None, None, None, None, FAKE, need, None) == 1


def _layout(lib, lens, q_seq, q_vis):
    off = np.zeros(len(lens) + 1, np.int64)
    off[1:] = np.cumsum(lens)
    return lib.HostLayout(off, q_seq, q_vis)


def test_layout_validation(lib):
    cfg = _cfg(lib)
    good = _layout(lib, [100, 50], [0, 0, 1], [100, 3, 50])
    assert lib.saki_workspace_size(cfg, lib.SAKI_OP_SCORE_TOPK, good) > 0
    for lay in (_layout(lib, [100], [1], [5]),          # sequence id out of range
                _layout(lib, [100], [0], [101]),        # sees more keys than its sequence holds
                _layout(lib, [100], [0], [-1])):
        assert lib.saki_workspace_size(cfg, lib.SAKI_OP_SCORE_TOPK, lay) == 0
        st = lib._lib.saki_score_topk(ctypes.byref(cfg), ctypes.byref(lay.c), FAKE, FAKE, FAKE, None, FAKE, None,
                                      FAKE, 1 << 40, None)
        assert st == 1
    st = lib._lib.saki_score_topk(ctypes.byref(cfg), ctypes.byref(good.c), FAKE, FAKE, FAKE, None, FAKE, None, FAKE,
                                  16, None)
    assert st == 6
    st = lib._lib.saki_recall(ctypes.byref(cfg), ctypes.byref(good.c), 65, FAKE, FAKE, FAKE, FAKE, None, None,
                              FAKE, 1 << 40, None)
    assert st == 1   # recall output missing


def test_workspace_grows_with_splits(lib):
    """A long decode sequence is split across CTAs; the split lists need room."""
    cfg = _cfg(lib, num_q_heads=32, num_kv_heads=8)
    short = _layout(lib, [4096], [0] * 8, [4096] * 8)
    long_ = _layout(lib, [1 << 20], [0] * 8, [1 << 20] * 8)
    assert lib.saki_workspace_size(cfg, lib.SAKI_OP_SCORE_TOPK, long_) > \
        lib.saki_workspace_size(cfg, lib.SAKI_OP_SCORE_TOPK, short)


def test_key_pca_fit_needs_more_workspace(lib):
    """Key PCA folds A into L after the fit: its workspace holds an identity
    operator per head and sigma; the SAKI fit does not pay for that."""
    saki = lib.saki_workspace_size(_cfg(lib), lib.SAKI_OP_FIT, n_calib=16)
    pca = lib.saki_workspace_size(_cfg(lib, method="key_pca"), lib.SAKI_OP_FIT, n_calib=16)
    wsvd = lib.saki_workspace_size(_cfg(lib, method="weight_svd"), lib.SAKI_OP_FIT, n_calib=16)
    assert wsvd == saki
    assert pca >= saki + 8 * 128 * 128 * 4


def test_seeded_decode_reserves_the_sample_pass(lib):
    """A bf16 decode group cut into eight or more splits runs the tensor-core
    kernel with a sample pass first: its plan adds the sample lists and a seed
    per row.  fp32 groups (CUDA-core kernel) and short sequences (fewer splits)
    are not seeded, so the same layout needs less workspace there."""
    lay = _layout(lib, [1 << 20], [0] * 8, [1 << 20] * 8)
    bf = lib.saki_workspace_size(_cfg(lib, num_q_heads=32, num_kv_heads=8), lib.SAKI_OP_SCORE_TOPK, lay)
    f32 = lib.saki_workspace_size(_cfg(lib, num_q_heads=32, num_kv_heads=8, dtype="f32"), lib.SAKI_OP_SCORE_TOPK,
                                  lay)
    # 38 splits x 8 rows of 64 keys per head for the sample lists, plus a seed per row
    assert bf - f32 >= 32 * 38 * 8 * 64 * 8 + 32 * 8 * 8
    short = _layout(lib, [9000], [0] * 8, [9000] * 8)
    assert lib.saki_workspace_size(_cfg(lib, num_q_heads=32, num_kv_heads=8), lib.SAKI_OP_SCORE_TOPK, short) == \
        lib.saki_workspace_size(_cfg(lib, num_q_heads=32, num_kv_heads=8, dtype="f32"), lib.SAKI_OP_SCORE_TOPK, short)
    # groups of fewer than four queries take the CUDA-core kernel: no sample pass
    one = _layout(lib, [1 << 20], [0], [1 << 20])
    assert lib.saki_workspace_size(_cfg(lib, num_q_heads=32, num_kv_heads=8), lib.SAKI_OP_SCORE_TOPK, one) == \
        lib.saki_workspace_size(_cfg(lib, num_q_heads=32, num_kv_heads=8, dtype="f32"), lib.SAKI_OP_SCORE_TOPK, one)


def test_build_index_argument_checks(lib):
    cfg = _cfg(lib)   # bf16, uncentered, r = 32, groups of 4: the tensor-core build
    call = lambda n, mu, sk, ws, nb: lib._lib.saki_build_index(ctypes.byref(cfg), n, FAKE, FAKE, mu, sk, ws, nb, None)
    need = lib.saki_workspace_size(cfg, lib.SAKI_OP_BUILD_INDEX, total_keys=100)
    assert need > 256
    assert call(100, None, None, FAKE, need) == 1        # no sketch
    assert call(-1, None, FAKE, FAKE, need) == 1         # negative key count
    assert call(100, None, FAKE, None, 0) == 1           # the tensor-core path needs its workspace
    assert call(100, None, FAKE, FAKE, need - 1) == 6
    cfg.center = 1
    assert call(100, None, FAKE, FAKE, need) == 1        # centered keys need mu


def test_selection_layout_and_size_limits(lib):
    cfg = _cfg(lib)
    call = lambda lay, ws=FAKE: lib._lib.saki_score_topk(ctypes.byref(cfg), ctypes.byref(lay.c), FAKE, FAKE, FAKE,
                                                         None, FAKE, None, ws, 1 << 40, None)
    bad_start = lib.HostLayout(np.array([5, 100], np.int64), [0], [3])
    decreasing = lib.HostLayout(np.array([0, 100, 50], np.int64), [0], [3])
    for lay in (bad_start, decreasing):
        assert call(lay) == 1
    huge = lib.HostLayout(np.array([0, 1 << 31], np.int64), np.zeros(0, np.int32), np.zeros(0, np.int64))
    assert call(huge) == 2                               # a sequence beyond 2^31 - 2 keys
    empty = _layout(lib, [100], np.zeros(0, np.int32), np.zeros(0, np.int64))
    assert call(empty, ws=None) == 0                     # no queries: nothing to do, nothing launched
    assert call(_layout(lib, [100], [0], [5]), ws=None) == 1   # queries need a workspace
    assert lib._lib.saki_recall(ctypes.byref(cfg), ctypes.byref(empty.c), 65, FAKE, FAKE, FAKE, FAKE, None, FAKE,
                                None, 1 << 40, None) == 1   # recall always needs its workspace
    big = _cfg(lib, num_q_heads=65536 * 2, num_kv_heads=2)
    assert lib._lib.saki_score_topk(ctypes.byref(big), ctypes.byref(empty.c), FAKE, FAKE, FAKE, None, FAKE, None,
                                    FAKE, 1 << 40, None) == 2


def test_score_mse_and_reconstruct_argument_checks(lib):
    cfg = _cfg(lib)
    lay = _layout(lib, [100], [0, 0], [10, 20])
    mse = lambda stride, out, ws, nb: lib._lib.saki_score_mse(ctypes.byref(cfg), ctypes.byref(lay.c), stride, FAKE,
                                                              FAKE, FAKE, FAKE, FAKE, None, out, ws, nb, None)
    need = lib.saki_workspace_size(cfg, lib.SAKI_OP_SCORE_MSE, lay)
    assert need >= 256 + 2 * 16
    assert mse(0, FAKE, FAKE, need) == 1
    assert mse(1, None, FAKE, need) == 1
    assert mse(1, FAKE, None, need) == 1
    assert mse(1, FAKE, FAKE, need - 1) == 6
    rec = lambda n, pos, theta, ws, nb: lib._lib.saki_reconstruct_keys(ctypes.byref(cfg), n, FAKE, 100, FAKE, FAKE,
                                                                        None, pos, theta, FAKE, ws, nb, None)
    assert rec(-1, None, 10000.0, None, 0) == 1
    assert rec(4, FAKE, 1.0, FAKE, 1 << 20) == 1         # rope_theta must exceed 1
    assert rec(4, FAKE, 10000.0, None, 0) == 1           # rotation needs its workspace
    need = lib.saki_workspace_size(cfg, lib.SAKI_OP_RECONSTRUCT, total_keys=4)
    assert need >= 4 * 64 * 8
    assert rec(4, FAKE, 10000.0, FAKE, 4 * 64 * 8 - 1) == 6


def test_merge_argument_checks(lib):
    cfg = _cfg(lib)
    offs = (ctypes.c_int64 * 65)(*range(0, 65 * 100, 100))
    call = lambda parts, o: lib._lib.saki_merge_topk(ctypes.byref(cfg), parts, 4, FAKE, FAKE, o, FAKE, None, None)
    assert call(0, offs) == 1
    assert call(65, offs) == 2                           # at most 64 parts
    neg = (ctypes.c_int64 * 2)(0, -5)
    assert call(2, neg) == 1
    assert lib.saki_status_string(99) == "unknown status"


def test_plain_c_program_links_and_calls_the_abi(lib, tmp_path):
    """The boundary is usable from C without Python: a C program includes
    saki.h, links libsaki.so, sizes workspaces and receives argument errors
    (every call here returns before any device work)."""
    src = tmp_path / "use.c"
    src.write_text(r'''
#include <stdio.h>
#include <stdint.h>
#include "saki.h"
int main(void) {
  saki_config c = {0};
  c.num_q_heads = 8; c.num_kv_heads = 2; c.head_dim = 128; c.rank = 32; c.topk = 64;
  c.dtype = SAKI_BF16; c.eig_floor_rel = 1e-6f;
  int64_t off[2] = {0, 4096};
  int32_t qs[1] = {0};
  int64_t qv[1] = {4096};
  saki_layout L = {1, off, 1, qs, qv};
  size_t fit = saki_workspace_size(&c, SAKI_OP_FIT, NULL, 16, 0);
  size_t sel = saki_workspace_size(&c, SAKI_OP_SCORE_TOPK, &L, 0, 0);
  c.rank = 0;
  size_t bad = saki_workspace_size(&c, SAKI_OP_FIT, NULL, 16, 0);
  saki_status st = saki_fit(&c, 16, NULL, NULL, NULL, NULL, NULL, NULL, NULL, NULL, NULL, NULL, 0, NULL);
  printf("%zu %zu %zu %d %s\n", fit, sel, bad, (int)st, saki_version());
  puts(saki_status_string(st));
  return 0;
}''')
    exe = tmp_path / "use"
    libdir = os.path.dirname(lib.library_path())
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), str(src), "-L", libdir,
                    "-lsaki", "-Wl,-rpath," + libdir, "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.splitlines()
    fit, sel, bad, st, ver = out[0].split()
    cfg = _cfg(lib)
    assert int(fit) == lib.saki_workspace_size(cfg, lib.SAKI_OP_FIT, n_calib=16) > 0
    lay = _layout(lib, [4096], [0], [4096])
    assert int(sel) == lib.saki_workspace_size(cfg, lib.SAKI_OP_SCORE_TOPK, lay) > 0
    assert int(bad) == 0 and int(st) == 1 and ver == lib.saki_version()
    assert out[1] == "invalid argument"

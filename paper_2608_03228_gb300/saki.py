"""Thin ctypes binding of libsaki.so (include/saki.h).

Argument marshalling only: every step of the path runs in the library's CUDA
kernels.  Device tensors are torch CUDA tensors (PyTorch supplies device memory
and the current stream); the layout arrays are host numpy arrays.  Importing
this module loads the library and raises if it has not been built -- there is
no fallback path.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "libsaki.so")
if not os.path.exists(_LIB_PATH):
    raise ImportError(f"{_LIB_PATH} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
_lib = ctypes.CDLL(_LIB_PATH)

SAKI_F32, SAKI_BF16 = 0, 1
SAKI_FLAG_SORTED, SAKI_FLAG_CHECK, SAKI_FLAG_SHRINK = 1, 2, 4
SAKI_METHOD_SAKI, SAKI_METHOD_KEY_PCA, SAKI_METHOD_WEIGHT_SVD, SAKI_METHOD_SAP_SVD, SAKI_METHOD_SAP_MAP = 0, 1, 2, 3, 4
METHODS = {"saki": SAKI_METHOD_SAKI, "key_pca": SAKI_METHOD_KEY_PCA, "weight_svd": SAKI_METHOD_WEIGHT_SVD,
           "sap_svd": SAKI_METHOD_SAP_SVD, "sap_map": SAKI_METHOD_SAP_MAP}
SAKI_OP_FIT, SAKI_OP_BUILD_INDEX, SAKI_OP_SCORE_TOPK, SAKI_OP_RECALL = 0, 1, 2, 3
SAKI_OP_KEY_SPECTRUM, SAKI_OP_SCORE_MSE, SAKI_OP_MOMENTS, SAKI_OP_RECONSTRUCT = 4, 5, 6, 7
STATUS = {0: "SAKI_OK", 1: "SAKI_ERR_INVALID_ARGUMENT", 2: "SAKI_ERR_UNSUPPORTED", 3: "SAKI_ERR_CUDA",
          4: "SAKI_ERR_NUMERIC", 5: "SAKI_ERR_NOT_CONVERGED", 6: "SAKI_ERR_WORKSPACE", 7: "SAKI_ERR_TIMEOUT"}
EXPORTS = ("saki_workspace_size", "saki_fit", "saki_build_index", "saki_score_topk", "saki_recall",
           "saki_status_string", "saki_version", "saki_score_topk_noalloc", "saki_launch_count",
           "saki_kernel_timer_start", "saki_kernel_timer_stop", "saki_workspace_status", "saki_noalloc_status",
           "saki_debug_inject_stall", "saki_merge_topk", "saki_key_spectrum", "saki_score_mse",
           "saki_moments", "saki_fit_moments", "saki_reconstruct_keys")
SAKI_KERNEL_SELECT, SAKI_KERNEL_EXACT, SAKI_KERNEL_FIT, SAKI_KERNEL_MOMENTS, SAKI_KERNEL_BUILD, SAKI_KERNEL_FACTOR = (
    1, 2, 3, 4, 5, 6)
SAKI_NOALLOC_SCRATCH_BYTES = 16 << 20


class Config(ctypes.Structure):
    _fields_ = [("num_q_heads", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("rank", ctypes.c_int32), ("topk", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("center", ctypes.c_int32), ("eig_floor_rel", ctypes.c_float), ("max_sweeps", ctypes.c_int32),
                ("flags", ctypes.c_int32), ("method", ctypes.c_int32)]


class Layout(ctypes.Structure):
    _fields_ = [("num_seqs", ctypes.c_int32), ("seq_offsets", ctypes.c_void_p), ("num_queries", ctypes.c_int64),
                ("q_seq", ctypes.c_void_p), ("q_visible", ctypes.c_void_p)]


_vp, _i64, _i32, _sz = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_size_t
_lib.saki_workspace_size.restype = _sz
_lib.saki_workspace_size.argtypes = [ctypes.POINTER(Config), _i32, ctypes.POINTER(Layout), _i64, _i64]
_lib.saki_fit.restype = ctypes.c_int
_lib.saki_fit.argtypes = [ctypes.POINTER(Config), _i64] + [_vp] * 10 + [_sz, _vp]
_lib.saki_build_index.restype = ctypes.c_int
_lib.saki_build_index.argtypes = [ctypes.POINTER(Config), _i64] + [_vp] * 5 + [_sz, _vp]
_lib.saki_score_topk.restype = ctypes.c_int
_lib.saki_score_topk.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(Layout)] + [_vp] * 7 + [_sz, _vp]
_lib.saki_recall.restype = ctypes.c_int
_lib.saki_recall.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(Layout), _i64] + [_vp] * 7 + [_sz, _vp]
_lib.saki_score_topk_noalloc.restype = ctypes.c_int
_lib.saki_score_topk_noalloc.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(Layout)] + [_vp] * 6 + [_vp]
_lib.saki_workspace_status.restype = ctypes.c_int
_lib.saki_workspace_status.argtypes = [_vp, _vp]
_lib.saki_noalloc_status.restype = ctypes.c_int
_lib.saki_noalloc_status.argtypes = [_vp]
_lib.saki_debug_inject_stall.restype = ctypes.c_int
_lib.saki_debug_inject_stall.argtypes = [_i32]
_lib.saki_merge_topk.restype = ctypes.c_int
_lib.saki_merge_topk.argtypes = [ctypes.POINTER(Config), _i32, _i64, _vp, _vp, _vp, _vp, _vp, _vp]
_lib.saki_key_spectrum.restype = ctypes.c_int
_lib.saki_key_spectrum.argtypes = [ctypes.POINTER(Config), _i64, _vp, ctypes.c_float, _vp, _vp, _vp, _sz, _vp]
_lib.saki_score_mse.restype = ctypes.c_int
_lib.saki_score_mse.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(Layout), _i64] + [_vp] * 8 + [_sz, _vp]
_lib.saki_moments.restype = ctypes.c_int
_lib.saki_moments.argtypes = [ctypes.POINTER(Config), _i64, _vp, _vp, _i64, _vp, _vp, _vp, _vp, _sz, _vp]
_lib.saki_fit_moments.restype = ctypes.c_int
_lib.saki_fit_moments.argtypes = [ctypes.POINTER(Config)] + [_vp] * 10 + [_sz, _vp]
_lib.saki_reconstruct_keys.restype = ctypes.c_int
_lib.saki_reconstruct_keys.argtypes = [ctypes.POINTER(Config), _i64, _vp, _i64, _vp, _vp, _vp, _vp, ctypes.c_float,
                                       _vp, _vp, _sz, _vp]
_lib.saki_status_string.restype = ctypes.c_char_p
_lib.saki_status_string.argtypes = [ctypes.c_int]
_lib.saki_version.restype = ctypes.c_char_p
_lib.saki_launch_count.restype = _i64
_lib.saki_launch_count.argtypes = []
_lib.saki_kernel_timer_start.restype = ctypes.c_int
_lib.saki_kernel_timer_start.argtypes = [_i32]
_lib.saki_kernel_timer_stop.restype = ctypes.c_int
_lib.saki_kernel_timer_stop.argtypes = [_i32, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(_i64)]


class SakiError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS.get(status, status)} ({_lib.saki_status_string(status).decode()})")


def library_path() -> str:
    return _LIB_PATH


def make_config(num_q_heads, num_kv_heads, rank, topk, dtype="bf16", center=0, eig_floor_rel=1e-6,
                max_sweeps=0, flags=0, head_dim=128, method="saki") -> Config:
    dt = {"f32": SAKI_F32, "bf16": SAKI_BF16}.get(dtype, dtype)
    m = METHODS.get(method, method)
    return Config(num_q_heads, num_kv_heads, head_dim, rank, topk, dt, center, eig_floor_rel, max_sweeps, flags, m)


class HostLayout:
    """Holds the host arrays of a saki_layout alive while a call uses them."""

    def __init__(self, seq_offsets, q_seq, q_visible):
        self.seq_offsets = np.ascontiguousarray(seq_offsets, np.int64)
        self.q_seq = np.ascontiguousarray(q_seq, np.int32)
        self.q_visible = np.ascontiguousarray(q_visible, np.int64)
        self.c = Layout(len(self.seq_offsets) - 1, self.seq_offsets.ctypes.data, len(self.q_seq),
                        self.q_seq.ctypes.data if len(self.q_seq) else None,
                        self.q_visible.ctypes.data if len(self.q_visible) else None)

    @property
    def total_keys(self) -> int:
        return int(self.seq_offsets[-1])


def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is not None:
        return stream if isinstance(stream, int) else stream.cuda_stream
    import torch
    return torch.cuda.current_stream().cuda_stream


def _check(status: int, where: str):
    if status != 0:
        raise SakiError(status, where)


def _workspace(nbytes: int, device):
    import torch
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


def saki_status_string(status: int) -> str:
    return _lib.saki_status_string(status).decode()


def saki_version() -> str:
    return _lib.saki_version().decode()


def saki_launch_count() -> int:
    return int(_lib.saki_launch_count())


def saki_kernel_timer_start(kind: int) -> None:
    _check(_lib.saki_kernel_timer_start(kind), "saki_kernel_timer_start")


def saki_kernel_timer_stop(kind: int) -> tuple[float, int]:
    """Summed device milliseconds and number of timed launches of the kind since it was armed."""
    ms, n = ctypes.c_double(0.0), _i64(0)
    _check(_lib.saki_kernel_timer_stop(kind, ctypes.byref(ms), ctypes.byref(n)), "saki_kernel_timer_stop")
    return ms.value, int(n.value)


def saki_workspace_status(workspace, stream=None) -> None:
    """Raise SakiError(SAKI_ERR_TIMEOUT) if a kernel of the last selection, recall
    or index call on this workspace gave up a bounded wait (synchronises stream)."""
    _check(_lib.saki_workspace_status(_ptr(workspace), _stream(stream)), "saki_workspace_status")


def saki_noalloc_status(stream=None) -> None:
    _check(_lib.saki_noalloc_status(_stream(stream)), "saki_noalloc_status")


def saki_debug_inject_stall(kind: int) -> None:
    """Test hook: the next tensor-core launch of this kernel kind stalls its producer."""
    _check(_lib.saki_debug_inject_stall(kind), "saki_debug_inject_stall")


def saki_key_spectrum(cfg: Config, k_calib, eig, spikes, tau_int=1.0, workspace=None, stream=None) -> None:
    """Sec. 7: eigenvalues of each KV head's key correlation matrix (descending,
    eig [Hk][d]) and the count above the Marchenko-Pastur edge (spikes [Hk] int32)."""
    n = k_calib.shape[1]
    need = saki_workspace_size(cfg, SAKI_OP_KEY_SPECTRUM)
    ws = workspace if workspace is not None else _workspace(need, k_calib.device)
    _check(_lib.saki_key_spectrum(ctypes.byref(cfg), n, _ptr(k_calib), float(tau_int), _ptr(eig), _ptr(spikes),
                                  _ptr(ws), ws.numel(), _stream(stream)), "saki_key_spectrum")


def saki_score_mse(cfg: Config, layout: HostLayout, Q, A, K, L, sketch, out, nu=None, key_stride=1, workspace=None,
                   stream=None) -> None:
    """App. C: per head sum s^2, sum (s - s_hat)^2, pairs (out [Hq][3] float64)."""
    need = saki_workspace_size(cfg, SAKI_OP_SCORE_MSE, layout)
    ws = workspace if workspace is not None else _workspace(need, Q.device)
    _check(_lib.saki_score_mse(ctypes.byref(cfg), ctypes.byref(layout.c), int(key_stride), _ptr(Q), _ptr(A), _ptr(K),
                               _ptr(L), _ptr(sketch), _ptr(nu), _ptr(out), _ptr(ws), ws.numel(), _stream(stream)),
           "saki_score_mse")


def saki_moments(cfg: Config, q_new, k_new, n_prev, Sq, Sk, mu=None, workspace=None, stream=None) -> None:
    """Add a batch of calibration rows to running moments covering n_prev rows."""
    need = saki_workspace_size(cfg, SAKI_OP_MOMENTS)
    ws = workspace if workspace is not None else _workspace(need, q_new.device)
    _check(_lib.saki_moments(ctypes.byref(cfg), q_new.shape[1], _ptr(q_new), _ptr(k_new), int(n_prev), _ptr(Sq),
                             _ptr(Sk), _ptr(mu), _ptr(ws), ws.numel(), _stream(stream)), "saki_moments")


def saki_fit_moments(cfg: Config, Sq, Sk, A, L, R, mu=None, nu=None, sigma=None, loss=None, workspace=None,
                     stream=None) -> None:
    need = saki_workspace_size(cfg, SAKI_OP_FIT, n_calib=1)
    ws = workspace if workspace is not None else _workspace(need, Sq.device)
    _check(_lib.saki_fit_moments(ctypes.byref(cfg), _ptr(Sq), _ptr(Sk), _ptr(mu), _ptr(A), _ptr(L), _ptr(R), _ptr(nu),
                                 _ptr(sigma), _ptr(loss), _ptr(ws), ws.numel(), _stream(stream)), "saki_fit_moments")


def saki_reconstruct_keys(cfg: Config, rows, sketch, L, keys, nu=None, positions=None, rope_theta=10000.0,
                          workspace=None, stream=None) -> None:
    """k_hat = nu + L c of the given code rows (device int64) of every head, RoPE-rotated at positions."""
    n = rows.numel()
    need = saki_workspace_size(cfg, SAKI_OP_RECONSTRUCT, total_keys=n)
    ws = workspace if workspace is not None else _workspace(need, sketch.device)
    _check(_lib.saki_reconstruct_keys(ctypes.byref(cfg), n, _ptr(rows), sketch.shape[1], _ptr(sketch), _ptr(L),
                                      _ptr(nu), _ptr(positions), float(rope_theta), _ptr(keys), _ptr(ws), ws.numel(),
                                      _stream(stream)), "saki_reconstruct_keys")


def saki_merge_topk(cfg: Config, idx_parts, score_parts, part_offsets, idx, score=None, stream=None) -> None:
    """The k best of per-part top-k lists (idx_parts, score_parts [P][rows][k] on
    the device, part-local indices); part_offsets: host sequence of P ints."""
    offs = np.ascontiguousarray(part_offsets, np.int64)
    P = idx_parts.shape[0]
    rows = idx_parts.numel() // (P * cfg.topk) if P else 0
    _check(_lib.saki_merge_topk(ctypes.byref(cfg), P, rows, _ptr(idx_parts), _ptr(score_parts), offs.ctypes.data,
                                _ptr(idx), _ptr(score), _stream(stream)), "saki_merge_topk")


def saki_workspace_size(cfg: Config, op: int, layout: HostLayout | None = None, n_calib: int = 0,
                        total_keys: int = 0) -> int:
    return int(_lib.saki_workspace_size(ctypes.byref(cfg), op, ctypes.byref(layout.c) if layout else None,
                                        n_calib, total_keys))


def saki_fit(cfg: Config, q_calib, k_calib, A, L, R, mu=None, nu=None, sigma=None, loss=None, workspace=None,
             stream=None):
    """Prop. 1 fit; all arguments are CUDA tensors laid out as in saki.h."""
    n = q_calib.shape[1]
    need = saki_workspace_size(cfg, SAKI_OP_FIT, n_calib=n)
    ws = workspace if workspace is not None else _workspace(need, q_calib.device)
    _check(_lib.saki_fit(ctypes.byref(cfg), n, _ptr(q_calib), _ptr(k_calib), _ptr(A), _ptr(L), _ptr(R), _ptr(mu),
                         _ptr(nu), _ptr(sigma), _ptr(loss), _ptr(ws), ws.numel(), _stream(stream)), "saki_fit")


def saki_build_index(cfg: Config, K, R, sketch, mu=None, workspace=None, stream=None):
    N = K.shape[1]
    need = saki_workspace_size(cfg, SAKI_OP_BUILD_INDEX, total_keys=N)
    ws = workspace if workspace is not None else _workspace(need, K.device)
    _check(_lib.saki_build_index(ctypes.byref(cfg), N, _ptr(K), _ptr(R), _ptr(mu), _ptr(sketch), _ptr(ws),
                                 ws.numel(), _stream(stream)), "saki_build_index")


def saki_score_topk(cfg: Config, layout: HostLayout, Q, L, sketch, idx, score=None, nu=None, workspace=None,
                    stream=None):
    need = saki_workspace_size(cfg, SAKI_OP_SCORE_TOPK, layout)
    ws = workspace if workspace is not None else _workspace(need, Q.device)
    _check(_lib.saki_score_topk(ctypes.byref(cfg), ctypes.byref(layout.c), _ptr(Q), _ptr(L), _ptr(sketch), _ptr(nu),
                                _ptr(idx), _ptr(score), _ptr(ws), ws.numel(), _stream(stream)), "saki_score_topk")


def saki_recall(cfg: Config, layout: HostLayout, min_visible: int, Q, A, K, idx_approx, recall, idx_exact=None,
                workspace=None, stream=None):
    need = saki_workspace_size(cfg, SAKI_OP_RECALL, layout)
    ws = workspace if workspace is not None else _workspace(need, Q.device)
    _check(_lib.saki_recall(ctypes.byref(cfg), ctypes.byref(layout.c), min_visible, _ptr(Q), _ptr(A), _ptr(K),
                            _ptr(idx_approx), _ptr(idx_exact), _ptr(recall), _ptr(ws), ws.numel(), _stream(stream)),
           "saki_recall")


def saki_score_topk_noalloc(cfg: Config, layout: HostLayout, Q, L, sketch, idx, score=None, nu=None, stream=None):
    """saki_score_topk without a workspace: the library's static device scratch
    serves instead (for callers that cannot allocate device memory)."""
    _check(_lib.saki_score_topk_noalloc(ctypes.byref(cfg), ctypes.byref(layout.c), _ptr(Q), _ptr(L), _ptr(sketch),
                                        _ptr(nu), _ptr(idx), _ptr(score), _stream(stream)),
           "saki_score_topk_noalloc")

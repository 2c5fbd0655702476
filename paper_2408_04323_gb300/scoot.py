"""ctypes binding of libscoot (include/scoot.h): argument marshalling only.

Every function here has the name of the C entry point it calls and does no
arithmetic of its own: host arrays are numpy arrays (passed by pointer),
device arrays are CUDA torch tensors (passed by data pointer), streams are
torch CUDA streams (passed by handle).  A non-zero status raises ScootError
with the library's message.  If libscoot.so has not been built, importing
the functions raises ImportError: there is no fallback path.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libscoot.so")

INT_UNIFORM, INT_LOG, CATEGORICAL, CONTINUOUS = 0, 1, 2, 3
MATERN52, MATERN32 = 0, 1
MAX_DIM, MAX_CLAUSES, MAX_OBJ, MAX_OBS, MAX_Q = 16, 16, 4, 640, 64

STATUS = {0: "SCOOT_OK", -1: "SCOOT_EINVAL", -2: "SCOOT_ENOMEM", -3: "SCOOT_ECUDA",
          -4: "SCOOT_EDEVICE", -5: "SCOOT_ETIMEOUT", -6: "SCOOT_EUNSUPPORTED"}


class ScootError(RuntimeError):
    def __init__(self, status: int, func: str, message: str = ""):
        self.status = status
        super().__init__(f"{func}: {STATUS.get(status, status)} {message}".rstrip())


class scoot_param(C.Structure):
    _fields_ = [("kind", C.c_int32), ("n_choices", C.c_int32), ("lo", C.c_float), ("hi", C.c_float)]


class scoot_clause(C.Structure):
    _fields_ = [("n_guard", C.c_int32), ("guard_param", C.c_int32 * 2), ("guard_value", C.c_int32 * 2),
                ("n_term", C.c_int32), ("term_param", C.c_int32 * 4), ("coef", C.c_int64 * 4),
                ("rhs", C.c_int64)]


class scoot_node(C.Structure):
    _fields_ = [("val", C.c_float), ("left", C.c_uint16), ("feat", C.c_uint8), ("flags", C.c_uint8)]


class scoot_forest_layout(C.Structure):
    _fields_ = [("n_trees", C.c_int32), ("n_nodes", C.c_int32), ("d", C.c_int32), ("leaf_scale", C.c_int32),
                ("max_depth", C.c_int32), ("n_chunks", C.c_int32), ("max_chunk_nodes", C.c_int32),
                ("reserved", C.c_int32), ("bytes", C.c_int64), ("off_chunks", C.c_int64),
                ("off_roots", C.c_int64), ("off_nodes", C.c_int64)]


class scoot_gp_layout(C.Structure):
    _fields_ = [("n", C.c_int32), ("d", C.c_int32), ("n_obj", C.c_int32), ("kernel", C.c_int32),
                ("n_rb", C.c_int32), ("n_tiles", C.c_int32), ("n_ord", C.c_int32), ("n_pat", C.c_int32),
                ("bytes", C.c_int64), ("off_fmap", C.c_int64), ("off_xs", C.c_int64), ("off_ils", C.c_int64),
                ("off_alpha", C.c_int64), ("off_linv", C.c_int64), ("off_scal", C.c_int64),
                ("off_cat", C.c_int64), ("off_warp", C.c_int64)]


class scoot_round_inputs(C.Structure):
    _fields_ = [("space", C.c_void_p), ("d", C.c_int32), ("x_obs", C.c_void_p), ("ld_obs", C.c_int64),
                ("n", C.c_int32), ("n_obj", C.c_int32), ("y", C.c_void_p), ("lengthscale", C.c_void_p),
                ("signal_var", C.c_void_p), ("noise_var", C.c_void_p), ("warp", C.c_void_p), ("kernel", C.c_int32),
                ("gp_on_device", C.c_int32), ("nodes", C.c_void_p), ("tree_offset", C.c_void_p),
                ("n_trees", C.c_int32), ("leaf_scale", C.c_int32), ("boxes", C.c_int32), ("ref", C.c_void_p),
                ("eps", C.c_void_p), ("n_mc", C.c_int32), ("grid_cap", C.c_int32), ("fantasy_q", C.c_int32)]


class scoot_round_state(C.Structure):
    _fields_ = [("bytes", C.c_int64), ("off_gp", C.c_int64), ("off_forest", C.c_int64),
                ("off_box_lo", C.c_int64), ("off_box_hi", C.c_int64), ("off_eps", C.c_int64),
                ("off_grid", C.c_int64), ("off_corner", C.c_int64), ("off_fant", C.c_int64),
                ("fant_box_cap", C.c_int32), ("n_boxes", C.c_int32),
                ("front_size", C.c_int32), ("grid_cap", C.c_int32), ("n_grid", C.c_int32 * 4),
                ("cond", C.c_double * 4), ("gp", scoot_gp_layout), ("forest", scoot_forest_layout)]


# scoot_node as a numpy record (host copies of trained trees)
NODE_DTYPE = np.dtype([("val", "<f4"), ("left", "<u2"), ("feat", "u1"), ("flags", "u1")])

assert C.sizeof(scoot_param) == 16 and C.sizeof(scoot_clause) == 80 and C.sizeof(scoot_node) == 8

_vp, _i32, _i64, _u32, _f32 = C.c_void_p, C.c_int32, C.c_int64, C.c_uint32, C.c_float
_PROTOS = {
    "scoot_ctx_create": [_i32, C.POINTER(_vp)],
    "scoot_ctx_destroy": [_vp],
    "scoot_last_error": [_vp],
    "scoot_status_string": [_i32],
    "scoot_ctx_check": [_vp, _vp],
    "scoot_ctx_workspace_bytes": [_vp, C.POINTER(_i64)],
    "scoot_ctx_set_timing": [_vp, _i32],
    "scoot_ctx_set_tensor_cores": [_vp, _i32],
    "scoot_probe_fma": [_vp, _i32, _i32, _i32, _vp, _vp],
    "scoot_probe_gather": [_vp, _i32, _i32, _i32, _vp, _vp],
    "scoot_ctx_phase_times": [_vp, _i32, _vp, _vp, C.POINTER(_i32)],
    "scoot_prune": [_vp, _vp, _i32, _vp, _i32, _vp, _i64, _i64, _vp, _vp, _vp],
    "scoot_forest_layout_init": [_vp, _vp, _i32, _i32, _i32, C.POINTER(scoot_forest_layout)],
    "scoot_forest_pack": [C.POINTER(scoot_forest_layout), _vp, _vp, _vp],
    "scoot_rf_predict": [_vp, C.POINTER(scoot_forest_layout), _vp, _vp, _vp, _i64, _i64, _u32, _u32,
                         _vp, _vp, _vp, _vp],
    "scoot_gp_layout_init": [_vp, _i32, _i32, _i32, _i32, C.POINTER(scoot_gp_layout)],
    "scoot_gp_prepare": [_vp, _vp, _i64, _vp, _vp, _vp, _vp, C.POINTER(scoot_gp_layout), _vp, _vp],
    "scoot_gp_prepare_warped": [_vp, _vp, _i64, _vp, _vp, _vp, _vp, _vp, C.POINTER(scoot_gp_layout), _vp, _vp],
    "scoot_gp_device_work_bytes": [C.POINTER(scoot_gp_layout), C.POINTER(_i64)],
    "scoot_gp_device_buffer_layout": [C.POINTER(scoot_gp_layout), _i32, C.POINTER(_i64), C.POINTER(_i64),
                                      C.POINTER(_i64), C.POINTER(_i64)],
    "scoot_gp_prepare_device_from_host": [_vp, _vp, C.POINTER(scoot_gp_layout), _vp, _i64, _vp, _vp, _vp, _vp, _vp,
                                          _vp, _vp, _i64, _vp],
    "scoot_gp_mle": [_vp, _vp, _i32, _vp, _i64, _i32, _vp, _i32, _i32, _vp, _i32, _vp, _vp, _u32, _i32,
                     C.c_double, _vp, _vp, _vp, _vp, _i64, _vp],
    "scoot_gp_mle_work_bytes": [_i32, _i32, _i32, _i32, C.POINTER(_i64)],
    "scoot_round_state_build": [C.POINTER(scoot_round_inputs), _vp, _i64, C.POINTER(scoot_round_state)],
    "scoot_gp_prepare_device": [_vp, _vp, C.POINTER(scoot_gp_layout), _vp, _i64, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                _i64, _vp],
    "scoot_gp_posterior": [_vp, C.POINTER(scoot_gp_layout), _vp, _vp, _i64, _i64, _vp, _vp, _vp, _i64, _vp],
    "scoot_acq_ei": [_vp, _vp, _vp, _vp, _i64, _f32, _f32, _vp, _vp],
    "scoot_boxes_build": [_vp, _i32, _i32, _vp, _i32, _vp, _vp, C.POINTER(_i32), C.POINTER(_i32)],
    "scoot_acq_ehvi": [_vp, _vp, _vp, _i64, _i32, _vp, _i64, _vp, _vp, _i32, _vp, _i32, _vp, _vp],
    "scoot_boxes_index": [_vp, _vp, _i32, _i32, _i32, _vp, _vp, _vp],
    "scoot_acq_ehvi_exact": [_vp, _vp, _vp, _i64, _i32, _vp, _i64, _vp, _i32, _vp, _vp, _i32, _vp, _vp],
    "scoot_score_ehvi_exact": [_vp, C.POINTER(scoot_gp_layout), _vp, _vp, _i64, _i64, _vp, _vp, _i32, _vp, _vp,
                               _i32, _vp, _vp],
    "scoot_score_ei": [_vp, C.POINTER(scoot_gp_layout), _vp, _vp, _i64, _i64, _vp, _f32, _vp, _vp],
    "scoot_score_ehvi": [_vp, C.POINTER(scoot_gp_layout), _vp, _vp, _i64, _i64, _vp, _vp, _vp, _i32,
                         _vp, _i32, _vp, _vp],
    "scoot_select_topq": [_vp, _vp, _vp, _i64, _i32, _vp, _vp, _vp, _vp],
    "scoot_acq_mace": [_vp, _vp, _vp, _vp, _i64, _f32, _f32, _f32, _vp, _i64, _vp],
    "scoot_score_mace": [_vp, C.POINTER(scoot_gp_layout), _vp, _vp, _i64, _i64, _vp, _f32, _f32, _vp, _i64, _vp],
    "scoot_sobol_configs": [_vp, _vp, _i32, _i64, _i64, _vp, _i64, _vp],
    "scoot_first_feasible": [_vp, _vp, _i64, _i32, _vp, _vp, _vp],
    "scoot_delta_update": [C.POINTER(C.c_double), C.POINTER(_i32), _i32, _i32],
    "scoot_ucb_beta": [_i32, C.POINTER(C.c_double)],
    "scoot_standardize": [_vp, _i32, _i32, _vp, _vp, _f32],
    "scoot_rf_train": [_vp, _vp, _i32, _vp, _i32, _i64, _vp, _vp, _i32, _i32, _i32, _i32, _vp, _i32, _vp, _vp,
                       _i64, _vp],
    "scoot_rf_train_work_bytes": [_i32, _i32, C.POINTER(_i64)],
    "scoot_select_pareto": [_vp, _vp, _i64, _vp, _i64, _i32, C.c_uint64, _vp, _vp, _vp, _i64, _vp],
    "scoot_select_topq_static": [_vp, _vp, _i64, _i32, _vp, _vp, _vp, _vp],
    "scoot_fantasy_state_bytes": [C.POINTER(scoot_gp_layout), _i32, C.POINTER(_i64)],
    "scoot_fantasy_prepare": [_vp, C.POINTER(scoot_gp_layout), _vp, _i64, _vp, _vp, _vp, _vp, _vp, _i32, _vp, _i64,
                              C.POINTER(_i32)],
    "scoot_fantasy_work_bytes": [C.POINTER(scoot_gp_layout), _i64, _i32, _i32, C.POINTER(_i64)],
    "scoot_fantasy_begin": [_vp, C.POINTER(scoot_gp_layout), _vp, _vp, _i32, _vp, _i64, _i64, _vp, _i64, _vp, _i32,
                            _i32, _vp, _i64, _vp, _vp, _vp, _vp],
    "scoot_fantasy_local_best": [_vp, _i32, _vp, _vp],
    "scoot_fantasy_commit": [_vp, _i32, _vp, _i32, _vp],
    "scoot_fantasy_end": [_vp, _vp, _vp],
    "scoot_suggest_fantasy": [_vp, C.POINTER(scoot_gp_layout), _vp, _vp, _i32, _vp, _i64, _i64, _vp, _vp, _i32,
                              _i32, _vp, _i64, _vp, _vp, _vp, _vp, _vp],
}
_STRING_FUNCS = {"scoot_last_error", "scoot_status_string"}
EXPORTS = tuple(_PROTOS)

_lib = None


def lib() -> C.CDLL:
    """The loaded libscoot.so (ImportError if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: build it with paper_2408_04323_gb300.build()")
        L = C.CDLL(LIB_PATH)
        for name, args in _PROTOS.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = C.c_char_p if name in _STRING_FUNCS else _i32
        _lib = L
    return _lib


# ------------------------------------------------------------------ marshalling

def _host(a, itemsize=None, dtype=None, name="array"):
    if a is None:
        return None
    if not isinstance(a, np.ndarray):
        raise TypeError(f"{name} must be a numpy array (host memory)")
    if not a.flags.c_contiguous:
        raise ValueError(f"{name} must be C-contiguous")
    if dtype is not None and a.dtype != np.dtype(dtype):
        raise TypeError(f"{name} must have dtype {np.dtype(dtype)}, got {a.dtype}")
    if itemsize is not None and a.dtype.itemsize != itemsize:
        raise TypeError(f"{name} items must be {itemsize} bytes, got {a.dtype.itemsize}")
    return a.ctypes.data_as(_vp)


def _dev(t, dtype=None, name="tensor"):
    if t is None:
        return None
    import torch
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA torch tensor (device memory)")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must have dtype {dtype}, got {t.dtype}")
    return _vp(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return _vp(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _check(status, func, ctx=None):
    if status != 0:
        msg = ""
        if ctx is not None:
            raw = lib().scoot_last_error(ctx)
            msg = raw.decode() if raw else ""
        raise ScootError(int(status), func, msg)


# ------------------------------------------------------------------ context

def scoot_ctx_create(device: int = 0) -> C.c_void_p:
    h = _vp()
    _check(lib().scoot_ctx_create(int(device), C.byref(h)), "scoot_ctx_create")
    return h


def scoot_ctx_destroy(ctx) -> None:
    _check(lib().scoot_ctx_destroy(ctx), "scoot_ctx_destroy")


def scoot_ctx_check(ctx, stream=None) -> None:
    _check(lib().scoot_ctx_check(ctx, _stream(stream)), "scoot_ctx_check", ctx)


def scoot_ctx_workspace_bytes(ctx) -> int:
    v = _i64()
    _check(lib().scoot_ctx_workspace_bytes(ctx, C.byref(v)), "scoot_ctx_workspace_bytes")
    return int(v.value)


PHASES = {0: "compact", 1: "posterior", 2: "fant_init", 3: "fant_pass", 4: "fant_pick", 5: "scatter"}


def scoot_ctx_set_timing(ctx, enable: bool) -> None:
    _check(lib().scoot_ctx_set_timing(_h(ctx), int(bool(enable))), "scoot_ctx_set_timing", _h(ctx))


def scoot_ctx_set_tensor_cores(ctx, enable: bool) -> None:
    _check(lib().scoot_ctx_set_tensor_cores(_h(ctx), int(bool(enable))), "scoot_ctx_set_tensor_cores", _h(ctx))


def scoot_ctx_phase_times(ctx, cap: int = 256):
    """[(phase name, milliseconds)] of the last timed call's launches, in order."""
    kind = np.zeros(cap, np.int32)
    ms = np.zeros(cap, np.float32)
    cnt = _i32()
    _check(lib().scoot_ctx_phase_times(_h(ctx), int(cap), _host(kind), _host(ms), C.byref(cnt)),
           "scoot_ctx_phase_times", _h(ctx))
    k = min(cnt.value, cap)
    return [(PHASES.get(int(kind[i]), str(int(kind[i]))), float(ms[i])) for i in range(k)]


def scoot_probe_fma(ctx, packed: bool, blocks: int, iters: int, sink, stream=None) -> None:
    import torch
    _check(lib().scoot_probe_fma(_h(ctx), int(bool(packed)), int(blocks), int(iters),
                                 _dev(sink, torch.float32, "sink"), _stream(stream)), "scoot_probe_fma", _h(ctx))


def scoot_probe_gather(ctx, n_nodes: int, blocks: int, steps: int, sink, stream=None) -> None:
    import torch
    _check(lib().scoot_probe_gather(_h(ctx), int(n_nodes), int(blocks), int(steps),
                                    _dev(sink, torch.float32, "sink"), _stream(stream)), "scoot_probe_gather", _h(ctx))


def scoot_status_string(status: int) -> str:
    return lib().scoot_status_string(int(status)).decode()


class Context:
    """A scoot_ctx bound to one CUDA device."""

    def __init__(self, device: int = 0):
        self.device = int(device)
        self.handle = scoot_ctx_create(self.device)

    def close(self):
        if self.handle:
            scoot_ctx_destroy(self.handle)
            self.handle = None

    def check(self, stream=None):
        scoot_ctx_check(self.handle, stream)

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def _h(ctx):
    return ctx.handle if isinstance(ctx, Context) else ctx


# ------------------------------------------------------------------ host-side preparation

def scoot_gp_layout_init(h_space, n: int, n_obj: int, kernel: int = MATERN52) -> scoot_gp_layout:
    L = scoot_gp_layout()
    _check(lib().scoot_gp_layout_init(_host(h_space, 16, name="h_space"), int(n), int(len(h_space)), int(n_obj),
                                      int(kernel), C.byref(L)), "scoot_gp_layout_init")
    return L


def scoot_gp_prepare(h_space, h_x_obs, h_y, h_lengthscale, h_signal_var, h_noise_var, layout):
    """Returns (host blob uint8[layout.bytes], cond float64[M])."""
    blob = np.zeros(layout.bytes, np.uint8)
    cond = np.zeros(layout.n_obj, np.float64)
    _check(lib().scoot_gp_prepare(_host(h_space, 16, name="h_space"), _host(h_x_obs, 4, name="h_x_obs"),
                                  int(h_x_obs.shape[1]), _host(h_y, dtype=np.float32, name="h_y"),
                                  _host(h_lengthscale, dtype=np.float32, name="h_lengthscale"),
                                  _host(h_signal_var, dtype=np.float32, name="h_signal_var"),
                                  _host(h_noise_var, dtype=np.float32, name="h_noise_var"),
                                  C.byref(layout), _host(blob), _host(cond)), "scoot_gp_prepare")
    return blob, cond


def scoot_gp_prepare_warped(h_space, h_x_obs, h_y, h_lengthscale, h_signal_var, h_noise_var, h_warp, layout):
    """scoot_gp_prepare with Kumaraswamy input warping h_warp float32 [M][d][2]."""
    blob = np.zeros(layout.bytes, np.uint8)
    cond = np.zeros(layout.n_obj, np.float64)
    _check(lib().scoot_gp_prepare_warped(_host(h_space, 16, name="h_space"), _host(h_x_obs, 4, name="h_x_obs"),
                                         int(h_x_obs.shape[1]), _host(h_y, dtype=np.float32, name="h_y"),
                                         _host(h_lengthscale, dtype=np.float32, name="h_lengthscale"),
                                         _host(h_signal_var, dtype=np.float32, name="h_signal_var"),
                                         _host(h_noise_var, dtype=np.float32, name="h_noise_var"),
                                         _host(np.ascontiguousarray(h_warp, np.float32), dtype=np.float32,
                                               name="h_warp"),
                                         C.byref(layout), _host(blob), _host(cond)), "scoot_gp_prepare_warped")
    return blob, cond


def scoot_forest_layout_init(h_nodes, h_tree_offset, d: int, leaf_scale: int) -> scoot_forest_layout:
    L = scoot_forest_layout()
    _check(lib().scoot_forest_layout_init(_host(h_nodes, 8, name="h_nodes"),
                                          _host(h_tree_offset, dtype=np.int32, name="h_tree_offset"),
                                          int(len(h_tree_offset) - 1), int(d), int(leaf_scale), C.byref(L)),
           "scoot_forest_layout_init")
    return L


def scoot_forest_pack(layout, h_nodes, h_tree_offset) -> np.ndarray:
    blob = np.zeros(layout.bytes, np.uint8)
    _check(lib().scoot_forest_pack(C.byref(layout), _host(h_nodes, 8, name="h_nodes"),
                                   _host(h_tree_offset, dtype=np.int32, name="h_tree_offset"), _host(blob)),
           "scoot_forest_pack")
    return blob


def scoot_boxes_build(h_y, h_ref, cap: int = 4096):
    """h_y float32 [M][n_pts], h_ref float32 [M] -> (lo [B][M], hi [B][M], front_size)."""
    M, n_pts = h_y.shape
    lo = np.zeros((max(cap, 1), M), np.float32)
    hi = np.zeros((max(cap, 1), M), np.float32)
    nb, fs = _i32(), _i32()
    _check(lib().scoot_boxes_build(_host(h_y, dtype=np.float32, name="h_y"), int(n_pts), int(M),
                                   _host(h_ref, dtype=np.float32, name="h_ref"), int(cap), _host(lo), _host(hi),
                                   C.byref(nb), C.byref(fs)), "scoot_boxes_build")
    return lo[:nb.value].copy(), hi[:nb.value].copy(), int(fs.value)


def scoot_boxes_index(h_lo, h_hi, grid_cap: int = 256):
    """Boxes [B][M] -> (grid float32 [M][grid_cap], n_grid int32 [M], corner uint32 [B][M])."""
    B, M = h_lo.shape
    grid = np.zeros((M, max(grid_cap, 1)), np.float32)
    n_grid = np.zeros(M, np.int32)
    corner = np.zeros((max(B, 1), M), np.uint32)
    _check(lib().scoot_boxes_index(_host(np.ascontiguousarray(h_lo), dtype=np.float32, name="h_lo"),
                                   _host(np.ascontiguousarray(h_hi), dtype=np.float32, name="h_hi"), int(B), int(M),
                                   int(grid_cap), _host(grid), _host(n_grid), _host(corner)), "scoot_boxes_index")
    return grid, n_grid, corner[:B].copy()


def scoot_round_state_build(h_space, h_x_obs, h_y, h_lengthscale, h_signal_var, h_noise_var, h_nodes,
                            h_tree_offset, leaf_scale: int, buf, kernel: int = 0, warp=None, boxes: int = 0,
                            h_ref=None, h_eps=None, grid_cap: int = 0, gp_on_device: bool = False,
                            fantasy_q: int = 0):
    """A round's host state packed into the host uint8 array buf (pinned
    staging memory; see include/scoot.h).  Returns the scoot_round_state, or
    None when buf is too small (the size needed is then in .bytes of the
    second return value).  Every array is kept alive by the caller for the
    duration of the call."""
    M, n = h_y.shape
    keep = [np.ascontiguousarray(h_y, np.float32), np.ascontiguousarray(h_lengthscale, np.float32),
            np.ascontiguousarray(h_signal_var, np.float32), np.ascontiguousarray(h_noise_var, np.float32)]
    inp = scoot_round_inputs()
    inp.space = _host(h_space, 16, name="h_space")
    inp.d = len(h_space)
    inp.x_obs = _host(h_x_obs, 4, name="h_x_obs")
    inp.ld_obs = int(h_x_obs.shape[1])
    inp.n, inp.n_obj = int(n), int(M)
    inp.y, inp.lengthscale, inp.signal_var, inp.noise_var = (_host(a) for a in keep)
    if warp is not None:
        keep.append(np.ascontiguousarray(warp, np.float32))
        inp.warp = _host(keep[-1])
    inp.kernel = int(kernel)
    inp.gp_on_device = int(bool(gp_on_device))
    inp.nodes = _host(h_nodes, 8, name="h_nodes")
    inp.tree_offset = _host(h_tree_offset, dtype=np.int32, name="h_tree_offset")
    inp.n_trees = int(len(h_tree_offset) - 1)
    inp.leaf_scale = int(leaf_scale)
    inp.boxes = int(boxes)
    if boxes:
        keep.append(np.ascontiguousarray(h_ref, np.float32))
        inp.ref = _host(keep[-1])
    if boxes == 1:
        keep.append(np.ascontiguousarray(h_eps, np.float32))
        inp.eps = _host(keep[-1])
        inp.n_mc = int(keep[-1].shape[0])
    inp.grid_cap = int(grid_cap)
    if fantasy_q:
        if not boxes:
            keep.append(np.ascontiguousarray(h_ref, np.float32))
            inp.ref = _host(keep[-1])
        inp.fantasy_q = int(fantasy_q)
    out = scoot_round_state()
    st = lib().scoot_round_state_build(C.byref(inp), _host(buf), int(buf.nbytes), C.byref(out))
    if st == -2 and out.bytes > buf.nbytes:  # SCOOT_ENOMEM: the buffer is too small
        return None, out
    _check(st, "scoot_round_state_build")
    return out, out


# ------------------------------------------------------------------ device calls

def scoot_prune(ctx, h_space, h_clauses, cand, n, mask, n_feasible=None, stream=None):
    import torch
    _check(lib().scoot_prune(_h(ctx), _host(h_space, 16, name="h_space"), int(len(h_space)),
                             _host(h_clauses, 80, name="h_clauses"), int(len(h_clauses)),
                             _dev(cand, torch.int32, "cand"), int(n), int(cand.shape[1]),
                             _dev(mask, torch.uint8, "mask"), _dev(n_feasible, torch.int64, "n_feasible"),
                             _stream(stream)), "scoot_prune", _h(ctx))


def scoot_rf_predict(ctx, layout, forest, h_space, cand, n, delta_num, delta_den, votes, mask=None,
                     n_feasible=None, stream=None):
    import torch
    _check(lib().scoot_rf_predict(_h(ctx), C.byref(layout), _dev(forest, torch.uint8, "forest"),
                                  _host(h_space, 16, name="h_space"), _dev(cand, torch.int32, "cand"),
                                  int(n), int(cand.shape[1]), int(delta_num), int(delta_den),
                                  _dev(votes, torch.int32, "votes"), _dev(mask, torch.uint8, "mask"),
                                  _dev(n_feasible, torch.int64, "n_feasible"), _stream(stream)),
           "scoot_rf_predict", _h(ctx))


def scoot_gp_posterior(ctx, layout, state, cand, n, mean, var, mask=None, stream=None):
    import torch
    _check(lib().scoot_gp_posterior(_h(ctx), C.byref(layout), _dev(state, torch.uint8, "state"),
                                    _dev(cand, torch.int32, "cand"), int(n), int(cand.shape[1]),
                                    _dev(mask, torch.uint8, "mask"), _dev(mean, torch.float32, "mean"),
                                    _dev(var, torch.float32, "var"), int(mean.shape[-1]), _stream(stream)),
           "scoot_gp_posterior", _h(ctx))


def scoot_acq_ei(ctx, mean, var, n, y_best, xi, acq, mask=None, stream=None):
    import torch
    _check(lib().scoot_acq_ei(_h(ctx), _dev(mean, torch.float32, "mean"), _dev(var, torch.float32, "var"),
                              _dev(mask, torch.uint8, "mask"), int(n), float(y_best), float(xi),
                              _dev(acq, torch.float32, "acq"), _stream(stream)), "scoot_acq_ei", _h(ctx))


def scoot_acq_ehvi(ctx, mean, var, n, box_lo, box_hi, eps, acq, mask=None, stream=None):
    import torch
    M = int(mean.shape[0])
    _check(lib().scoot_acq_ehvi(_h(ctx), _dev(mean, torch.float32, "mean"), _dev(var, torch.float32, "var"),
                                int(mean.shape[1]), M, _dev(mask, torch.uint8, "mask"), int(n),
                                _dev(box_lo, torch.float32, "box_lo"), _dev(box_hi, torch.float32, "box_hi"),
                                int(box_lo.shape[0]), _dev(eps, torch.float32, "eps"), int(eps.shape[0]),
                                _dev(acq, torch.float32, "acq"), _stream(stream)), "scoot_acq_ehvi", _h(ctx))


def scoot_acq_ehvi_exact(ctx, mean, var, n, grid, h_n_grid, corner, acq, mask=None, stream=None):
    """grid: float32 [M][grid_cap], h_n_grid: host int32 [M], corner: [B][M] (int32 view of uint32)."""
    import torch
    M = int(mean.shape[0])
    n_grid = np.ascontiguousarray(h_n_grid, np.int32)
    _check(lib().scoot_acq_ehvi_exact(_h(ctx), _dev(mean, torch.float32, "mean"), _dev(var, torch.float32, "var"),
                                      int(mean.shape[1]), M, _dev(mask, torch.uint8, "mask"), int(n),
                                      _dev(grid, torch.float32, "grid"), int(grid.shape[1]), _host(n_grid),
                                      _dev(corner, torch.int32, "corner"), int(corner.shape[0]),
                                      _dev(acq, torch.float32, "acq"), _stream(stream)), "scoot_acq_ehvi_exact", _h(ctx))


def scoot_score_ehvi_exact(ctx, layout, state, cand, n, grid, h_n_grid, corner, acq, mask=None, stream=None):
    import torch
    n_grid = np.ascontiguousarray(h_n_grid, np.int32)
    _check(lib().scoot_score_ehvi_exact(_h(ctx), C.byref(layout), _dev(state, torch.uint8, "state"),
                                        _dev(cand, torch.int32, "cand"), int(n), int(cand.shape[1]),
                                        _dev(mask, torch.uint8, "mask"), _dev(grid, torch.float32, "grid"),
                                        int(grid.shape[1]), _host(n_grid), _dev(corner, torch.int32, "corner"),
                                        int(corner.shape[0]), _dev(acq, torch.float32, "acq"), _stream(stream)),
           "scoot_score_ehvi_exact", _h(ctx))


def scoot_score_ei(ctx, layout, state, cand, n, xi, acq, mask=None, stream=None):
    import torch
    _check(lib().scoot_score_ei(_h(ctx), C.byref(layout), _dev(state, torch.uint8, "state"),
                                _dev(cand, torch.int32, "cand"), int(n), int(cand.shape[1]),
                                _dev(mask, torch.uint8, "mask"), float(xi), _dev(acq, torch.float32, "acq"),
                                _stream(stream)), "scoot_score_ei", _h(ctx))


def scoot_score_ehvi(ctx, layout, state, cand, n, box_lo, box_hi, eps, acq, mask=None, stream=None):
    import torch
    _check(lib().scoot_score_ehvi(_h(ctx), C.byref(layout), _dev(state, torch.uint8, "state"),
                                  _dev(cand, torch.int32, "cand"), int(n), int(cand.shape[1]),
                                  _dev(mask, torch.uint8, "mask"), _dev(box_lo, torch.float32, "box_lo"),
                                  _dev(box_hi, torch.float32, "box_hi"), int(box_lo.shape[0]),
                                  _dev(eps, torch.float32, "eps"), int(eps.shape[0]),
                                  _dev(acq, torch.float32, "acq"), _stream(stream)), "scoot_score_ehvi", _h(ctx))


def scoot_select_topq(ctx, acq, n, q, idx, val, count, mask=None, stream=None):
    import torch
    _check(lib().scoot_select_topq(_h(ctx), _dev(acq, torch.float32, "acq"), _dev(mask, torch.uint8, "mask"),
                                   int(n), int(q), _dev(idx, torch.int64, "idx"), _dev(val, torch.float32, "val"),
                                   _dev(count, torch.int32, "count"), _stream(stream)), "scoot_select_topq", _h(ctx))


def scoot_acq_mace(ctx, mean, var, n, y_best, xi, kappa, acq, mask=None, stream=None):
    """acq: float32 [3][lda] (rows UCB, PI, EI)."""
    import torch
    _check(lib().scoot_acq_mace(_h(ctx), _dev(mean, torch.float32, "mean"), _dev(var, torch.float32, "var"),
                                _dev(mask, torch.uint8, "mask"), int(n), float(y_best), float(xi), float(kappa),
                                _dev(acq, torch.float32, "acq"), int(acq.shape[-1]), _stream(stream)),
           "scoot_acq_mace", _h(ctx))


def scoot_score_mace(ctx, layout, state, cand, n, xi, kappa, acq, mask=None, stream=None):
    """acq: float32 [3][lda] (rows UCB, PI, EI)."""
    import torch
    _check(lib().scoot_score_mace(_h(ctx), C.byref(layout), _dev(state, torch.uint8, "state"),
                                  _dev(cand, torch.int32, "cand"), int(n), int(cand.shape[1]),
                                  _dev(mask, torch.uint8, "mask"), float(xi), float(kappa),
                                  _dev(acq, torch.float32, "acq"), int(acq.shape[-1]), _stream(stream)),
           "scoot_score_mace", _h(ctx))


def scoot_select_pareto(ctx, acq, n, k, seed, idx, count, mask=None, front=None, stream=None):
    """idx: int64 [k]; count: int32 [2] (picks, front size); front: optional int64 [cap]."""
    import torch
    _check(lib().scoot_select_pareto(_h(ctx), _dev(acq, torch.float32, "acq"), int(acq.shape[-1]),
                                     _dev(mask, torch.uint8, "mask"), int(n), int(k),
                                     C.c_uint64(int(seed) & 0xFFFFFFFFFFFFFFFF), _dev(idx, torch.int64, "idx"),
                                     _dev(count, torch.int32, "count"), _dev(front, torch.int64, "front"),
                                     int(front.shape[0]) if front is not None else 0, _stream(stream)),
           "scoot_select_pareto", _h(ctx))


def scoot_select_topq_static(acq, n, q, idx, val, count, mask=None, stream=None):
    """Top-q without a context and without allocating (see include/scoot.h):
    for callers that cannot allocate device memory when they select.  Calls
    that overlap on the GPU share one scratch array and must not be issued."""
    import torch
    _check(lib().scoot_select_topq_static(_dev(acq, torch.float32, "acq"), _dev(mask, torch.uint8, "mask"),
                                          int(n), int(q), _dev(idx, torch.int64, "idx"),
                                          _dev(val, torch.float32, "val"), _dev(count, torch.int32, "count"),
                                          _stream(stream)), "scoot_select_topq_static")


def scoot_sobol_configs(ctx, h_space, skip, n, cand, stream=None):
    """cand: int32 [d][ld] device tensor receiving Sobol points skip .. skip + n - 1."""
    import torch
    _check(lib().scoot_sobol_configs(_h(ctx), _host(h_space, 16, name="h_space"), len(h_space), int(skip), int(n),
                                     _dev(cand, torch.int32, "cand"), int(cand.shape[1]), _stream(stream)),
           "scoot_sobol_configs", _h(ctx))


def scoot_first_feasible(ctx, mask, n, need, idx, count, stream=None):
    import torch
    _check(lib().scoot_first_feasible(_h(ctx), _dev(mask, torch.uint8, "mask"), int(n), int(need),
                                      _dev(idx, torch.int64, "idx"), _dev(count, torch.int32, "count"),
                                      _stream(stream)), "scoot_first_feasible", _h(ctx))


def scoot_ucb_beta(t: int) -> float:
    v = C.c_double()
    _check(lib().scoot_ucb_beta(int(t), C.byref(v)), "scoot_ucb_beta")
    return float(v.value)


def scoot_standardize(h_y, ref_margin: float = 1e-3):
    """(standardised objectives float32 [M][n], reference point float32 [M])."""
    y = np.ascontiguousarray(h_y, np.float32)
    out = np.empty_like(y)
    ref = np.empty(y.shape[0], np.float32)
    _check(lib().scoot_standardize(_host(y), int(y.shape[0]), int(y.shape[1]), _host(out), _host(ref),
                                   float(ref_margin)), "scoot_standardize")
    return out, ref


def scoot_delta_update(delta: float, count: int, k: int, any_invalid: bool):
    """Returns the new (delta, count)."""
    d, c = C.c_double(delta), _i32(count)
    _check(lib().scoot_delta_update(C.byref(d), C.byref(c), int(k), int(bool(any_invalid))), "scoot_delta_update")
    return float(d.value), int(c.value)


def scoot_gp_device_work_bytes(layout) -> int:
    v = _i64()
    _check(lib().scoot_gp_device_work_bytes(C.byref(layout), C.byref(v)), "scoot_gp_device_work_bytes")
    return int(v.value)


def scoot_gp_prepare_device(ctx, h_space, layout, obs, y, lengthscale, signal_var, noise_var, blob, work=None,
                            warp=None, stream=None):
    """Device inputs: obs int32 [d][ld], y float32 [M][n], lengthscale float32
    [M][d], signal_var / noise_var float32 [M], warp float32 [M][d][2] or None;
    blob: uint8 device tensor of layout.bytes; work: uint8 device scratch of
    scoot_gp_device_work_bytes(layout) bytes (allocated here when None)."""
    import torch
    if work is None:
        work = torch.empty(scoot_gp_device_work_bytes(layout), dtype=torch.uint8, device=blob.device)
    _check(lib().scoot_gp_prepare_device(_h(ctx), _host(h_space, 16, name="h_space"), C.byref(layout),
                                         _dev(obs, torch.int32, "obs"), int(obs.shape[1]),
                                         _dev(y, torch.float32, "y"), _dev(lengthscale, torch.float32, "lengthscale"),
                                         _dev(signal_var, torch.float32, "signal_var"),
                                         _dev(noise_var, torch.float32, "noise_var"), _dev(warp, torch.float32, "warp"),
                                         _dev(blob, torch.uint8, "blob"), _dev(work, torch.uint8, "work"),
                                         int(work.numel()), _stream(stream)),
           "scoot_gp_prepare_device", _h(ctx))


def scoot_gp_mle_work_bytes(n: int, d: int, n_obj: int, n_starts: int) -> int:
    v = _i64()
    _check(lib().scoot_gp_mle_work_bytes(int(n), int(d), int(n_obj), int(n_starts), C.byref(v)),
           "scoot_gp_mle_work_bytes")
    return int(v.value)


def scoot_gp_mle(ctx, h_space, obs, n, y, theta0, h_lo, h_hi, free_mask, steps, lr, theta, lml, grad=None,
                 kernel=0, work=None, stream=None):
    """obs int32 [d][ld]; y float32 [M][n]; theta0 / theta float64 [S][M][d+2];
    lml float64 [S][M]; grad float64 [S][M][d+2] or None (all device);
    h_lo / h_hi host float64 [d+2]."""
    import torch
    S_, M = int(theta0.shape[0]), int(y.shape[0])
    d = len(h_space)
    if work is None:
        work = torch.empty(scoot_gp_mle_work_bytes(n, d, M, S_), dtype=torch.uint8, device=obs.device)
    lo = np.ascontiguousarray(h_lo, np.float64)
    hi = np.ascontiguousarray(h_hi, np.float64)
    _check(lib().scoot_gp_mle(_h(ctx), _host(h_space, 16, name="h_space"), d, _dev(obs, torch.int32, "obs"),
                              int(obs.shape[1]), int(n), _dev(y, torch.float32, "y"), M, int(kernel),
                              _dev(theta0, torch.float64, "theta0"), S_, _host(lo), _host(hi),
                              int(free_mask) & 0xFFFFFFFF, int(steps), float(lr), _dev(theta, torch.float64, "theta"),
                              _dev(lml, torch.float64, "lml"), _dev(grad, torch.float64, "grad"),
                              _dev(work, torch.uint8, "work"), int(work.numel()), _stream(stream)),
           "scoot_gp_mle", _h(ctx))


def scoot_gp_device_buffer_layout(layout, warped: bool):
    """(upload_bytes, blob_off, work_off, total_bytes)."""
    v = [_i64() for _ in range(4)]
    _check(lib().scoot_gp_device_buffer_layout(C.byref(layout), int(bool(warped)), *[C.byref(x) for x in v]),
           "scoot_gp_device_buffer_layout")
    return tuple(int(x.value) for x in v)


def scoot_gp_prepare_device_from_host(ctx, h_space, layout, h_x_obs, h_y, h_lengthscale, h_signal_var, h_noise_var,
                                      h_stage, buf, warp=None, stream=None):
    """h_stage: pinned uint8 host tensor; buf: uint8 device tensor (scoot_gp_device_buffer_layout)."""
    import torch
    _check(lib().scoot_gp_prepare_device_from_host(
        _h(ctx), _host(h_space, 16, name="h_space"), C.byref(layout), _host(h_x_obs, 4, name="h_x_obs"),
        int(h_x_obs.shape[1]), _host(h_y, dtype=np.float32, name="h_y"),
        _host(h_lengthscale, dtype=np.float32, name="h_lengthscale"),
        _host(h_signal_var, dtype=np.float32, name="h_signal_var"),
        _host(h_noise_var, dtype=np.float32, name="h_noise_var"),
        _host(warp, dtype=np.float32, name="warp") if warp is not None else None,
        _vp(h_stage.data_ptr()), _dev(buf, torch.uint8, "buf"), int(buf.numel()), _stream(stream)),
        "scoot_gp_prepare_device_from_host", _h(ctx))


def scoot_rf_train_work_bytes(n: int, d: int) -> int:
    v = _i64()
    _check(lib().scoot_rf_train_work_bytes(int(n), int(d), C.byref(v)), "scoot_rf_train_work_bytes")
    return int(v.value)


def scoot_rf_train(ctx, h_space, obs, n, labels, boot, max_depth, leaf_scale, nodes, n_nodes, work=None,
                   stream=None):
    """obs: int32 [d][ld] observation words; labels: uint8 [n]; boot: int32
    [T][m]; nodes: int64 [T][node_cap] receiving scoot_node records (view the
    host copy as the node dtype); n_nodes: int32 [T]; work: uint8 device
    scratch of scoot_rf_train_work_bytes(n, d) bytes (allocated here when None)."""
    import torch
    T, m = (int(boot.shape[0]), int(boot.shape[1])) if boot.dim() == 2 else (0, 1)
    if work is None:
        work = torch.empty(scoot_rf_train_work_bytes(n, len(h_space)), dtype=torch.uint8, device=obs.device)
    _check(lib().scoot_rf_train(_h(ctx), _host(h_space, 16, name="h_space"), len(h_space),
                                _dev(obs, torch.int32, "obs"), int(n), int(obs.shape[1]),
                                _dev(labels, torch.uint8, "labels"), _dev(boot, torch.int32, "boot"), T, m,
                                int(max_depth), int(leaf_scale), _dev(nodes, torch.int64, "nodes"),
                                int(nodes.shape[1]), _dev(n_nodes, torch.int32, "n_nodes"),
                                _dev(work, torch.uint8, "work"), int(work.numel()), _stream(stream)),
           "scoot_rf_train", _h(ctx))


def compact_forest(nodes: np.ndarray, n_nodes: np.ndarray):
    """Host copy of scoot_rf_train's output (int64 [T][node_cap], int32 [T])
    -> (scoot_node records of all trees back to back, tree offsets [T + 1])."""
    recs = np.ascontiguousarray(nodes).view(NODE_DTYPE)
    offs = np.zeros(len(n_nodes) + 1, np.int32)
    offs[1:] = np.cumsum(n_nodes)
    out = np.concatenate([recs[t, :int(c)] for t, c in enumerate(n_nodes)]) if len(n_nodes) else recs[:0, 0]
    return out, offs


def scoot_fantasy_state_bytes(layout, q: int) -> int:
    v = _i64()
    _check(lib().scoot_fantasy_state_bytes(C.byref(layout), int(q), C.byref(v)), "scoot_fantasy_state_bytes")
    return int(v.value)


def scoot_fantasy_prepare(h_space, h_x_obs, h_y, h_lengthscale, h_signal_var, h_noise_var, h_ref, q, layout):
    """The fp64 fantasy state (host uint8 array) and its box_cap."""
    out = np.zeros(scoot_fantasy_state_bytes(layout, q), np.uint8)
    box_cap = _i32()
    _check(lib().scoot_fantasy_prepare(
        _host(h_space, 16, name="h_space"), C.byref(layout), _host(h_x_obs, 4, name="h_x_obs"), int(h_x_obs.shape[1]),
        _host(h_y, dtype=np.float32, name="h_y"), _host(h_lengthscale, dtype=np.float32, name="h_lengthscale"),
        _host(h_signal_var, dtype=np.float32, name="h_signal_var"),
        _host(h_noise_var, dtype=np.float32, name="h_noise_var"), _host(h_ref, dtype=np.float32, name="h_ref"),
        int(q), _host(out), int(out.nbytes), C.byref(box_cap)), "scoot_fantasy_prepare")
    return out, int(box_cap.value)


def scoot_fantasy_work_bytes(layout, n: int, q: int, box_cap: int) -> int:
    v = _i64()
    _check(lib().scoot_fantasy_work_bytes(C.byref(layout), int(n), int(q), int(box_cap), C.byref(v)),
           "scoot_fantasy_work_bytes")
    return int(v.value)


def scoot_suggest_fantasy(ctx, layout, state, fant_state, box_cap, cand, n, eps, q, work, idx, val, count,
                          mask=None, var_out=None, stream=None):
    """q sequential fantasised picks into the device arrays idx (int64 [q]),
    val (float32 [q]) and count (int32 [1]); asynchronous on stream."""
    import torch
    _check(lib().scoot_suggest_fantasy(
        _h(ctx), C.byref(layout), _dev(state, torch.uint8, "state"), _dev(fant_state, torch.uint8, "fant_state"),
        int(box_cap), _dev(cand, torch.int32, "cand"), int(n), int(cand.shape[1]), _dev(mask, torch.uint8, "mask"),
        _dev(eps, torch.float32, "eps"), int(eps.shape[0]), int(q), _vp(work.data_ptr()), int(work.numel()),
        _dev(idx, torch.int64, "idx"), _dev(val, torch.float32, "val"), _dev(count, torch.int32, "count"),
        _dev(var_out, torch.float32, "var_out"), _stream(stream)),
        "scoot_suggest_fantasy", _h(ctx))


FANT_REC = 9  # SCOOT_FANT_REC: 64-bit words of a shard's record


def scoot_fantasy_begin(ctx, layout, state, fant_state, box_cap, cand, n, eps, q, work, idx, val, count, mask=None,
                        index_offset=0, stream=None):
    import torch
    _check(lib().scoot_fantasy_begin(
        _h(ctx), C.byref(layout), _dev(state, torch.uint8, "state"), _dev(fant_state, torch.uint8, "fant_state"),
        int(box_cap), _dev(cand, torch.int32, "cand"), int(n), int(cand.shape[1]), _dev(mask, torch.uint8, "mask"),
        int(index_offset), _dev(eps, torch.float32, "eps"), int(eps.shape[0]), int(q), _vp(work.data_ptr()),
        int(work.numel()), _dev(idx, torch.int64, "idx"), _dev(val, torch.float32, "val"),
        _dev(count, torch.int32, "count"), _stream(stream)), "scoot_fantasy_begin", _h(ctx))


def scoot_fantasy_local_best(ctx, j, rec=None, stream=None):
    """rec: device int64 [FANT_REC] (the uint64 record's bits) or None."""
    import torch
    _check(lib().scoot_fantasy_local_best(_h(ctx), int(j), _dev(rec, torch.int64, "rec"), _stream(stream)),
           "scoot_fantasy_local_best", _h(ctx))


def scoot_fantasy_commit(ctx, j, recs, stream=None):
    """recs: device int64 [n_rec][FANT_REC], the gathered records."""
    import torch
    _check(lib().scoot_fantasy_commit(_h(ctx), int(j), _dev(recs, torch.int64, "recs"), int(recs.shape[0]),
                                      _stream(stream)), "scoot_fantasy_commit", _h(ctx))


def scoot_fantasy_end(ctx, var_out=None, stream=None):
    import torch
    _check(lib().scoot_fantasy_end(_h(ctx), _dev(var_out, torch.float32, "var_out"), _stream(stream)),
           "scoot_fantasy_end", _h(ctx))

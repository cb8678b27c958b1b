"""ctypes binding of libmoara (declarations in include/moara.h).

Argument marshalling only: every function below forwards to the C entry point
of the same name.  Device buffers are passed as integer addresses (e.g. a
torch tensor's ``data_ptr()``) and streams as ``cudaStream_t`` handles
(``torch.cuda.Stream.cuda_stream``).  There is no fallback: if the shared
library is missing, importing this module raises.
"""

from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmoara.so")

MOARA_OK = 0
MOARA_ERR_INVALID_ARG = -1
MOARA_ERR_SHAPE = -2
MOARA_ERR_RANK = -3
MOARA_ERR_ALIGN = -4
MOARA_ERR_UNKNOWN_MODULE = -5
MOARA_ERR_CUDA = -6
MOARA_ERR_DEVICE_TIMEOUT = -7
MOARA_ERR_WORKSPACE = -8
MOARA_ERR_UNSUPPORTED = -9

MOARA_DTYPE_F32 = 0
MOARA_DTYPE_BF16 = 1
MOARA_REFRESH_SRC_V = 0
MOARA_REFRESH_SRC_G = 1
MOARA_PREC_AUTO = 0
MOARA_PREC_FP32 = 1
MOARA_PREC_BF16_TC = 2
MOARA_PROJ_LEFT = 0
MOARA_PROJ_SMALLER = 1
MOARA_DRULE_N = 0
MOARA_DRULE_MAX = 1
MODULE_BITS = {"q": 0, "k": 1, "v": 2, "o": 3, "gate": 4, "up": 5, "down": 6}


class moara_hparams(ctypes.Structure):
    _fields_ = [
        ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
        ("adam_eps", ctypes.c_float), ("decomp_eps", ctypes.c_float),
        ("scale", ctypes.c_float),
        ("block_size", ctypes.c_int), ("refresh_interval", ctypes.c_int),
        ("decompose", ctypes.c_int), ("refresh_src", ctypes.c_int),
        ("oversample", ctypes.c_int), ("power_iters", ctypes.c_int),
        ("ritz_iters", ctypes.c_int), ("precision", ctypes.c_int),
        ("seed", ctypes.c_uint64),
        ("clip_norm", ctypes.c_float),
        ("state_dtype", ctypes.c_int),
        ("proj_rule", ctypes.c_int),
    ]


class moara_module_desc(ctypes.Structure):
    _fields_ = [
        ("m", ctypes.c_int), ("n", ctypes.c_int), ("r", ctypes.c_int),
        ("grad_dtype", ctypes.c_int),
        ("W", ctypes.c_void_p), ("P", ctypes.c_void_p), ("P_bf16", ctypes.c_void_p),
        ("exp_avg", ctypes.c_void_p), ("exp_avg_sq", ctypes.c_void_p),
        ("mag_avg", ctypes.c_void_p), ("mag_avg_sq", ctypes.c_void_p),
        ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t),
    ]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(
            f"libmoara.so not found at {LIB_PATH}; build it with "
            "`python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32, i64, f32, sz = (ctypes.c_void_p, ctypes.c_int, ctypes.c_int64,
                             ctypes.c_float, ctypes.c_size_t)
    P = ctypes.POINTER
    sig = {
        "moara_default_hparams": (i32, [P(moara_hparams)]),
        "moara_create": (i32, [P(vp), P(moara_hparams), i32]),
        "moara_destroy": (None, [vp]),
        "moara_get_hparams": (i32, [vp, P(moara_hparams)]),
        "moara_state_bytes": (i32, [i32, i32, i32, i32, i32, i32, i32, i32, P(sz)]),
        "moara_rank_table": (i32, [i32, ctypes.c_uint32, ctypes.c_uint32, i32, P(i32)]),
        "moara_workspace_bytes": (i32, [i32, i32, i32, i32, P(sz)]),
        "moara_init_module": (i32, [vp, P(moara_module_desc), P(i32)]),
        "moara_load_projector": (i32, [vp, i32, vp, vp]),
        "moara_refresh_workspace_bytes": (i32, [vp, i32, i32, i32, P(sz)]),
        "moara_set_refresh_workspace": (i32, [vp, vp, sz]),
        "moara_refresh_projector": (i32, [vp, i32, P(i32), P(vp), vp]),
        "moara_step_grouped": (i32, [vp, i32, P(i32), P(vp), i64, f32, i32, vp]),
        "moara_step_grouped_host": (i32, [vp, i32, P(i32), P(vp), i64, f32, i32, sz, vp]),
        "moara_alignment": (i32, [vp, i32, P(i32), P(vp), vp, vp]),
        "moara_set_clip_extra": (i32, [vp, vp]),
        "moara_clip_state": (i32, [vp, P(vp)]),
        "moara_flatten_shape": (i32, [i32, P(ctypes.c_int64), P(i32), P(i32)]),
        "moara_get_device_status": (i32, [vp, P(i32), vp]),
        "moara_last_error": (ctypes.c_char_p, [vp]),
        "moara_status_string": (ctypes.c_char_p, [i32]),
        "moara_launch_count": (i64, [vp]),
        "moara_set_wait_limit": (i32, [vp, i64]),
        "moara_profile_enable": (i32, [vp, i32]),
        "moara_profile_read": (i32, [vp, P(ctypes.c_double), P(i64)]),
        "moara_step_static_scratch": (i32, [P(moara_hparams), i32, i32, i32, i32, vp, vp, vp, vp,
                                            vp, vp, vp, i64, f32, vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = _load()
lib = _lib


class MoaraError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"{msg} (status {code}: {moara_status_string(code)})")
        self.code = code


def _check(code, ctx=None, what=""):
    if code != MOARA_OK:
        detail = moara_last_error(ctx) if ctx is not None else ""
        raise MoaraError(code, f"{what}: {detail}" if detail else what)
    return code


# --------------------------------------------------------------- entry points
def moara_status_string(code):
    return _lib.moara_status_string(int(code)).decode()


def moara_last_error(ctx):
    return _lib.moara_last_error(ctx).decode()


def moara_default_hparams():
    hp = moara_hparams()
    _check(_lib.moara_default_hparams(ctypes.byref(hp)), what="moara_default_hparams")
    return hp


def moara_create(hp, device=0):
    """Returns an opaque context handle (int)."""
    h = ctypes.c_void_p()
    _check(_lib.moara_create(ctypes.byref(h), ctypes.byref(hp), int(device)), what="moara_create")
    return h.value


def moara_destroy(ctx):
    _lib.moara_destroy(ctx)


def moara_get_hparams(ctx):
    hp = moara_hparams()
    _check(_lib.moara_get_hparams(ctx, ctypes.byref(hp)), ctx, "moara_get_hparams")
    return hp


def moara_state_bytes(m, n, r, block_size, b_V, b_M, d_rule=MOARA_DRULE_N, decompose=1):
    out = ctypes.c_size_t()
    _check(_lib.moara_state_bytes(m, n, r, block_size, b_V, b_M, d_rule, decompose,
                                  ctypes.byref(out)), what="moara_state_bytes")
    return out.value


def moara_rank_table(r_base, donor_mask, receiver_mask, delta_r):
    out = (ctypes.c_int * 7)()
    _check(_lib.moara_rank_table(r_base, donor_mask, receiver_mask, delta_r, out),
           what="moara_rank_table")
    return list(out)


def moara_workspace_bytes(m, n, r, block_size):
    out = ctypes.c_size_t()
    _check(_lib.moara_workspace_bytes(m, n, r, block_size, ctypes.byref(out)),
           what="moara_workspace_bytes")
    return out.value


def moara_init_module(ctx, desc):
    mid = ctypes.c_int()
    _check(_lib.moara_init_module(ctx, ctypes.byref(desc), ctypes.byref(mid)), ctx,
           "moara_init_module")
    return mid.value


def moara_load_projector(ctx, module_id, P_src, stream=0):
    _check(_lib.moara_load_projector(ctx, module_id, P_src, stream), ctx, "moara_load_projector")


def moara_refresh_workspace_bytes(ctx, m, n, r):
    out = ctypes.c_size_t()
    _check(_lib.moara_refresh_workspace_bytes(ctx, m, n, r, ctypes.byref(out)), ctx,
           "moara_refresh_workspace_bytes")
    return out.value


def moara_set_refresh_workspace(ctx, ptr, nbytes):
    _check(_lib.moara_set_refresh_workspace(ctx, ptr, nbytes), ctx, "moara_set_refresh_workspace")


def _arrays(ids, grads):
    n = len(ids)
    ia = (ctypes.c_int * n)(*[int(i) for i in ids])
    ga = (ctypes.c_void_p * n)(*[int(g) for g in grads])
    return n, ia, ga


def moara_refresh_projector(ctx, ids, grads, stream=0):
    n, ia, ga = _arrays(ids, grads)
    _check(_lib.moara_refresh_projector(ctx, n, ia, ga, stream), ctx, "moara_refresh_projector")


def moara_step_grouped(ctx, ids, grads, t, lr, auto_refresh=False, stream=0):
    n, ia, ga = _arrays(ids, grads)
    _check(_lib.moara_step_grouped(ctx, n, ia, ga, int(t), float(lr), int(bool(auto_refresh)),
                                   stream), ctx, "moara_step_grouped")


def moara_step_grouped_host(ctx, ids, host_grads, t, lr, auto_refresh=False,
                            chunk_bytes=256 << 20, stream=0):
    """host_grads: addresses of page-locked host gradients (one per id)."""
    n, ia, ga = _arrays(ids, host_grads)
    _check(_lib.moara_step_grouped_host(ctx, n, ia, ga, int(t), float(lr), int(bool(auto_refresh)),
                                        int(chunk_bytes), stream), ctx, "moara_step_grouped_host")


def moara_alignment(ctx, ids, grads, S_out, stream=0):
    """S_out: device address of len(ids) floats."""
    n, ia, ga = _arrays(ids, grads)
    _check(_lib.moara_alignment(ctx, n, ia, ga, S_out, stream), ctx, "moara_alignment")


def moara_set_clip_extra(ctx, extra_sq_ptr):
    """extra_sq_ptr: device address of a float (sum of squares of other
    gradients), or 0 for none."""
    _check(_lib.moara_set_clip_extra(ctx, extra_sq_ptr or None), ctx, "moara_set_clip_extra")


def moara_clip_state(ctx):
    """Device address of the context's {total norm, coefficient} floats."""
    out = ctypes.c_void_p()
    _check(_lib.moara_clip_state(ctx, ctypes.byref(out)), ctx, "moara_clip_state")
    return out.value


def moara_flatten_shape(shape):
    """(m, n) of the N-D flatten rule for a gradient of this shape."""
    shp = (ctypes.c_int64 * len(shape))(*[int(x) for x in shape])
    m, n = ctypes.c_int(), ctypes.c_int()
    _check(_lib.moara_flatten_shape(len(shape), shp, ctypes.byref(m), ctypes.byref(n)),
           what="moara_flatten_shape")
    return m.value, n.value


def moara_get_device_status(ctx, stream=0):
    st = ctypes.c_int()
    _check(_lib.moara_get_device_status(ctx, ctypes.byref(st), stream), ctx,
           "moara_get_device_status")
    return st.value


def moara_launch_count(ctx):
    return int(_lib.moara_launch_count(ctx))


def moara_set_wait_limit(ctx, cycles):
    _check(_lib.moara_set_wait_limit(ctx, int(cycles)), ctx, "moara_set_wait_limit")


def moara_step_static_scratch(hp, m, n, r, grad_dtype, G, W, P, exp_avg, exp_avg_sq,
                              mag_avg, mag_avg_sq, t, lr, stream=0):
    """Single-module step with the library's built-in scratch (no device
    allocation); returns the status code instead of raising."""
    return _lib.moara_step_static_scratch(ctypes.byref(hp), m, n, r, grad_dtype, G, W, P,
                                          exp_avg, exp_avg_sq, mag_avg, mag_avg_sq,
                                          int(t), float(lr), stream)


PHASES = ["decompose", "project", "backproject", "refresh", "tc_project",
          "tc_backproject", "tc_decompose", "tc_refresh", "tc_decompose_overlap", "clip_norm"]


def moara_profile_enable(ctx, enable=True):
    _check(_lib.moara_profile_enable(ctx, int(bool(enable))), ctx, "moara_profile_enable")


def moara_profile_read(ctx):
    """{phase name: (milliseconds, launches)} since the last read."""
    ms = (ctypes.c_double * len(PHASES))()
    n = (ctypes.c_int64 * len(PHASES))()
    _check(_lib.moara_profile_read(ctx, ms, n), ctx, "moara_profile_read")
    return {PHASES[i]: (ms[i], n[i]) for i in range(len(PHASES))}


EXPORTED = [
    "moara_default_hparams", "moara_create", "moara_destroy", "moara_get_hparams",
    "moara_state_bytes", "moara_rank_table", "moara_workspace_bytes", "moara_init_module",
    "moara_load_projector", "moara_refresh_workspace_bytes", "moara_set_refresh_workspace",
    "moara_refresh_projector", "moara_step_grouped", "moara_step_grouped_host",
    "moara_get_device_status", "moara_alignment", "moara_set_clip_extra", "moara_clip_state",
    "moara_flatten_shape",
    "moara_last_error", "moara_status_string", "moara_launch_count", "moara_set_wait_limit",
    "moara_profile_enable", "moara_profile_read", "moara_step_static_scratch",
]

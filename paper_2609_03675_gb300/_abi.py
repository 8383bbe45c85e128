"""ctypes view of the C ABI in include/cofie_ngff.h (argument marshalling only).

Loads ``libcofie_ngff.so`` from this package directory. There is no fallback:
if the library has not been built, loading it (the first NGFF or QER handle
created) fails with an error that says how to build it.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libcofie_ngff.so")

OK, EINVAL, ENOMEM, ECUDA, ETIMEOUT, EDEVICE = 0, 1, 2, 3, 4, 5
KEEP_DROP, KEEP_NOVELTY, KEEP_GAP, KEEP_FIRST, KEEP_SCENE = 0, 1, 2, 3, 4
MAX_BINS, MAX_LMAX, MAX_BATCH = 256, 256, 64
SIGNAL_HISTOGRAM, SIGNAL_LOWRES, SIGNAL_DHASH, SIGNAL_SCD = 0, 1, 2, 3

# Every symbol include/cofie_ngff.h declares.
EXPORTS = (
    "cofie_ngff_default_params",
    "cofie_ngff_feature_words",
    "cofie_ngff_create",
    "cofie_ngff_destroy",
    "cofie_ngff_push",
    "cofie_ngff_push_ex",
    "cofie_ngff_push_batch",
    "cofie_ngff_candidates",
    "cofie_ngff_candidates_from_keep",
    "cofie_ngff_gather",
    "cofie_ngff_reset",
    "cofie_ngff_state_bytes",
    "cofie_ngff_state_save",
    "cofie_ngff_state_load",
    "cofie_ngff_shard_prepare",
    "cofie_ngff_shard_commit",
    "cofie_ngff_status",
    "cofie_ngff_frames_seen",
    "cofie_ngff_debug_bins",
    "cofie_ngff_debug_fail_alloc",
    "cofie_ngff_checked_build",
    "cofie_ngff_debug_wait",
    "cofie_ngff_profile_reset",
    "cofie_ngff_profile_read",
    "cofie_ngff_select_static",
    "cofie_ngff_last_error",
    "cofie_ngff_global_error",
    "cofie_qer_create",
    "cofie_qer_destroy",
    "cofie_qer_run",
    "cofie_qer_status",
    "cofie_qer_kernel_in_use",
    "cofie_qer_profile_reset",
    "cofie_qer_profile_read",
    "cofie_qer_last_error",
)


class Params(ctypes.Structure):
    _fields_ = [
        ("width", ctypes.c_uint32),
        ("height", ctypes.c_uint32),
        ("bins", ctypes.c_uint32),
        ("l_max", ctypes.c_uint32),
        ("m_min", ctypes.c_uint32),
        ("tau", ctypes.c_float),
        ("luma_w", ctypes.c_uint32 * 3),
        ("luma_den", ctypes.c_uint32),
        ("max_streams", ctypes.c_uint32),
        ("max_frames_per_push", ctypes.c_uint32),
        ("device", ctypes.c_int32),
        ("host_stage_bytes", ctypes.c_uint64),
        ("signal", ctypes.c_uint32),
        ("scd_cut", ctypes.c_float),
        ("scd_gradual", ctypes.c_float),
        ("max_stream_frames", ctypes.c_uint32),
    ]


class PushDesc(ctypes.Structure):
    _fields_ = [
        ("stream", ctypes.c_uint32),
        ("n", ctypes.c_uint32),
        ("frames", ctypes.c_void_p),
        ("scores_out", ctypes.c_void_p),
        ("keep_out", ctypes.c_void_p),
    ]


class Profile(ctypes.Structure):
    _fields_ = [
        ("hist_launches", ctypes.c_uint64),
        ("select_launches", ctypes.c_uint64),
        ("hist_bytes", ctypes.c_uint64),
        ("hist_timed", ctypes.c_uint64),
        ("hist_ms", ctypes.c_double),
        ("select_timed", ctypes.c_uint64),
        ("select_ms", ctypes.c_double),
        ("other_launches", ctypes.c_uint64),
    ]


class QerParams(ctypes.Structure):
    _fields_ = [
        ("n_text", ctypes.c_uint32),
        ("n_heads", ctypes.c_uint32),
        ("n_kv_heads", ctypes.c_uint32),
        ("head_dim", ctypes.c_uint32),
        ("max_frames", ctypes.c_uint32),
        ("tokens_per_frame", ctypes.c_uint32),
        ("rho", ctypes.c_float),
        ("device", ctypes.c_int32),
        ("kernel", ctypes.c_uint32),
    ]


QER_KERNEL_AUTO, QER_KERNEL_ONE_SM, QER_KERNEL_PAIR = 0, 1, 2


class NGFFError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"cofie_ngff error {code}: {message}")
        self.code = code


_lib = None


def load():
    """The loaded library (ctypes.CDLL) with prototypes set."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: the CUDA library has not been built "
                           "(run `python -c 'import __graft_entry__ as g; g.build()'`)")
    lib = ctypes.CDLL(LIB_PATH)
    vp, u32, u64 = ctypes.c_void_p, ctypes.c_uint32, ctypes.c_uint64
    P = ctypes.POINTER(Params)
    H = ctypes.c_void_p
    lib.cofie_ngff_default_params.argtypes = [P, u32, u32]
    lib.cofie_ngff_default_params.restype = None
    lib.cofie_ngff_feature_words.argtypes = [H]
    lib.cofie_ngff_feature_words.restype = u32
    lib.cofie_ngff_create.argtypes = [P, ctypes.POINTER(H)]
    lib.cofie_ngff_create.restype = ctypes.c_int
    lib.cofie_ngff_destroy.argtypes = [H]
    lib.cofie_ngff_destroy.restype = None
    lib.cofie_ngff_push.argtypes = [H, u32, vp, u32, vp, vp, vp]
    lib.cofie_ngff_push.restype = ctypes.c_int
    lib.cofie_ngff_push_ex.argtypes = [H, u32, vp, u32, vp, vp, vp, vp]
    lib.cofie_ngff_push_ex.restype = ctypes.c_int
    lib.cofie_ngff_push_batch.argtypes = [H, ctypes.POINTER(PushDesc), u32, vp]
    lib.cofie_ngff_push_batch.restype = ctypes.c_int
    lib.cofie_ngff_candidates.argtypes = [H, u32, vp, u32, vp, vp]
    lib.cofie_ngff_candidates.restype = ctypes.c_int
    lib.cofie_ngff_candidates_from_keep.argtypes = [H, vp, u32, vp, vp, vp]
    lib.cofie_ngff_candidates_from_keep.restype = ctypes.c_int
    lib.cofie_ngff_gather.argtypes = [H, vp, u32, vp, u32, vp, vp]
    lib.cofie_ngff_gather.restype = ctypes.c_int
    lib.cofie_ngff_state_bytes.argtypes = [H]
    lib.cofie_ngff_state_bytes.restype = ctypes.c_size_t
    lib.cofie_ngff_state_save.argtypes = [H, u32, vp, vp]
    lib.cofie_ngff_state_save.restype = ctypes.c_int
    lib.cofie_ngff_state_load.argtypes = [H, u32, vp, vp]
    lib.cofie_ngff_state_load.restype = ctypes.c_int
    lib.cofie_ngff_shard_prepare.argtypes = [H, u32, vp, u32, u32, u64, vp, vp]
    lib.cofie_ngff_shard_prepare.restype = ctypes.c_int
    lib.cofie_ngff_shard_commit.argtypes = [H, u32, u32, vp, vp, vp]
    lib.cofie_ngff_shard_commit.restype = ctypes.c_int
    lib.cofie_ngff_reset.argtypes = [H, u32, vp]
    lib.cofie_ngff_reset.restype = ctypes.c_int
    lib.cofie_ngff_status.argtypes = [H, vp]
    lib.cofie_ngff_status.restype = ctypes.c_int
    lib.cofie_ngff_frames_seen.argtypes = [H, u32, ctypes.POINTER(u64)]
    lib.cofie_ngff_frames_seen.restype = ctypes.c_int
    lib.cofie_ngff_debug_bins.argtypes = [H, vp, u64, vp, vp]
    lib.cofie_ngff_debug_bins.restype = ctypes.c_int
    lib.cofie_ngff_checked_build.argtypes = []
    lib.cofie_ngff_checked_build.restype = ctypes.c_int
    lib.cofie_ngff_debug_fail_alloc.argtypes = [ctypes.c_int32]
    lib.cofie_ngff_debug_fail_alloc.restype = None
    lib.cofie_ngff_debug_wait.argtypes = [H, u64, vp]
    lib.cofie_ngff_debug_wait.restype = ctypes.c_int
    lib.cofie_ngff_profile_reset.argtypes = [H, ctypes.c_int]
    lib.cofie_ngff_profile_reset.restype = ctypes.c_int
    lib.cofie_ngff_profile_read.argtypes = [H, ctypes.POINTER(Profile)]
    lib.cofie_ngff_profile_read.restype = ctypes.c_int
    lib.cofie_ngff_select_static.argtypes = [P, vp, u32, vp, vp, ctypes.c_char_p, ctypes.c_size_t, vp]
    lib.cofie_ngff_select_static.restype = ctypes.c_int
    lib.cofie_qer_create.argtypes = [ctypes.POINTER(QerParams), ctypes.POINTER(H)]
    lib.cofie_qer_create.restype = ctypes.c_int
    lib.cofie_qer_destroy.argtypes = [H]
    lib.cofie_qer_destroy.restype = None
    lib.cofie_qer_run.argtypes = [H, vp, vp, u32, vp, vp, vp, vp]
    lib.cofie_qer_run.restype = ctypes.c_int
    lib.cofie_qer_status.argtypes = [H, vp]
    lib.cofie_qer_status.restype = ctypes.c_int
    lib.cofie_qer_kernel_in_use.argtypes = [H]
    lib.cofie_qer_kernel_in_use.restype = ctypes.c_uint32
    lib.cofie_qer_profile_reset.argtypes = [H, ctypes.c_int]
    lib.cofie_qer_profile_reset.restype = ctypes.c_int
    pu64 = ctypes.POINTER(ctypes.c_uint64)
    pdbl = ctypes.POINTER(ctypes.c_double)
    lib.cofie_qer_profile_read.argtypes = [H, pu64, pu64, pdbl, pdbl, pdbl]
    lib.cofie_qer_profile_read.restype = ctypes.c_int
    lib.cofie_qer_last_error.argtypes = [H]
    lib.cofie_qer_last_error.restype = ctypes.c_char_p
    lib.cofie_ngff_last_error.argtypes = [H]
    lib.cofie_ngff_last_error.restype = ctypes.c_char_p
    lib.cofie_ngff_global_error.argtypes = []
    lib.cofie_ngff_global_error.restype = ctypes.c_char_p
    _lib = lib
    return lib

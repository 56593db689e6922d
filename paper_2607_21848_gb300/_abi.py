"""ctypes mirror of include/crc.h and loader for the in-tree libcrc.so.

There is no fallback: if the library is missing or fails to load, every call
raises.  Build it with `python -m paper_2607_21848_gb300.build`.
"""

from __future__ import annotations

import ctypes as C
import os

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libcrc.so")

CRC_OK = 0
CRC_ERR_INVALID_ARG = 1
CRC_ERR_SHAPE = 2
CRC_ERR_UNSUPPORTED = 3
CRC_ERR_CUDA = 4
CRC_ERR_DEVICE = 5
CRC_ERR_TOO_LARGE = 6
CRC_NOALLOC_SCRATCH_BYTES = 65536

CRC_F32 = 0
CRC_BF16 = 1

CRC_SEG_SINK = 0
CRC_SEG_RETRIEVED = 1
CRC_SEG_WINDOW = 2
CRC_SEG_CURRENT = 3

CRC_MAX_SEGMENTS = 16
CRC_MAX_FRAMES = 4
CRC_MAX_K = 8
CRC_MAX_ROPE_PAIRS = 64

CRC_ATTN_DEFAULT = 0
CRC_ATTN_SIMT = 1
CRC_ATTN_GAUSSIAN = 2
CRC_ATTN_SKIP_FAR = 4
CRC_ATTN_BIAS_DIRECT = 8
CRC_ATTN_FRAME_CAUSAL = 16


class crc_frame(C.Structure):
    _fields_ = [("K", C.c_double * 9), ("R", C.c_double * 9), ("c", C.c_double * 3)]


class crc_shape(C.Structure):
    _fields_ = [("L", C.c_int32), ("H", C.c_int32), ("d", C.c_int32), ("F", C.c_int32), ("h", C.c_int32),
                ("w", C.c_int32), ("dtype", C.c_int32)]


class crc_tensor(C.Structure):
    _fields_ = [("data", C.c_void_p), ("stride_layer", C.c_int64), ("stride_token", C.c_int64),
                ("stride_head", C.c_int64)]


class crc_segment(C.Structure):
    _fields_ = [("offset", C.c_int32), ("length", C.c_int32), ("kind", C.c_int32), ("slot", C.c_int32)]


class crc_cache(C.Structure):
    _fields_ = [("k", crc_tensor), ("v", crc_tensor), ("n_keys", C.c_int32), ("nseg", C.c_int32),
                ("seg", crc_segment * CRC_MAX_SEGMENTS)]


class crc_bank(C.Structure):
    _fields_ = [("capacity", C.c_int32), ("num_slabs", C.c_int32), ("frames", C.c_void_p), ("centre", C.c_void_p),
                ("view", C.c_void_p), ("depth", C.c_void_p), ("kv", C.c_void_p), ("slab_chunk", C.c_void_p)]


class crc_retrieval(C.Structure):
    _fields_ = [("E", C.c_double), ("w_v", C.c_double), ("tau_c", C.c_double), ("cos_tau_v", C.c_double),
                ("delta", C.c_int32), ("k", C.c_int32), ("ext_first", C.c_int32), ("ext_min", C.c_int32),
                ("exclude_sink", C.c_int32)]


class crc_rope(C.Structure):
    _fields_ = [("channel0", C.c_int32), ("pairs", C.c_int32), ("interleaved", C.c_int32), ("pos_slot0", C.c_int32),
                ("pos_stride", C.c_int32), ("frame_pos0", C.c_int32), ("theta", C.c_double)]


class crc_step(C.Structure):
    _fields_ = [("n", C.c_int32), ("window_offset", C.c_int32), ("ext_first", C.c_int32),
                ("rope_pos_slot0", C.c_int32), ("seg_length", C.c_int32 * CRC_MAX_SEGMENTS),
                ("frames", crc_frame * CRC_MAX_FRAMES)]


class crc_step_plan(C.Structure):
    _fields_ = [("shape", crc_shape), ("bank", crc_bank), ("cache", crc_cache), ("retrieval", crc_retrieval),
                ("rope", crc_rope), ("eps", C.c_float), ("lam", C.c_float), ("sigma", C.c_float),
                ("attn_flags", C.c_int32), ("d_depth", C.c_void_p), ("d_k", C.c_void_p), ("d_v", C.c_void_p),
                ("q", crc_tensor), ("o", crc_tensor), ("d_lse", C.c_void_p), ("d_idx", C.c_void_p),
                ("d_score", C.c_void_p), ("d_count", C.c_void_p), ("d_uv", C.c_void_p), ("d_cell", C.c_void_p),
                ("d_valid", C.c_void_p), ("d_status", C.c_void_p), ("d_workspace", C.c_void_p),
                ("workspace_bytes", C.c_size_t)]


CRC_STEP_BAD_DESCRIPTOR = 100

_P = C.POINTER
_SIGS = {
    "crc_version": (C.c_char_p, []),
    "crc_status_string": (C.c_char_p, [C.c_int32]),
    "crc_last_cuda_error": (C.c_int32, []),
    "crc_bank_insert_poses": (C.c_int32, [_P(crc_bank), _P(crc_shape), C.c_int32, C.c_int32, _P(crc_frame),
                                          C.c_void_p]),
    "crc_cache_update": (C.c_int32, [_P(crc_bank), _P(crc_shape), C.c_int32, _P(crc_frame), C.c_void_p, C.c_void_p,
                                     C.c_void_p, _P(crc_cache), C.c_int32, C.c_void_p]),
    "crc_retrieve": (C.c_int32, [_P(crc_bank), C.c_int32, _P(crc_shape), _P(crc_frame), C.c_int32,
                                 _P(crc_retrieval), _P(crc_cache), _P(crc_rope), C.c_void_p, C.c_void_p, C.c_void_p,
                                 C.c_void_p, C.c_size_t, C.c_void_p]),
    "crc_retrieve_workspace_size": (C.c_size_t, [C.c_int32, C.c_int32]),
    "crc_retrieve_noalloc": (C.c_int32, [_P(crc_bank), C.c_int32, _P(crc_shape), _P(crc_frame), C.c_int32,
                                         _P(crc_retrieval), _P(crc_cache), _P(crc_rope), C.c_void_p, C.c_void_p,
                                         C.c_void_p, C.c_void_p]),
    "crc_gather": (C.c_int32, [_P(crc_shape), C.c_void_p, C.c_int32, C.c_void_p, C.c_int32, _P(crc_cache),
                               _P(crc_rope), C.c_void_p]),
    "crc_correspond": (C.c_int32, [_P(crc_shape), _P(crc_frame), C.c_void_p, _P(crc_bank), C.c_void_p, C.c_void_p,
                                   C.c_int32, C.c_float, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "crc_biased_attention": (C.c_int32, [_P(crc_shape), crc_tensor, _P(crc_cache), crc_tensor, C.c_void_p, C.c_int32,
                                         C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p, C.c_float, C.c_float,
                                         C.c_int32, C.c_void_p, C.c_void_p]),
    "crc_bias_expansion_bound": (C.c_double, [C.c_float, C.c_float, C.c_int32, C.c_int32]),
    "crc_chunk_step": (C.c_int32, [_P(crc_step_plan), C.c_void_p, C.c_void_p]),
    "crc_host_copy": (C.c_int32, [C.c_void_p, C.c_void_p, C.c_size_t, C.c_int32, C.c_void_p]),
}

EXPORTED = tuple(_SIGS)

_lib = None


def lib_path() -> str:
    return _LIB_PATH


def load() -> C.CDLL:
    """Load libcrc.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"{_LIB_PATH} is missing: build it with `python -m paper_2607_21848_gb300.build`")
        lib = C.CDLL(_LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


class CrcError(RuntimeError):
    def __init__(self, fn: str, status: int):
        lib = load()
        msg = lib.crc_status_string(status).decode()
        if status == CRC_ERR_CUDA:
            msg += f" (cudaError {lib.crc_last_cuda_error()})"
        super().__init__(f"{fn}: {msg}")
        self.status = status


def check(fn: str, status: int) -> None:
    if status != CRC_OK:
        raise CrcError(fn, status)

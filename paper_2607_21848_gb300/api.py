"""Python binding of the C ABI (argument marshalling only).

Every function has the name of its C entry point and forwards to it; all
arithmetic of the path runs in the CUDA kernels of libcrc.so.  PyTorch supplies
device memory (tensors) and the current CUDA stream.  `Bank` and `Cache` are
conveniences that allocate the caller-owned device buffers the C ABI expects.
"""

from __future__ import annotations

import ctypes as C
import math
from typing import Iterable, Optional, Sequence, Tuple

import numpy as np
import torch

from . import _abi
from ._abi import CrcError  # noqa: F401

SEG_SINK = _abi.CRC_SEG_SINK
SEG_RETRIEVED = _abi.CRC_SEG_RETRIEVED
SEG_WINDOW = _abi.CRC_SEG_WINDOW
SEG_CURRENT = _abi.CRC_SEG_CURRENT
ATTN_DEFAULT = _abi.CRC_ATTN_DEFAULT
ATTN_SIMT = _abi.CRC_ATTN_SIMT
ATTN_GAUSSIAN = _abi.CRC_ATTN_GAUSSIAN
ATTN_SKIP_FAR = _abi.CRC_ATTN_SKIP_FAR
ATTN_BIAS_DIRECT = _abi.CRC_ATTN_BIAS_DIRECT
ATTN_FRAME_CAUSAL = _abi.CRC_ATTN_FRAME_CAUSAL


def _dtype_code(dt: torch.dtype) -> int:
    if dt == torch.float32:
        return _abi.CRC_F32
    if dt == torch.bfloat16:
        return _abi.CRC_BF16
    raise ValueError(f"unsupported dtype {dt}")


def _stream(stream: Optional[torch.cuda.Stream]) -> C.c_void_p:
    s = stream if stream is not None else torch.cuda.current_stream()
    return C.c_void_p(s.cuda_stream)


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    return t.data_ptr()


def shape(L: int, H: int, d: int, F: int, h: int, w: int, dtype: torch.dtype) -> _abi.crc_shape:
    return _abi.crc_shape(L, H, d, F, h, w, _dtype_code(dtype))


def frames_struct(records: np.ndarray):
    """[N, 21] fp64 records (K 9, R 9, c 3) -> ctypes array of crc_frame."""
    rec = np.ascontiguousarray(records, dtype=np.float64).reshape(-1, 21)
    arr = (_abi.crc_frame * rec.shape[0])()
    C.memmove(arr, rec.ctypes.data, rec.nbytes)
    return arr


def tensor_view(t: torch.Tensor) -> _abi.crc_tensor:
    """crc_tensor of a [L, N, H, d] tensor with a contiguous last dimension."""
    if t.dim() != 4 or t.stride(3) != 1:
        raise ValueError("expected a [L, N, H, d] tensor with contiguous d")
    return _abi.crc_tensor(_ptr(t), t.stride(0), t.stride(1), t.stride(2))


def crc_retrieve_workspace_size(bank_count: int, k: int) -> int:
    return int(_abi.load().crc_retrieve_workspace_size(bank_count, k))


class Bank:
    """Device memory of the chunk bank (frames, pose summaries, depth, K/V slabs).

    track_slabs: keep the chunk held by each K/V slab (crc_bank.slab_chunk), so that
    retrieval never returns a chunk whose slab a newer chunk has overwritten.  The
    bank also owns the retrieval workspace for its capacity (crc_retrieve)."""

    def __init__(self, capacity: int, F: int, h: int, w: int, L: int, H: int, d: int, dtype: torch.dtype,
                 num_slabs: int, device="cuda", with_kv: bool = True, track_slabs: bool = False):
        self.capacity, self.F, self.h, self.w = capacity, F, h, w
        self.L, self.H, self.d, self.dtype, self.num_slabs = L, H, d, dtype, num_slabs
        self.frames = torch.zeros(capacity, F, 21, dtype=torch.float64, device=device)
        self.centre = torch.zeros(capacity, 3, dtype=torch.float64, device=device)
        self.view = torch.zeros(capacity, 3, dtype=torch.float64, device=device)
        self.depth = torch.zeros(capacity, F, h, w, dtype=torch.float32, device=device)
        self.kv = (torch.zeros(num_slabs, 2, L, F * h * w, H, d, dtype=dtype, device=device)
                   if with_kv else None)
        self.slab_chunk = (torch.full((num_slabs,), -1, dtype=torch.int32, device=device)
                           if track_slabs and with_kv else None)
        ws = crc_retrieve_workspace_size(capacity, _abi.CRC_MAX_K)
        self.workspace = torch.empty(max(ws, 16), dtype=torch.uint8, device=device) if ws else None

    def struct(self) -> _abi.crc_bank:
        return _abi.crc_bank(self.capacity, self.num_slabs, _ptr(self.frames), _ptr(self.centre), _ptr(self.view),
                             _ptr(self.depth), _ptr(self.kv) if self.kv is not None else None,
                             _ptr(self.slab_chunk))


class Cache:
    """Segmented clean KV cache [L, n_keys, H, d] with its segment table."""

    def __init__(self, k: torch.Tensor, v: torch.Tensor, segments: Sequence[Tuple[int, int, int, int]]):
        self.k, self.v = k, v
        self.segments = [tuple(int(x) for x in s) for s in segments]

    @classmethod
    def empty(cls, L: int, n_keys: int, H: int, d: int, dtype: torch.dtype, segments, device="cuda"):
        k = torch.zeros(L, n_keys, H, d, dtype=dtype, device=device)
        v = torch.zeros_like(k)
        return cls(k, v, segments)

    @property
    def n_keys(self) -> int:
        return self.k.shape[1]

    def heads(self, h0: int, count: int) -> "Cache":
        """The same cache restricted to heads [h0, h0 + count): strided views, same segments."""
        return Cache(head_view(self.k, h0, count), head_view(self.v, h0, count), self.segments)

    def struct(self) -> _abi.crc_cache:
        c = _abi.crc_cache()
        c.k = tensor_view(self.k)
        c.v = tensor_view(self.v)
        c.n_keys = self.n_keys
        if len(self.segments) > _abi.CRC_MAX_SEGMENTS:
            raise ValueError("too many segments")
        c.nseg = len(self.segments)
        for i, (off, length, kind, slot) in enumerate(self.segments):
            c.seg[i] = _abi.crc_segment(off, length, kind, slot)
        return c


def head_range(H: int, rank: int, world: int) -> Tuple[int, int]:
    """Heads [h0, h0 + count) of rank `rank` when H heads are split over `world` ranks as
    evenly as possible (heads are independent in Eq. 2, so each rank runs its own range
    with its own bank and cache views; nothing is exchanged)."""
    if world < 1 or not 0 <= rank < world or H < world:
        raise ValueError("need 0 <= rank < world <= H")
    base, extra = divmod(H, world)
    h0 = rank * base + min(rank, extra)
    return h0, base + (1 if rank < extra else 0)


def head_view(t: torch.Tensor, h0: int, count: int) -> torch.Tensor:
    """Heads [h0, h0 + count) of a [L, N, H, d] tensor, as a strided view of the same memory."""
    return t[:, :, h0:h0 + count, :]


def retrieval_params(E: float, w_v: float, tau_c: float, cos_tau_v: float, delta: int, k: int,
                     ext_first: int = -1, ext_min: int = 0, exclude_sink: bool = False) -> _abi.crc_retrieval:
    return _abi.crc_retrieval(E, w_v, tau_c, cos_tau_v, delta, k, ext_first, ext_min, int(bool(exclude_sink)))


def rope_params(channel0: int, pairs: int, theta: float, interleaved: bool, pos_slot0: int, pos_stride: int,
                frame_pos0: int = 0) -> _abi.crc_rope:
    """Temporal RoPE re-positioning of gathered keys (crc_rope in include/crc.h)."""
    return _abi.crc_rope(channel0, pairs, int(bool(interleaved)), pos_slot0, pos_stride, frame_pos0, float(theta))


def crc_chunk_step(plan: _abi.crc_step_plan, d_step: torch.Tensor, stream=None) -> None:
    """One chunk step with its per-step values read from the device descriptor d_step
    (a uint8 tensor holding one crc_step)."""
    if d_step.numel() * d_step.element_size() < C.sizeof(_abi.crc_step):
        raise ValueError("d_step is smaller than a crc_step")
    _abi.check("crc_chunk_step", _abi.load().crc_chunk_step(C.byref(plan), _ptr(d_step), _stream(stream)))


def crc_bias_expansion_bound(lam: float, sigma: float, h: int, w: int) -> float:
    return float(_abi.load().crc_bias_expansion_bound(lam, sigma, h, w))


def crc_version() -> str:
    return _abi.load().crc_version().decode()


def crc_bank_insert_poses(bank: Bank, shp: _abi.crc_shape, first: int, frames: np.ndarray, stream=None) -> None:
    lib = _abi.load()
    fr = frames_struct(frames)
    count = len(fr) // shp.F
    b = bank.struct()
    _abi.check("crc_bank_insert_poses",
               lib.crc_bank_insert_poses(C.byref(b), C.byref(shp), first, count, fr, _stream(stream)))


def crc_cache_update(bank: Bank, shp: _abi.crc_shape, chunk: int, frames: np.ndarray, depth: torch.Tensor,
                     k_new: Optional[torch.Tensor], v_new: Optional[torch.Tensor], cache: Optional[Cache],
                     window_offset: int, stream=None) -> None:
    lib = _abi.load()
    fr = frames_struct(frames)
    b = bank.struct()
    cs = cache.struct() if cache is not None else None
    _abi.check("crc_cache_update",
               lib.crc_cache_update(C.byref(b), C.byref(shp), chunk, fr, _ptr(depth), _ptr(k_new), _ptr(v_new),
                                    C.byref(cs) if cs is not None else None, window_offset, _stream(stream)))


def crc_retrieve(bank: Bank, bank_count: int, shp: _abi.crc_shape, cur_frames: np.ndarray, n: int,
                 params: _abi.crc_retrieval, cache: Optional[Cache], idx: torch.Tensor, score: Optional[torch.Tensor],
                 count: torch.Tensor, stream=None, rope: Optional[_abi.crc_rope] = None,
                 workspace: Optional[torch.Tensor] = None) -> None:
    """`workspace` defaults to the bank's own (sized for its capacity)."""
    lib = _abi.load()
    fr = frames_struct(cur_frames)
    b = bank.struct()
    cs = cache.struct() if cache is not None else None
    ws = bank.workspace if workspace is None else workspace
    _abi.check("crc_retrieve",
               lib.crc_retrieve(C.byref(b), bank_count, C.byref(shp), fr, n, C.byref(params),
                                C.byref(cs) if cs is not None else None, C.byref(rope) if rope is not None else None,
                                _ptr(idx), _ptr(score), _ptr(count), _ptr(ws),
                                0 if ws is None else ws.numel() * ws.element_size(), _stream(stream)))


def crc_retrieve_noalloc(bank: Bank, bank_count: int, shp: _abi.crc_shape, cur_frames: np.ndarray, n: int,
                         params: _abi.crc_retrieval, cache: Optional[Cache], idx: torch.Tensor,
                         score: Optional[torch.Tensor], count: torch.Tensor, stream=None,
                         rope: Optional[_abi.crc_rope] = None) -> None:
    """crc_retrieve with the library's fixed scratch in place of a workspace, for callers
    that cannot allocate device memory (see include/crc.h)."""
    lib = _abi.load()
    fr = frames_struct(cur_frames)
    b = bank.struct()
    cs = cache.struct() if cache is not None else None
    _abi.check("crc_retrieve_noalloc",
               lib.crc_retrieve_noalloc(C.byref(b), bank_count, C.byref(shp), fr, n, C.byref(params),
                                        C.byref(cs) if cs is not None else None,
                                        C.byref(rope) if rope is not None else None, _ptr(idx), _ptr(score),
                                        _ptr(count), _stream(stream)))


def crc_gather(shp: _abi.crc_shape, pool: torch.Tensor, idx: torch.Tensor, k: int, cache: Cache,
               rope: Optional[_abi.crc_rope] = None, stream=None) -> None:
    """Mirror the retrieved slots d_idx of a step into a second cache from its own slab pool
    `pool` [num_slabs, 2, L, N_c, H, d]."""
    lib = _abi.load()
    if pool.dim() != 6 or not pool.is_contiguous():
        raise ValueError("expected a dense [num_slabs, 2, L, N_c, H, d] slab pool")
    cs = cache.struct()
    _abi.check("crc_gather",
               lib.crc_gather(C.byref(shp), _ptr(pool), pool.shape[0], _ptr(idx), k, C.byref(cs),
                              C.byref(rope) if rope is not None else None, _stream(stream)))


def crc_host_copy(dst: torch.Tensor, src: torch.Tensor, stream=None, blocks: int = 0) -> None:
    """Copy src into dst (same number of bytes, both contiguous) with the GPU's SMs;
    either side may be a CUDA tensor or a pinned CPU tensor."""
    lib = _abi.load()
    if not (dst.is_contiguous() and src.is_contiguous()):
        raise ValueError("expected contiguous tensors")
    nbytes = dst.numel() * dst.element_size()
    if nbytes != src.numel() * src.element_size():
        raise ValueError("dst and src differ in size")
    _abi.check("crc_host_copy", lib.crc_host_copy(dst.data_ptr(), src.data_ptr(), nbytes, blocks, _stream(stream)))


def crc_correspond(shp: _abi.crc_shape, cur_frames: np.ndarray, depth: torch.Tensor, bank: Bank, idx: torch.Tensor,
                   count: Optional[torch.Tensor], k: int, eps: float, uv: torch.Tensor, cell: Optional[torch.Tensor],
                   valid: torch.Tensor, stream=None) -> None:
    lib = _abi.load()
    fr = frames_struct(cur_frames)
    b = bank.struct()
    _abi.check("crc_correspond",
               lib.crc_correspond(C.byref(shp), fr, _ptr(depth), C.byref(b), _ptr(idx), _ptr(count), k,
                                  float(eps), _ptr(uv), _ptr(cell), _ptr(valid), _stream(stream)))


def crc_biased_attention(shp: _abi.crc_shape, q: torch.Tensor, cache: Cache, o: torch.Tensor,
                         lse: Optional[torch.Tensor], uv: Optional[torch.Tensor], valid: Optional[torch.Tensor], k: int,
                         slot_chunk: Optional[torch.Tensor], lam: float, sigma: float, flags: int = 0,
                         status: Optional[torch.Tensor] = None, stream=None) -> None:
    lib = _abi.load()
    cs = cache.struct()
    _abi.check("crc_biased_attention",
               lib.crc_biased_attention(C.byref(shp), tensor_view(q), C.byref(cs), tensor_view(o), _ptr(lse),
                                        q.shape[1], _ptr(uv), _ptr(valid), k, _ptr(slot_chunk), float(lam),
                                        float(sigma), flags, _ptr(status), _stream(stream)))

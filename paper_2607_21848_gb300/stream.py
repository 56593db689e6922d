"""Chunk-step driver for a long autoregressive stream (host-side bookkeeping only).

Cache layout (Sec. 4.2): [sink | retrieved slot 0 .. k-1 | window ring 0 .. W-1],
each region one chunk (N_c tokens) long.  The first chunk becomes the sink and is
never evicted; chunk n >= 1 goes into window ring slot n % W, evicting the chunk
W steps older; every chunk's poses and depth stay in the bank, and its K/V as long as
its slab (chunk % num_slabs) is not reused.  One step n runs, on one stream and
without any host synchronisation:

  crc_cache_update    chunk n's K/V, depth and poses enter the window and the bank
  crc_retrieve        Eq. 1 over chunks 0..n, gates (distance, angle, gap delta),
                      top-k gather into the retrieved slots; an empty admissible set
                      extends the window with the next-older chunks n-W, n-W-1, ...
  crc_gather          (optional) the same slots into the control-branch cache
  crc_correspond      Eq. 3-4 for every query of chunk n in every retrieved frame
  crc_biased_attention  Eq. 2 over all layers of the call

With `rope_pairs` > 0 the retrieved chunks' keys (cached with their rotary
embedding at the frame positions where they were produced, frame f of chunk j at
j F + f) are re-packed at the positions just before the recent window: slot r
at (n - W + 1 - k + r) F + f at step n (Sec. 4.2 "Cache packing").

Everything numeric happens in the CUDA kernels; this module only decides which
cache region each chunk occupies and which segments are live at step n.
"""

from __future__ import annotations

import dataclasses
from typing import List, Optional, Tuple

import numpy as np
import torch

from . import api


@dataclasses.dataclass
class StreamConfig:
    L: int
    H: int
    d: int
    F: int
    h: int
    w: int
    k: int
    window: int  # chunks in the recent window (the current chunk included)
    capacity: int  # chunks the bank can hold
    num_slabs: int  # K/V slabs; with fewer than `capacity`, only the newest num_slabs chunks can be retrieved
    E: float
    w_v: float
    tau_c: float
    cos_tau_v: float
    delta: int
    lam: float
    sigma: float
    eps: float
    dtype: torch.dtype = torch.bfloat16
    # temporal RoPE re-positioning of retrieved keys (0 pairs: off)
    rope_pairs: int = 0
    rope_channel0: int = 0
    rope_theta: float = 10000.0
    rope_interleaved: bool = True
    # control-branch mirror cache with its own layer count (0: none)
    control_L: int = 0

    @property
    def Nc(self) -> int:
        return self.F * self.h * self.w

    @property
    def n_keys(self) -> int:
        return (1 + self.k + self.window) * self.Nc


class ChunkStream:
    """Owns the bank, the segmented cache and the per-step scratch outputs."""

    def __init__(self, cfg: StreamConfig, device="cuda"):
        self.cfg = cfg
        c = cfg
        self.shape = api.shape(c.L, c.H, c.d, c.F, c.h, c.w, c.dtype)
        # the bank records which chunk each K/V slab holds: with fewer slabs than chunks, a chunk
        # whose slab a newer chunk overwrote is never retrieved
        self.bank = api.Bank(c.capacity, c.F, c.h, c.w, c.L, c.H, c.d, c.dtype, c.num_slabs, device=device,
                             track_slabs=True)
        self.cache = api.Cache.empty(c.L, c.n_keys, c.H, c.d, c.dtype, [], device=device)
        self.idx = torch.full((c.k,), -1, dtype=torch.int32, device=device)
        self.score = torch.zeros(c.k, dtype=torch.float64, device=device)
        self.count = torch.zeros(1, dtype=torch.int32, device=device)
        S = c.k * c.F
        self.uv = torch.zeros(c.Nc, S, 2, dtype=torch.float32, device=device)
        self.cell = torch.zeros(c.Nc, S, dtype=torch.int32, device=device)
        self.valid = torch.zeros(c.Nc, S, dtype=torch.uint8, device=device)
        self.status = torch.zeros(1, dtype=torch.int32, device=device)
        self.params = api.retrieval_params(c.E, c.w_v, c.tau_c, c.cos_tau_v, c.delta, c.k)
        self.control_shape = None
        if c.control_L > 0:
            # the control branch keeps its own slab pool and cache; poses and depth live in the main bank
            self.control_shape = api.shape(c.control_L, c.H, c.d, c.F, c.h, c.w, c.dtype)
            self.control_bank = api.Bank(c.capacity, c.F, c.h, c.w, c.control_L, c.H, c.d, c.dtype, c.num_slabs,
                                         device=device, track_slabs=True)
            self.control_cache = api.Cache.empty(c.control_L, c.n_keys, c.H, c.d, c.dtype, [], device=device)

    # ---- checkpoint -------------------------------------------------------
    def state_dict(self) -> dict:
        """Everything a later step reads: the bank (poses, pose summaries, depth, K/V
        slabs), the cache and, if present, the control branch's pool and cache.  The
        step index is the caller's (segments and ring slots follow from it).  The
        tensors are the stream's own; save or clone them before stepping on."""
        sd = {"bank." + k: getattr(self.bank, k) for k in ("frames", "centre", "view", "depth", "kv", "slab_chunk")}
        sd["cache.k"], sd["cache.v"] = self.cache.k, self.cache.v
        if self.control_shape is not None:
            sd["control_bank.kv"] = self.control_bank.kv
            sd["control_cache.k"], sd["control_cache.v"] = self.control_cache.k, self.control_cache.v
        return sd

    def load_state_dict(self, sd: dict) -> None:
        """Restore a state_dict() of a stream with the same configuration."""
        own = self.state_dict()
        if set(own) != set(sd):
            raise ValueError(f"state keys differ: {sorted(set(own) ^ set(sd))}")
        for k, t in own.items():
            if tuple(t.shape) != tuple(sd[k].shape) or t.dtype != sd[k].dtype:
                raise ValueError(f"{k}: expected {tuple(t.shape)} {t.dtype}")
            t.copy_(sd[k])

    # ---- layout -----------------------------------------------------------
    def slot_offset(self, r: int) -> int:
        return (1 + r) * self.cfg.Nc

    def window_offset(self, q: int) -> int:
        return (1 + self.cfg.k + q) * self.cfg.Nc

    def segments(self, n: int) -> List[Tuple[int, int, int, int]]:
        """Live segments at step n (after chunk n has been written)."""
        c = self.cfg
        segs = [(0, c.Nc, api.SEG_SINK, 0)]
        for r in range(c.k):
            segs.append((self.slot_offset(r), c.Nc, api.SEG_RETRIEVED, r))
        for q in range(c.window):
            # ring slot q holds the newest chunk m in [1, n] with m % window == q
            present = any(m >= 1 and m % c.window == q for m in range(max(1, n - c.window + 1), n + 1))
            segs.append((self.window_offset(q), c.Nc if present else 0, api.SEG_WINDOW, q))
        return segs

    def rope(self, n: int):
        """Re-positioning of step n: slot r just before the window's oldest chunk."""
        c = self.cfg
        if c.rope_pairs <= 0:
            return None
        first_window_chunk = max(1, n - c.window + 1)
        return api.rope_params(c.rope_channel0, c.rope_pairs, c.rope_theta, c.rope_interleaved,
                               pos_slot0=(first_window_chunk - c.k) * c.F, pos_stride=c.F, frame_pos0=0)

    def ext_first(self, n: int) -> int:
        """Newest chunk that is neither in the window nor the sink (-1 if none)."""
        e = n - self.cfg.window
        return e if e >= 1 else -1

    # ---- one chunk step ---------------------------------------------------
    def step(self, n: int, frames: np.ndarray, depth: torch.Tensor, k_new: torch.Tensor, v_new: torch.Tensor,
             q: torch.Tensor, o: torch.Tensor, lse: Optional[torch.Tensor] = None, stream=None,
             k_ctl: Optional[torch.Tensor] = None, v_ctl: Optional[torch.Tensor] = None) -> None:
        c = self.cfg
        woff = 0 if n == 0 else self.window_offset(n % c.window)
        self.cache.segments = self.segments(n)
        api.crc_cache_update(self.bank, self.shape, n, frames, depth, k_new, v_new, self.cache, woff, stream)
        if self.control_shape is not None:
            self.control_cache.segments = self.cache.segments
            api.crc_cache_update(self.control_bank, self.control_shape, n, frames, depth, k_ctl, v_ctl,
                                 self.control_cache, woff, stream)
        params = api.retrieval_params(c.E, c.w_v, c.tau_c, c.cos_tau_v, c.delta, c.k, self.ext_first(n), 1)
        rope = self.rope(n)
        api.crc_retrieve(self.bank, n + 1, self.shape, frames, n, params, self.cache, self.idx, self.score,
                         self.count, stream, rope=rope)
        if self.control_shape is not None:
            api.crc_gather(self.control_shape, self.control_bank.kv, self.idx, c.k, self.control_cache, rope=rope,
                           stream=stream)
        api.crc_correspond(self.shape, frames, depth, self.bank, self.idx, self.count, c.k, c.eps, self.uv,
                           self.cell, self.valid, stream)
        api.crc_biased_attention(self.shape, q, self.cache, o, lse, self.uv, self.valid, c.k, self.idx, c.lam,
                                 c.sigma, 0, self.status, stream)

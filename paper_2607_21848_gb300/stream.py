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

import ctypes as C
import dataclasses
from typing import List, Optional, Tuple

import numpy as np
import torch

from . import _abi, api


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
    def window_slot_offset(self, n: int) -> int:
        """Cache offset that receives chunk n: the sink for chunk 0, else ring slot n % W."""
        return 0 if n == 0 else self.window_offset(n % self.cfg.window)

    def step(self, n: int, frames: np.ndarray, depth: torch.Tensor, k_new: torch.Tensor, v_new: torch.Tensor,
             q: torch.Tensor, o: torch.Tensor, lse: Optional[torch.Tensor] = None, stream=None,
             k_ctl: Optional[torch.Tensor] = None, v_ctl: Optional[torch.Tensor] = None, events=None) -> None:
        """One chunk step through the separate entry points.  `events` (five CUDA events)
        are recorded on `stream` around the update, the retrieval (with the control
        mirror), the reprojection and the attention, for per-stage timing."""
        c = self.cfg
        s = stream if stream is not None else torch.cuda.current_stream()
        woff = self.window_slot_offset(n)
        self.cache.segments = self.segments(n)
        if events:
            events[0].record(s)
        api.crc_cache_update(self.bank, self.shape, n, frames, depth, k_new, v_new, self.cache, woff, s)
        if self.control_shape is not None:
            self.control_cache.segments = self.cache.segments
            api.crc_cache_update(self.control_bank, self.control_shape, n, frames, depth, k_ctl, v_ctl,
                                 self.control_cache, woff, s)
        if events:
            events[1].record(s)
        params = api.retrieval_params(c.E, c.w_v, c.tau_c, c.cos_tau_v, c.delta, c.k, self.ext_first(n), 1)
        rope = self.rope(n)
        api.crc_retrieve(self.bank, n + 1, self.shape, frames, n, params, self.cache, self.idx, self.score,
                         self.count, s, rope=rope)
        if self.control_shape is not None:
            api.crc_gather(self.control_shape, self.control_bank.kv, self.idx, c.k, self.control_cache, rope=rope,
                           stream=s)
        if events:
            events[2].record(s)
        api.crc_correspond(self.shape, frames, depth, self.bank, self.idx, self.count, c.k, c.eps, self.uv,
                           self.cell, self.valid, s)
        if events:
            events[3].record(s)
        api.crc_biased_attention(self.shape, q, self.cache, o, lse, self.uv, self.valid, c.k, self.idx, c.lam,
                                 c.sigma, 0, self.status, s)
        if events:
            events[4].record(s)

    # ---- the step as one replayed CUDA graph ------------------------------
    def descriptor(self, n: int, frames: np.ndarray) -> _abi.crc_step:
        """The per-step values of step n (crc_step): the chunk, its window slot, the
        fallback chunk, the re-positioning target, the live segments and the frames."""
        c = self.cfg
        d = _abi.crc_step()
        d.n = n
        d.window_offset = self.window_slot_offset(n)
        d.ext_first = self.ext_first(n)
        rope = self.rope(n)
        d.rope_pos_slot0 = rope.pos_slot0 if rope is not None else 0
        for g, seg in enumerate(self.segments(n)):
            d.seg_length[g] = seg[1]
        rec = np.ascontiguousarray(frames, dtype=np.float64).reshape(-1, 21)
        if rec.shape[0] != c.F:
            raise ValueError(f"expected {c.F} frame records")
        C.memmove(C.addressof(d.frames), rec.ctypes.data, rec.nbytes)
        return d

    def plan(self, depth: torch.Tensor, k_new: torch.Tensor, v_new: torch.Tensor, q: torch.Tensor, o: torch.Tensor,
             lse: Optional[torch.Tensor] = None) -> _abi.crc_step_plan:
        """The fixed part of crc_chunk_step: this stream's bank, cache and outputs, and the
        input buffers that every step reads (their addresses are captured)."""
        c = self.cfg
        if self.control_shape is not None:
            raise ValueError("the graph-replayed step has no control-branch mirror")
        p = _abi.crc_step_plan()
        p.shape = self.shape
        p.bank = self.bank.struct()
        full = api.Cache(self.cache.k, self.cache.v, self.segments(c.window + 1))  # every segment at its length
        p.cache = full.struct()
        p.retrieval = api.retrieval_params(c.E, c.w_v, c.tau_c, c.cos_tau_v, c.delta, c.k, -1, 1)
        r = self.rope(c.window + 1)
        if r is not None:
            p.rope = r
        p.eps, p.lam, p.sigma, p.attn_flags = c.eps, c.lam, c.sigma, 0
        p.d_depth, p.d_k, p.d_v = depth.data_ptr(), k_new.data_ptr(), v_new.data_ptr()
        p.q, p.o = api.tensor_view(q), api.tensor_view(o)
        p.d_lse = lse.data_ptr() if lse is not None else None
        p.d_idx, p.d_score, p.d_count = self.idx.data_ptr(), self.score.data_ptr(), self.count.data_ptr()
        p.d_uv, p.d_cell, p.d_valid = self.uv.data_ptr(), self.cell.data_ptr(), self.valid.data_ptr()
        p.d_status = self.status.data_ptr()
        ws = self.bank.workspace
        p.d_workspace = ws.data_ptr() if ws is not None else None
        p.workspace_bytes = 0 if ws is None else ws.numel()
        return p

    def capture(self, depth: torch.Tensor, k_new: torch.Tensor, v_new: torch.Tensor, q: torch.Tensor,
                o: torch.Tensor, lse: Optional[torch.Tensor] = None, ring: int = 3) -> None:
        """Capture one CUDA graph of crc_chunk_step per descriptor slot (`ring` slots, each a
        device crc_step fed from its own pinned host copy).  replay() then serves every step:
        the caller fills depth / k_new / v_new / q (the captured buffers) and calls
        replay(n, frames)."""
        nb = C.sizeof(_abi.crc_step)
        self._plan = self.plan(depth, k_new, v_new, q, o, lse)
        self._h_desc = [torch.zeros(nb, dtype=torch.uint8, pin_memory=True) for _ in range(ring)]
        self._d_desc = [torch.zeros(nb, dtype=torch.uint8, device=self.idx.device) for _ in range(ring)]
        self._done = [torch.cuda.Event() for _ in range(ring)]
        self._graphs = []
        torch.cuda.synchronize()
        for i in range(ring):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                api.crc_chunk_step(self._plan, self._d_desc[i], torch.cuda.current_stream())
            self._graphs.append(g)
        self._replays = 0

    def replay(self, n: int, frames: np.ndarray, stream=None) -> None:
        """Step n by graph replay (after capture()): the descriptor goes to the device with one
        copy on `stream`, then the graph runs.  The host waits only for the step that last used
        this descriptor slot, `ring` steps ago, before it rewrites the slot's pinned copy."""
        i = self._replays % len(self._graphs)
        self._done[i].synchronize()
        d = self.descriptor(n, frames)
        C.memmove(self._h_desc[i].data_ptr(), C.addressof(d), C.sizeof(d))
        s = stream if stream is not None else torch.cuda.current_stream()
        with torch.cuda.stream(s):
            self._d_desc[i].copy_(self._h_desc[i], non_blocking=True)
            self._graphs[i].replay()
        self._done[i].record(s)
        self._replays += 1
        self.cache.segments = self.segments(n)

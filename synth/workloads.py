"""Seeded synthetic workloads for the per-chunk revisit-consistency path.

Shapes follow the paper's setup (Sec. 4.1: F=3 latent frames per chunk on a
30x52 token grid; Sec. 4.2: a clean cache of M=4F frames split into an anchor
chunk, retrieved chunk(s) and a recent window) and the five benchmark
workloads:

  1  tiny fp32       H=1  d=64  F=2  8x8    Nk=512   (128|128|256)  bank 8,    k=1
  2  wan1.3b k=1     H=12 d=128 F=3  30x52  Nk=18720 (4680|4680|9360) bank 64, k=1
  3  wan1.3b k=3     H=12 d=128 F=3  30x52  Nk=28080, 30 layers, bank 2000,   k=3
  4  14b 720p k=2    H=40 d=128 F=3  45x80  Nk=64800 (10800|21600|32400) bank 500
  5  loop stream     wan1.3b head shape, 200 steps on a 20 m circle, k=2

Motion statistics follow the paper's evaluation data (Sec. 5.1): ground
trajectories with translation-dominant, parallax-heavy motion and revisits
within about 2 m and 45 degrees.  None of the paper's datasets are used; these
inputs stand in for them.

Camera convention: camera-to-world rotation R whose columns are the camera's
right, down and forward (optical) axes in world coordinates; world z is up.
Depth is planar metric depth (distance along the optical axis), rendered by
ray casting an analytic scene of planes, as a 3D engine would supply it.
All random numbers come from numpy PCG64 streams keyed by (seed, purpose).
"""

from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Tuple

import numpy as np

SEG_SINK = 0
SEG_RETRIEVED = 1
SEG_WINDOW = 2

# The five workloads, by what they are (make_workload takes the index).
WORKLOAD_NAMES = {
    1: "tiny_fp32_8x8_k1",        # 1 head, d = 64, 2 frames of 8x8, 512 keys, fp32
    2: "wan1.3b_30x52_k1",        # 12 heads, d = 128, 3 frames of 30x52, 18 720 keys, bank 64
    3: "wan1.3b_30x52_k3_30L",    # as above with k = 3, 28 080 keys, bank 2000, 30 layers per call
    4: "14b_45x80_k2",            # 40 heads, 3 frames of 45x80, 64 800 keys, bank 500
    5: "wan1.3b_loop_stream_k2",  # the 200-step loop-closure stream, 30 layers
}

_PURPOSES = ("poses", "depth", "q", "k", "v", "bank", "scene", "pool", "step", "sweep")


def rng(seed: int, purpose: str, *extra: int) -> np.random.Generator:
    """Independent PCG64 stream for (seed, purpose, extra...)."""
    key = (_PURPOSES.index(purpose),) + tuple(int(e) for e in extra)
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(seed, spawn_key=key)))


# ----------------------------------------------------------------------------
# cameras
# ----------------------------------------------------------------------------


@dataclasses.dataclass
class Frames:
    """A stack of per-frame camera annotations (Sec. 4.1).

    K: [..., 3, 3] pinhole intrinsics on the token grid;
    R: [..., 3, 3] camera-to-world rotation;  c: [..., 3] camera centre.
    """

    K: np.ndarray
    R: np.ndarray
    c: np.ndarray

    def __getitem__(self, idx) -> "Frames":
        return Frames(self.K[idx], self.R[idx], self.c[idx])

    @property
    def shape(self) -> Tuple[int, ...]:
        return self.c.shape[:-1]

    def reshape(self, *shape) -> "Frames":
        return Frames(self.K.reshape(*shape, 3, 3), self.R.reshape(*shape, 3, 3), self.c.reshape(*shape, 3))


def frame_records(fr: Frames) -> np.ndarray:
    """Pack frames into the C ABI record layout: [N][21] fp64 = K(9) R(9) c(3), row-major."""
    n = int(np.prod(fr.shape)) if fr.shape else 1
    out = np.empty((n, 21), dtype=np.float64)
    out[:, 0:9] = fr.K.reshape(n, 9)
    out[:, 9:18] = fr.R.reshape(n, 9)
    out[:, 18:21] = fr.c.reshape(n, 3)
    return out


def pinhole(h: int, w: int, fov_x_deg: float) -> np.ndarray:
    """Intrinsics on an h x w token grid; token (row i, col j) sits at pixel (j, i)."""
    f = (w / 2.0) / math.tan(math.radians(fov_x_deg) / 2.0)
    return np.array([[f, 0.0, (w - 1) / 2.0], [0.0, f, (h - 1) / 2.0], [0.0, 0.0, 1.0]])


def camera_rotation(yaw: float, pitch: float = 0.0, roll: float = 0.0) -> np.ndarray:
    """Camera-to-world rotation for a camera looking along (yaw, pitch) radians."""
    fwd = np.array([math.cos(pitch) * math.cos(yaw), math.cos(pitch) * math.sin(yaw), math.sin(pitch)])
    right = np.array([math.sin(yaw), -math.cos(yaw), 0.0])
    down = np.cross(fwd, right)
    R = np.stack([right, down, fwd], axis=1)
    if roll != 0.0:
        cr, sr = math.cos(roll), math.sin(roll)
        R = R @ np.array([[cr, -sr, 0.0], [sr, cr, 0.0], [0.0, 0.0, 1.0]])
    return R


def random_rotation(g: np.random.Generator, max_deg: float) -> np.ndarray:
    """Rotation about a uniformly random axis by an angle uniform in [0, max_deg]."""
    a = g.normal(size=3)
    a /= np.linalg.norm(a)
    th = math.radians(g.uniform(0.0, max_deg))
    A = np.array([[0.0, -a[2], a[1]], [a[2], 0.0, -a[0]], [-a[1], a[0], 0.0]])
    return np.eye(3) + math.sin(th) * A + (1.0 - math.cos(th)) * (A @ A)


def random_unit(g: np.random.Generator) -> np.ndarray:
    a = g.normal(size=3)
    return a / np.linalg.norm(a)


# ----------------------------------------------------------------------------
# analytic scene + depth rendering
# ----------------------------------------------------------------------------


@dataclasses.dataclass
class Scene:
    """Ground plane z=0, an N-gon of infinite vertical walls, and finite vertical boards.

    Boards are double-sided rectangles: centre (x, y), horizontal unit tangent,
    half width, height from the ground.
    """

    wall_n: np.ndarray  # [W, 3] inward normals n with n.X >= b inside
    wall_b: np.ndarray  # [W]
    board_p: np.ndarray  # [B, 2] centres
    board_t: np.ndarray  # [B, 2] unit tangents
    board_hw: np.ndarray  # [B] half widths
    board_top: np.ndarray  # [B] heights

    @staticmethod
    def room(g: np.random.Generator, radius: float, n_walls: int, n_boards: int,
             board_rmin: float, board_rmax: float) -> "Scene":
        ang = 2.0 * math.pi * (np.arange(n_walls) + 0.5) / n_walls
        wall_n = np.stack([-np.cos(ang), -np.sin(ang), np.zeros(n_walls)], axis=1)
        wall_b = -radius * np.ones(n_walls)
        r = np.sqrt(g.uniform(board_rmin ** 2, board_rmax ** 2, size=n_boards))
        phi = g.uniform(0.0, 2.0 * math.pi, size=n_boards)
        board_p = np.stack([r * np.cos(phi), r * np.sin(phi)], axis=1)
        t_ang = g.uniform(0.0, math.pi, size=n_boards)
        board_t = np.stack([np.cos(t_ang), np.sin(t_ang)], axis=1)
        board_hw = g.uniform(0.5, 3.0, size=n_boards)
        board_top = g.uniform(1.0, 6.0, size=n_boards)
        return Scene(wall_n, wall_b, board_p, board_t, board_hw, board_top)


def _ray_hits(scene: Scene, origin: np.ndarray, dirs: np.ndarray) -> np.ndarray:
    """Smallest positive ray parameter t for rays origin + t*dirs ([N,3]); inf if none."""
    best = np.full(dirs.shape[0], np.inf)
    with np.errstate(divide="ignore", invalid="ignore"):
        # ground
        t = -origin[2] / dirs[:, 2]
        best = np.where((t > 1e-9) & (t < best), t, best)
        # walls n.X = b
        for n, b in zip(scene.wall_n, scene.wall_b):
            t = (b - n @ origin) / (dirs @ n)
            best = np.where((t > 1e-9) & (t < best), t, best)
        # boards: vertical plane through p with normal perpendicular to the tangent
        for p, tg, hw, top in zip(scene.board_p, scene.board_t, scene.board_hw, scene.board_top):
            n = np.array([-tg[1], tg[0], 0.0])
            b = n[0] * p[0] + n[1] * p[1]
            t = (b - n @ origin) / (dirs @ n)
            X = origin[None, :] + t[:, None] * dirs
            lat = (X[:, 0] - p[0]) * tg[0] + (X[:, 1] - p[1]) * tg[1]
            ok = (t > 1e-9) & (t < best) & (np.abs(lat) <= hw) & (X[:, 2] >= 0.0) & (X[:, 2] <= top)
            best = np.where(ok, t, best)
    return best


def render_depth(scene: Scene, K: np.ndarray, R: np.ndarray, c: np.ndarray, h: int, w: int,
                 dmin: float, dmax: float, pix: Optional[np.ndarray] = None) -> np.ndarray:
    """Planar depth seen by camera (K, R, c) at every token centre (or at pixels `pix` [N,2] = (x, y)).

    The ray through pixel (x, y) is R @ K^-1 (x, y, 1); its third camera
    component is 1, so the ray parameter at the hit is the planar depth.
    Values are clamped to [dmin, dmax] (rays that escape read dmax).
    """
    grid_out = pix is None
    if grid_out:
        ii, jj = np.meshgrid(np.arange(h, dtype=np.float64), np.arange(w, dtype=np.float64), indexing="ij")
        pix = np.stack([jj.ravel(), ii.ravel()], axis=1)
    hom = np.concatenate([pix, np.ones((pix.shape[0], 1))], axis=1)
    cam = np.linalg.solve(K, hom.T).T
    dirs = cam @ R.T
    t = _ray_hits(scene, np.asarray(c, dtype=np.float64), dirs)
    t = np.clip(t, dmin, dmax)
    return t.reshape(h, w) if grid_out else t


# ----------------------------------------------------------------------------
# trajectories
# ----------------------------------------------------------------------------


def _frames_from_path(pos: np.ndarray, yaw: np.ndarray, pitch: np.ndarray, K: np.ndarray) -> Frames:
    n = pos.shape[0]
    R = np.stack([camera_rotation(yaw[i], pitch[i]) for i in range(n)])
    return Frames(np.broadcast_to(K, (n, 3, 3)).copy(), R, pos.copy())


def random_walk(g: np.random.Generator, n_chunks: int, F: int, K: np.ndarray, step: float = 0.5,
                yaw_jitter_deg: float = 10.0, pitch_jitter_deg: float = 3.0, radius: float = 24.0,
                height: float = 1.6) -> Frames:
    """Ground random walk: per chunk the heading turns by U[-jitter, jitter] and the
    camera advances `step` metres; frames inside a chunk are interpolated.  The walk
    turns back toward the origin when it nears `radius`.  Returns Frames [n_chunks, F]."""
    p = np.zeros(2)
    yaw = g.uniform(0.0, 2.0 * math.pi)
    pos = np.zeros((n_chunks, F, 3))
    yaws = np.zeros((n_chunks, F))
    for n in range(n_chunks):
        y0 = yaw
        yaw = yaw + math.radians(g.uniform(-yaw_jitter_deg, yaw_jitter_deg))
        if np.linalg.norm(p) > radius:
            yaw = math.atan2(-p[1], -p[0]) + math.radians(g.uniform(-30.0, 30.0))
        p0 = p.copy()
        p = p + step * np.array([math.cos(yaw), math.sin(yaw)])
        for f in range(F):
            a = f / F
            pos[n, f, :2] = p0 + a * (p - p0)
            pos[n, f, 2] = height
            yaws[n, f] = y0 + a * (yaw - y0)
    pitch = np.radians(g.uniform(-pitch_jitter_deg, pitch_jitter_deg, size=(n_chunks, F)))
    fr = _frames_from_path(pos.reshape(-1, 3), yaws.ravel(), pitch.ravel(), K)
    return fr.reshape(n_chunks, F)


def circle_loop(g: np.random.Generator, n_chunks: int, F: int, K: np.ndarray, radius: float = 20.0,
                height: float = 1.6, steps_per_lap: int = 150, yaw_jitter_deg: float = 10.0) -> Frames:
    """Closed loop: counter-clockwise circle, camera facing the tangent with a per-chunk
    yaw jitter U[-jitter, jitter]; it is back at its start after `steps_per_lap` chunks."""
    pos = np.zeros((n_chunks, F, 3))
    yaws = np.zeros((n_chunks, F))
    jit = np.radians(g.uniform(-yaw_jitter_deg, yaw_jitter_deg, size=n_chunks))
    for n in range(n_chunks):
        for f in range(F):
            th = 2.0 * math.pi * (n + f / F) / steps_per_lap
            pos[n, f] = (radius * math.cos(th), radius * math.sin(th), height)
            yaws[n, f] = th + math.pi / 2.0 + jit[n]
    fr = _frames_from_path(pos.reshape(-1, 3), yaws.ravel(), np.zeros(n_chunks * F), K)
    return fr.reshape(n_chunks, F)


# ----------------------------------------------------------------------------
# workloads
# ----------------------------------------------------------------------------


@dataclasses.dataclass
class Workload:
    cfg: int
    name: str
    H: int
    d: int
    F: int
    h: int
    w: int
    L: int
    k: int
    dtype: str  # "f32" or "bf16"
    segments: List[Tuple[int, int, int, int]]  # (offset, length, kind, slot)
    n_keys: int
    # retrieval parameters (Eq. 1)
    E: float
    w_v: float
    tau_c: float
    cos_tau_v: float
    delta: int
    # bias / visibility parameters (Eq. 2, Eq. 4)
    lam: float
    sigma: float
    eps: float
    # cameras
    bank_frames: Frames  # [B, F]
    cur_frames: Frames  # [F]
    n: int  # current chunk index
    num_slabs: int  # K/V slab pool size; chunk j lives in slab j % num_slabs
    seed: int
    dmin: float
    dmax: float
    scene: Optional[Scene] = None
    iid_depth: bool = False
    qkv_scale: float = 1.0
    _depth_cache: dict = dataclasses.field(default_factory=dict, repr=False)

    @property
    def Nc(self) -> int:
        return self.F * self.h * self.w

    @property
    def Nq(self) -> int:
        return self.Nc

    @property
    def bank_size(self) -> int:
        return self.bank_frames.shape[0]

    @property
    def S(self) -> int:
        return self.k * self.F

    def depth_of(self, chunk: int) -> np.ndarray:
        """Planar depth [F, h, w] fp32 of chunk `chunk` (chunk == n is the current chunk)."""
        if chunk in self._depth_cache:
            return self._depth_cache[chunk]
        fr = self.cur_frames if chunk == self.n else self.bank_frames[chunk]
        if self.iid_depth:
            g = rng(self.seed, "depth", chunk)
            dep = np.exp(g.uniform(math.log(self.dmin), math.log(self.dmax), size=(self.F, self.h, self.w)))
        else:
            dep = np.stack([render_depth(self.scene, fr.K[f], fr.R[f], fr.c[f], self.h, self.w,
                                         self.dmin, self.dmax) for f in range(self.F)])
        dep = dep.astype(np.float32)
        self._depth_cache[chunk] = dep
        return dep

    def depth_bank(self, upto: Optional[int] = None) -> np.ndarray:
        """Depth of bank chunks 0..upto-1 as [upto, F, h, w] fp32."""
        upto = self.bank_size if upto is None else upto
        return np.stack([self.depth_of(j) for j in range(upto)])


def _segments(Nc: int, k: int, window_chunks: int) -> Tuple[List[Tuple[int, int, int, int]], int]:
    segs = [(0, Nc, SEG_SINK, 0)]
    off = Nc
    for r in range(k):
        segs.append((off, Nc, SEG_RETRIEVED, r))
        off += Nc
    for r in range(window_chunks):
        segs.append((off, Nc, SEG_WINDOW, r))
        off += Nc
    return segs, off


def make_workload(cfg: int, *, layers: Optional[int] = None, heads: Optional[int] = None,
                  bank: Optional[int] = None, grid: Optional[Tuple[int, int]] = None,
                  seed: Optional[int] = None) -> Workload:
    """Build workload `cfg` of WORKLOAD_NAMES (1..5).  `layers`, `heads`, `bank` and `grid`
    shrink it for seconds-scale parity runs while keeping its structure."""
    seed = 1000 + cfg if seed is None else seed
    gp = rng(seed, "poses")
    if cfg == 1:
        H, d, F, (h, w), L, k, dtype, B = 1, 64, 2, (8, 8), 1, 1, "f32", 8
        window_chunks, dmin, dmax, fov = 2, 0.5, 20.0, 90.0
    elif cfg == 2:
        H, d, F, (h, w), L, k, dtype, B = 12, 128, 3, (30, 52), 1, 1, "bf16", 64
        window_chunks, dmin, dmax, fov = 2, 0.5, 50.0, 90.0
    elif cfg == 3:
        H, d, F, (h, w), L, k, dtype, B = 12, 128, 3, (30, 52), 30, 3, "bf16", 2000
        window_chunks, dmin, dmax, fov = 2, 0.5, 50.0, 90.0
    elif cfg == 4:
        H, d, F, (h, w), L, k, dtype, B = 40, 128, 3, (45, 80), 1, 2, "bf16", 500
        window_chunks, dmin, dmax, fov = 3, 0.5, 100.0, 90.0
    elif cfg == 5:
        H, d, F, (h, w), L, k, dtype, B = 12, 128, 3, (30, 52), 30, 2, "bf16", 200
        window_chunks, dmin, dmax, fov = 2, 0.5, 50.0, 90.0
    else:
        raise ValueError(f"unknown config {cfg}")
    if layers is not None:
        L = layers
    if heads is not None:
        H = heads
    if bank is not None:
        B = bank
    if grid is not None:
        h, w = grid
    K = pinhole(h, w, fov)
    Nc = F * h * w
    segs, Nk = _segments(Nc, k, window_chunks)

    scene = None
    iid = False
    if cfg == 1:
        iid = True
        walk = random_walk(gp, B, F, K, step=0.5)
        # current chunk: a bank chunk moved by a rotation <= 15 deg and a translation <= 0.5 m
        target = int(gp.integers(0, B))
        dR = random_rotation(gp, 15.0)
        dt = random_unit(gp) * gp.uniform(0.0, 0.5)
        cur = Frames(walk.K[target].copy(), np.einsum("ij,fjk->fik", dR, walk.R[target]),
                     walk.c[target] + dt[None, :])
        E, w_v, tau_c, cos_tau_v, delta, eps = 1.0, 0.5, math.inf, -1.0, 1, math.inf
        scale = 1.0
    elif cfg in (2, 3, 4):
        scene = Scene.room(rng(seed, "scene"), radius=40.0, n_walls=12, n_boards=60,
                           board_rmin=2.0, board_rmax=36.0)
        walk = random_walk(gp, B + 1, F, K, step=0.5, radius=24.0)
        # force a revisit: the current chunk returns near a chunk from the middle of the bank
        target = B // 2
        dR = camera_rotation(math.radians(gp.uniform(-10.0, 10.0)), 0.0) @ camera_rotation(0.0).T
        dt = np.array([gp.uniform(-0.5, 0.5), gp.uniform(-0.5, 0.5), 0.0])
        cur = Frames(walk.K[target].copy(), np.einsum("ij,fjk->fik", dR, walk.R[target]),
                     walk.c[target] + dt[None, :])
        walk = walk[:B]
        E, w_v, tau_c, cos_tau_v, delta, eps = 1.0, 0.5, math.inf, -1.0, 1, math.inf
        scale = 1.0 / math.sqrt(128.0)
    else:  # 5: loop stream; the bank holds the whole loop, step n uses chunks 0..n
        scene = Scene.room(rng(seed, "scene"), radius=32.0, n_walls=16, n_boards=40,
                           board_rmin=6.0, board_rmax=30.0)
        walk = circle_loop(gp, B, F, K)
        cur = walk[B - 1]
        E, w_v, tau_c, cos_tau_v, delta, eps = 20.0, 0.5, 0.1, math.cos(math.radians(45.0)), 3, 0.05
        scale = 1.0 / math.sqrt(128.0)
    num_slabs = min(B, 16)
    return Workload(cfg=cfg, name=WORKLOAD_NAMES[cfg], H=H, d=d, F=F, h=h, w=w, L=L, k=k, dtype=dtype,
                    segments=segs, n_keys=Nk, E=E, w_v=w_v, tau_c=tau_c, cos_tau_v=cos_tau_v,
                    delta=delta, lam=2.0, sigma=1.0, eps=eps, bank_frames=walk, cur_frames=cur,
                    n=B if cfg != 5 else B - 1, num_slabs=num_slabs, seed=seed, dmin=dmin, dmax=dmax,
                    scene=scene, iid_depth=iid, qkv_scale=scale)


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bf16 (ties to even); returns fp32 holding bf16 values."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    u = (u + 0x7FFF + lsb) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


def _normal(g: np.random.Generator, shape, scale: float, dtype: str) -> np.ndarray:
    x = g.standard_normal(size=shape, dtype=np.float32) * np.float32(scale)
    return bf16_round(x) if dtype == "bf16" else x


def make_qkv(wl: Workload, layers: Optional[int] = None, tag: int = 0):
    """Q [L, Nq, H, d] and cache K, V [L, Nk, H, d] as fp32 arrays (bf16-representable for bf16)."""
    L = wl.L if layers is None else layers
    q = _normal(rng(wl.seed, "q", tag), (L, wl.Nq, wl.H, wl.d), wl.qkv_scale, wl.dtype)
    k = _normal(rng(wl.seed, "k", tag), (L, wl.n_keys, wl.H, wl.d), wl.qkv_scale, wl.dtype)
    v = _normal(rng(wl.seed, "v", tag), (L, wl.n_keys, wl.H, wl.d), wl.qkv_scale, wl.dtype)
    return q, k, v


def make_kv_pool(wl: Workload, num_slabs: Optional[int] = None, layers: Optional[int] = None):
    """K/V slab pool [P, 2, L, Nc, H, d] (index 0 = K, 1 = V)."""
    P = wl.num_slabs if num_slabs is None else num_slabs
    L = wl.L if layers is None else layers
    return _normal(rng(wl.seed, "pool"), (P, 2, L, wl.Nc, wl.H, wl.d), wl.qkv_scale, wl.dtype)

"""Helpers shared by the GPU parity tests: move seeded inputs to the device, run
the oracle on the same inputs, compare with the tolerances of the path."""

from __future__ import annotations

import math

import numpy as np
import torch

import oracle
import synth
from paper_2607_21848_gb300 import api


def dev_dtype(wl):
    return torch.bfloat16 if wl.dtype == "bf16" else torch.float32


def oracle_bank_poses(fr: synth.Frames):
    """(c_j, v_j) of every chunk of Frames [B, F] from the oracle."""
    B = fr.shape[0]
    c = np.zeros((B, 3))
    v = np.zeros((B, 3))
    for j in range(B):
        c[j], v[j] = oracle.chunk_pose(fr.R[j], fr.c[j])
    return c, v


def oracle_retrieve(wl, bank_count=None, n=None, k=None, ext_first=-1, ext_min=0, resident=None, **over):
    fr = wl.bank_frames
    B = fr.shape[0] if bank_count is None else bank_count
    bc, bv = oracle_bank_poses(fr[:B])
    cur = wl.cur_frames if n is None else fr[n]
    cn, vn = oracle.chunk_pose(cur.R, cur.c)
    p = dict(E=wl.E, w_v=wl.w_v, tau_c=wl.tau_c, cos_tau_v=wl.cos_tau_v, delta=wl.delta)
    p.update(over)
    n = wl.n if n is None else n
    idx, score, count = oracle.retrieve(bc, bv, cn, vn, n, k=wl.k if k is None else k, resident=resident, **p)
    slots = oracle.fill_slots(idx, count, ext_first, ext_min, resident=resident)
    return idx, score, count, slots


def make_bank(wl, dtype, capacity=None, with_kv=False, device="cuda"):
    cap = wl.bank_size if capacity is None else capacity
    bank = api.Bank(cap, wl.F, wl.h, wl.w, wl.L, wl.H, wl.d, dtype, wl.num_slabs, device=device, with_kv=with_kv)
    shp = api.shape(wl.L, wl.H, wl.d, wl.F, wl.h, wl.w, dtype)
    return bank, shp


def insert_poses(bank, shp, fr: synth.Frames, first=0):
    api.crc_bank_insert_poses(bank, shp, first, synth.frame_records(fr))


def oracle_correspond(wl, slots, count, eps=None, cur=None, depth_cur=None, depth_of=None):
    """Oracle correspondences of the current chunk against the chunks in `slots`."""
    eps = wl.eps if eps is None else eps
    cur = wl.cur_frames if cur is None else cur
    depth_cur = wl.depth_of(wl.n) if depth_cur is None else depth_cur
    depth_of = wl.depth_of if depth_of is None else depth_of
    F = wl.F
    S = len(slots) * F
    Ks = np.zeros((S, 3, 3))
    Rs = np.zeros((S, 3, 3))
    cs = np.zeros((S, 3))
    ds = np.ones((S, wl.h, wl.w), dtype=np.float32)
    ok = np.zeros(S, dtype=bool)
    for r, j in enumerate(slots):
        for f in range(F):
            s = r * F + f
            if j >= 0 and r < count:
                fr = wl.bank_frames[j]
                Ks[s], Rs[s], cs[s] = fr.K[f], fr.R[f], fr.c[f]
                ds[s] = depth_of(j)[f]
                ok[s] = True
            else:
                Ks[s], Rs[s], cs[s] = cur.K[0], cur.R[0], cur.c[0]
    uv, cell, valid, zs = oracle.correspond(depth_cur, cur.K, cur.R, cur.c, ds, Ks, Rs, cs, eps, source_ok=ok,
                                            with_zs=True)
    return uv, cell, valid, zs, ds, ok


def exempt_pairs(wl, uv, zs, ds, depth_cur, eps):
    """Pairs whose integer decision sits within rounding distance of a boundary:
    u^ + 1/2 within 1e-4 of an integer, [X_s]_z within 1e-6 z_p of zero, or
    [X_s]_z within 1e-5 D_s of the visibility threshold (1 + eps) D_s."""
    Nq, S = zs.shape
    with np.errstate(invalid="ignore"):
        fx = uv[..., 0] + 0.5
        fy = uv[..., 1] + 0.5
        near = (np.abs(fx - np.round(fx)) < 1e-4) | (np.abs(fy - np.round(fy)) < 1e-4)
        z = depth_cur.reshape(-1).astype(np.float64)[:, None]
        near |= np.abs(zs) < 1e-6 * np.abs(z)
        if not math.isinf(eps):
            cx = np.floor(fx)
            cy = np.floor(fy)
            inb = np.isfinite(cx) & np.isfinite(cy) & (cx >= 0) & (cx < wl.w) & (cy >= 0) & (cy < wl.h)
            xi = np.where(inb, cx, 0).astype(np.int64)
            yi = np.where(inb, cy, 0).astype(np.int64)
            Ds = ds.astype(np.float64)[np.arange(S)[None, :].repeat(Nq, 0), yi, xi]
            near |= inb & (np.abs(zs - (1 + eps) * Ds) <= 1e-5 * Ds)
    return near


def compare_correspondence(wl, o, g_uv, g_cell, g_valid, eps, depth_cur=None):
    uv, cell, valid, zs, ds, ok = o
    depth_cur = wl.depth_of(wl.n) if depth_cur is None else depth_cur
    ex = exempt_pairs(wl, uv, zs, ds, depth_cur, eps)
    ex &= ok[None, :]
    gv = g_valid.astype(bool)
    bad_valid = (gv != valid) & ~ex
    bad_cell = (g_cell != cell) & ~ex
    both = gv & valid & ~ex
    uv_err = np.abs(g_uv - uv)[both].max() if both.any() else 0.0
    return dict(n=valid.size, n_valid=int(valid.sum()), exempt=int(ex.sum()), bad_valid=int(bad_valid.sum()),
                bad_cell=int(bad_cell.sum()), uv_err=float(uv_err))


def to_dev(a, dtype=None, device="cuda"):
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.to(dtype)
    return t.to(device)


def attn_errors(O_gpu: np.ndarray, O_ref: np.ndarray):
    err = np.abs(O_gpu.astype(np.float64) - O_ref)
    rms = math.sqrt(float(np.mean(O_ref ** 2)))
    return float(err.max()), float(err.max() / rms) if rms > 0 else float("inf"), rms

"""Stand-alone sweeps of single kernels, for measurement and profiling (e.g. under ncu):

  python sweeps.py correspond      # 126 MB reprojection sweep, scene depth
  python sweeps.py correspond-iid  # the same with depth drawn per token
  python sweeps.py gather          # crc_gather, plain and re-positioned
  python sweeps.py retrieve        # Eq. 1 scoring and top-k over banks of 64 to 261 120 entries

Measurement tooling beside bench.py (which imports it for its context block); not part
of the library package.
"""

from __future__ import annotations

import json
import sys


def correspond_sweep(device="cuda:0", iters: int = 20, depth: str = "scene"):
    """Reprojection (Eq. 3-4) at a scale where it is no longer launch-bound: 4 frames of
    180 x 320 tokens (230400 queries) against 8 retrieved chunks (32 source frames),
    7.4 M (query, frame) pairs and 126 MB in one launch.  A sweep, not a configuration.

    depth="scene": the chunks are 9 consecutive chunks of a ground random walk through
    a room of walls and boards (the scene model of the synthetic workloads), and every
    depth map is rendered from that scene, so depth is piecewise smooth as in real
    footage.  depth="iid": depth drawn independently per token, log-uniform on
    [0.5, 20]; neighbouring tokens then land in unrelated cells of every source map,
    the worst case for the source-depth reads of the visibility test."""
    import math

    import numpy as np
    import torch

    import synth
    from synth import workloads as W
    from paper_2607_21848_gb300 import api

    F, h, w, k = 4, 180, 320, 8
    K = synth.pinhole(h, w, 90.0)
    fr = synth.random_walk(synth.rng(999, "sweep"), k + 1, F, K, step=0.5, radius=24.0)
    bank = api.Bank(k + 1, F, h, w, 1, 1, 64, torch.float32, 1, device=device, with_kv=False)
    shp = api.shape(1, 1, 64, F, h, w, torch.float32)
    api.crc_bank_insert_poses(bank, shp, 0, synth.frame_records(fr))
    if depth == "scene":
        scene = W.Scene.room(synth.rng(999, "scene"), radius=40.0, n_walls=12, n_boards=60, board_rmin=2.0,
                             board_rmax=36.0)
        dep = np.stack([np.stack([W.render_depth(scene, fr.K[j, f], fr.R[j, f], fr.c[j, f], h, w, 0.5, 50.0)
                                  for f in range(F)]) for j in range(k + 1)]).astype(np.float32)
        bank.depth.copy_(torch.from_numpy(dep).to(device))
    elif depth == "iid":
        g = torch.Generator(device=device).manual_seed(99)
        bank.depth.copy_(torch.exp(torch.rand(bank.depth.shape, generator=g, device=device) * math.log(40.0)) * 0.5)
    else:
        raise ValueError(f"unknown depth model {depth!r}")
    depth_cur = bank.depth[k].clone()
    idx = torch.arange(k, dtype=torch.int32, device=device)
    count = torch.full((1,), k, dtype=torch.int32, device=device)
    Nq, S = F * h * w, k * F
    uv = torch.empty(Nq, S, 2, device=device)
    cell = torch.empty(Nq, S, dtype=torch.int32, device=device)
    valid = torch.empty(Nq, S, dtype=torch.uint8, device=device)
    cur = synth.frame_records(fr[k])

    def run():
        api.crc_correspond(shp, cur, depth_cur, bank, idx, count, k, 0.05, uv, cell, valid)

    run()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    # eager: back-to-back calls through the Python binding
    e0.record()
    for _ in range(iters):
        run()
    e1.record()
    torch.cuda.synchronize()
    t_eager = e0.elapsed_time(e1) / 1e3 / iters
    # the same launches captured in one CUDA graph and replayed: launch overhead removed
    g = torch.cuda.CUDAGraph()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        run()
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    with torch.cuda.graph(g):
        for _ in range(iters):
            run()
    g.replay()
    torch.cuda.synchronize()
    e0.record()
    g.replay()
    e1.record()
    torch.cuda.synchronize()
    t = e0.elapsed_time(e1) / 1e3 / iters
    nbytes = Nq * 4 + Nq * S * (8 + 4 + 1 + 4)
    return {"depth": depth, "queries": Nq, "source_frames": S, "pairs": Nq * S, "bytes": nbytes, "ms": t * 1e3,
            "gbs": nbytes / t / 1e9, "eager_ms": t_eager * 1e3, "valid_fraction": float(valid.float().mean()),
            "timing": f"{iters} launches in one CUDA graph, outputs (95 MB) rewritten each launch"}


def gather_sweep(device="cuda:0", iters: int = 10):
    """crc_gather of one retrieved chunk at the Wan-1.3B chunk shape (30 layers, 12 heads,
    d = 128, 4680 tokens), plain and with the keys re-positioned (22 interleaved temporal
    rotary pairs): 862.6 MB read and 862.6 MB written per call either way."""
    import torch

    import synth
    from paper_2607_21848_gb300 import api

    wl = synth.make_workload(2, layers=30)
    L, Nc, H, d = wl.L, wl.Nc, wl.H, wl.d
    g = torch.Generator(device=device).manual_seed(3)
    pool = (torch.randn(2, 2, L, Nc, H, d, generator=g, device=device) * wl.qkv_scale).to(torch.bfloat16)
    segs = [(0, Nc, api.SEG_SINK, 0), (Nc, Nc, api.SEG_RETRIEVED, 0), (2 * Nc, 2 * Nc, api.SEG_WINDOW, 0)]
    cache = api.Cache.empty(L, 4 * Nc, H, d, torch.bfloat16, segs, device=device)
    shp = api.shape(L, H, d, wl.F, wl.h, wl.w, torch.bfloat16)
    idx = torch.tensor([33], dtype=torch.int32, device=device)
    out = {}
    for name, rope in (("plain", None), ("rope", api.rope_params(0, 22, 10000.0, True, pos_slot0=189, pos_stride=3))):
        api.crc_gather(shp, pool, idx, 1, cache, rope=rope)
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(iters):
            api.crc_gather(shp, pool, idx, 1, cache, rope=rope)
        e1.record()
        torch.cuda.synchronize()
        t = e0.elapsed_time(e1) / 1e3 / iters
        nbytes = 2 * 2 * L * Nc * H * d * 2
        out[name] = {"bytes": nbytes, "ms": t * 1e3, "gbs": nbytes / t / 1e9}
    return out


def retrieve_sweep(device="cuda:0", iters: int = 20):
    """Eq. 1 scoring and top-k alone (no gather) over banks from 64 to 261 120 entries,
    at k = 1 and k = 8: the bank's chunk poses are drawn at random, every entry is
    admissible (E = 1, no centre or view gate, delta = 1), so every entry is scored and
    merged.  Through the workspace call and through crc_retrieve_noalloc."""
    import numpy as np
    import torch

    import synth
    from paper_2607_21848_gb300 import _abi, api

    F, h, w = 3, 30, 52
    walk = synth.random_walk(synth.rng(7, "sweep"), 1, F, synth.pinhole(h, w, 90.0), step=0.5, radius=24.0)
    cur = synth.frame_records(walk[0])
    out = {}
    for B in (64, 2000, 20000, 100003, 261120):
        bank = api.Bank(B, F, h, w, 1, 1, 64, torch.float32, 1, device=device, with_kv=False)
        g = np.random.default_rng(B)
        c = g.normal(size=(B, 3)) * 20.0
        v = g.normal(size=(B, 3))
        v /= np.linalg.norm(v, axis=1, keepdims=True)
        bank.centre.copy_(torch.from_numpy(c))
        bank.view.copy_(torch.from_numpy(v))
        shp = api.shape(1, 1, 64, F, h, w, torch.float32)
        row = {}
        for k in (1, 8):
            params = api.retrieval_params(1.0, 0.5, float("inf"), -1.0, 1, k)
            idx = torch.empty(k, dtype=torch.int32, device=device)
            cnt = torch.empty(1, dtype=torch.int32, device=device)
            calls = {"workspace": lambda: api.crc_retrieve(bank, B, shp, cur, B, params, None, idx, None, cnt)}
            if _abi.load().crc_retrieve_workspace_size(B, k) <= _abi.CRC_NOALLOC_SCRATCH_BYTES:
                calls["noalloc"] = lambda: api.crc_retrieve_noalloc(bank, B, shp, cur, B, params, None, idx, None, cnt)
            got = {}
            for name, fn in calls.items():
                fn()
                torch.cuda.synchronize()
                got[name] = idx.cpu().clone()
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record()
                for _ in range(iters):
                    fn()
                e1.record()
                torch.cuda.synchronize()
                row[f"k{k}_{name}_us"] = e0.elapsed_time(e1) / iters * 1e3
            assert all(torch.equal(x, got["workspace"]) for x in got.values()), "noalloc and workspace calls disagree"
            assert int(cnt.item()) == min(k, B)
        out[str(B)] = row
    return out


def main(argv=None):
    argv = sys.argv[1:] if argv is None else argv
    what = argv[0] if argv else "correspond"
    import os

    sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))  # the package and the synth module
    from paper_2607_21848_gb300 import build

    build.build()
    if what == "correspond":
        print(json.dumps(correspond_sweep("cuda:0")))
    elif what == "correspond-iid":
        print(json.dumps(correspond_sweep("cuda:0", depth="iid")))
    elif what == "gather":
        print(json.dumps(gather_sweep("cuda:0")))
    elif what == "retrieve":
        print(json.dumps(retrieve_sweep("cuda:0")))
    else:
        raise SystemExit(f"unknown sweep {what}")


if __name__ == "__main__":
    main()

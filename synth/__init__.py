"""Seeded synthetic inputs shaped like the paper's chunk-step workloads.

This package only *generates inputs*: camera trajectories, per-frame pinhole
intrinsics on the token grid, engine-style planar metric depth (by ray casting
an analytic scene), segmented KV-cache layouts and random Q/K/V.  It holds none
of the method's arithmetic (no retrieval scoring, no reprojection warp, no
attention), so both the fp64 oracle and the CUDA path can draw from it.
"""

from .workloads import (  # noqa: F401
    Frames,
    Workload,
    SEG_SINK,
    SEG_RETRIEVED,
    SEG_WINDOW,
    pinhole,
    camera_rotation,
    random_rotation,
    Scene,
    render_depth,
    make_workload,
    make_qkv,
    make_kv_pool,
    bf16_round,
    frame_records,
    WORKLOAD_NAMES,
    rng,
    random_walk,
    circle_loop,
)

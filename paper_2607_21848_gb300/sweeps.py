"""Stand-alone sweeps of single kernels at scales larger than the chunk step, for
profiling (e.g. under ncu): `python -m paper_2607_21848_gb300.sweeps correspond`."""

from __future__ import annotations

import json
import sys


def main(argv=None):
    argv = sys.argv[1:] if argv is None else argv
    what = argv[0] if argv else "correspond"
    import os

    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    from paper_2607_21848_gb300 import build

    build.build()
    if what == "correspond":
        print(json.dumps(bench.correspond_sweep("cuda:0")))
    else:
        raise SystemExit(f"unknown sweep {what}")


if __name__ == "__main__":
    main()

"""Replay frames of a synthetic workload through the library (for profiling).

    python -m paper_2608_08330_gb300.replay --workload stress8 --frames 3 \
        --mode barrier --spread zero [--multiscale] [--resident]

Builds the library if needed, creates one context, and runs `--frames` frames:
every agent's payload completes at the times of the chosen spread ("zero": all
at once; "spaced": agent k at k x --gap ms, so each branch runs alone;
"preset": the workload's own arrival recipe), in RTCC or Barrier mode.  The
context's initialisation runs every graph once (n_agents branch graphs twice,
one launch per batch size 2..n_agents, the post-join once) before the first
frame; a profiler that counts launches must skip those.  Prints the backbone
launch sizes of each frame.
"""
from __future__ import annotations

import argparse
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main(argv=None) -> int:
    import synth
    from paper_2608_08330_gb300 import build as B
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="stress8")
    ap.add_argument("--frames", type=int, default=3)
    ap.add_argument("--mode", choices=["rtcc", "barrier"], default="barrier")
    ap.add_argument("--spread", choices=["zero", "spaced", "preset"], default="zero")
    ap.add_argument("--gap", type=float, default=2.0, help="ms between arrivals when spaced")
    ap.add_argument("--multiscale", action="store_true")
    ap.add_argument("--resident", action="store_true", help="payloads staged in HBM first")
    a = ap.parse_args(argv)
    B.build()
    from paper_2608_08330_gb300 import rtcc as R
    R.load()
    cfg = synth.get_config(a.workload)
    K = cfg.n_agents
    flags = R.FLAG_MULTISCALE if a.multiscale else 0
    ctx = R.rtcc_init(R.model_config(cfg, flags=flags), synth.weight_blob(synth.weights_for(cfg)))
    mode = R.MODE_RTCC if a.mode == "rtcc" else R.MODE_BARRIER
    try:
        for f in range(a.frames):
            pts = [synth.points_for(cfg, f, k) for k in range(K)]
            if a.spread == "zero":
                t = [0.0] * K
            elif a.spread == "spaced":
                t = [a.gap * k for k in range(K)]
            else:
                t = [float(x) for x in synth.arrivals_for(cfg, f)]
            if a.resident:
                for k in range(K):
                    assert R.rtcc_stage_resident(ctx, k, pts[k]) == R.OK
            assert R.rtcc_set_mode(ctx, mode) == R.OK
            assert R.rtcc_frame_begin(ctx, f + 1, 0.0) == R.OK
            t0 = R.rtcc_now_ms()
            for k in sorted(range(K), key=lambda k: (t[k], k)):
                while R.rtcc_now_ms() < t0 + t[k]:
                    pass
                s = (R.rtcc_payload_resident(ctx, k, t[k]) if a.resident else
                     R.rtcc_payload_complete(ctx, k, pts[k], t[k]))
                assert s == R.OK, R.rtcc_status_str(s)
            s, boxes, _ = R.rtcc_wait_detection(ctx, 60000)
            assert s == R.OK, R.rtcc_status_str(s)
            info = R.rtcc_get_frame_info(ctx)
            sizes = [info.backbone_batch[j] for j in range(min(info.n_backbone_launches, R.MAX_AGENTS))]
            print(f"frame {f}: backbone launches {sizes}, {len(boxes)} boxes", flush=True)
    finally:
        R.rtcc_destroy(ctx)
    return 0


if __name__ == "__main__":
    sys.exit(main())

"""Helpers shared by the GPU tests: running frames through the C ABI and
comparing against the oracle."""
from __future__ import annotations

import numpy as np

import synth
from oracle import forward as of
from oracle import nms as onms
from paper_2608_08330_gb300 import build as B
from paper_2608_08330_gb300 import rtcc as R

# Tolerance for floating-point outputs (fp16/bf16 storage, fp32 accumulation):
# |gpu - oracle| <= ATOL + RTOL * |oracle|, elementwise.
ATOL = 2e-2
RTOL = 1e-2


def load():
    B.build()
    R.load()
    return R


def assert_close(g, o, what="", atol=ATOL, rtol=RTOL):
    g = np.asarray(g, dtype=np.float64)
    o = np.asarray(o, dtype=np.float64)
    assert g.shape == o.shape, (what, g.shape, o.shape)
    err = np.abs(g - o)
    lim = atol + rtol * np.abs(o)
    bad = err > lim
    if bad.any():
        i = np.argmax(err - lim)
        raise AssertionError(f"{what}: {int(bad.sum())}/{bad.size} outside tol; worst at flat "
                             f"{i}: gpu {g.reshape(-1)[i]!r} oracle {o.reshape(-1)[i]!r}")


def u16_to_f64(u: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "fp16":
        return u.view(np.float16).astype(np.float64)
    return (u.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


DEBUG_FLAGS = R.FLAG_KEEP_FUSED | R.FLAG_TIMELINE | R.FLAG_KEEP_LAYERS


def make_ctx(cfg, flags=DEBUG_FLAGS, max_points=None):
    w = synth.weights_for(cfg)
    blob = synth.weight_blob(w)
    ctx = R.rtcc_init(R.model_config(cfg, max_points=max_points, flags=flags), blob)
    return ctx, w


def run_frame(ctx, cfg, pts, arrivals, mode, frame_id=0, absent=()):
    """Replay one frame: events in (a_k, k) order; returns the boxes."""
    assert R.rtcc_set_mode(ctx, mode) == R.OK
    assert R.rtcc_frame_begin(ctx, frame_id, 0.0) == R.OK
    for k in sorted(range(cfg.n_agents), key=lambda k: (arrivals[k], k)):
        if k in absent:
            s = R.rtcc_payload_absent(ctx, k, float(arrivals[k]))
        else:
            s = R.rtcc_payload_complete(ctx, k, pts[k], float(arrivals[k]))
        assert s == R.OK, R.rtcc_status_str(s)
    s, boxes, _ = R.rtcc_wait_detection(ctx, 60000)
    assert s == R.OK, R.rtcc_status_str(s)
    return boxes


def gpu_tensor(ctx, cfg, agent, which, shape):
    """16-bit tensor as float64 in oracle layout [C][H][W] (from NHWC)."""
    u = R.rtcc_get_tensor(ctx, agent, which)
    x = u16_to_f64(u, cfg.dtype).reshape(shape[1], shape[2], shape[0])
    return x.transpose(2, 0, 1)


def block_shapes(cfg):
    out = []
    w, h = cfg.grid_w, cfg.grid_h
    for (_, ch, st) in cfg.blocks:
        w, h = w // st, h // st
        out.append((ch, h, w))
    return out


def conv_layers(cfg):
    """(block, layer, stride, output shape [C][H][W]) of every 3x3 conv in order."""
    out = []
    w, h = cfg.grid_w, cfg.grid_h
    for bi, (n, ch, st) in enumerate(cfg.blocks):
        w, h = w // st, h // st
        for li in range(n):
            out.append((bi, li, st if li == 0 else 1, (ch, h, w)))
    return out


def oracle_conv_layer(x, weights, bi, li, stride, store):
    """One conv + bias + ReLU + storage rounding of the oracle."""
    w = of.store_round(weights[f"b{bi}.c{li}.w"], store)
    b = of.store_round(weights[f"b{bi}.c{li}.b"], store)
    return of.store_round(of.relu(of.conv3x3(x, w, b, stride)), store)


def oracle_neck(blocks, weights, cfg, store):
    if not cfg.up_strides:
        return blocks[-1]
    ups = []
    for bi, s in enumerate(cfg.up_strides):
        w = of.store_round(weights[f"up{bi}.w"], store)
        b = of.store_round(weights[f"up{bi}.b"], store)
        ups.append(of.store_round(of.relu(of.deconv(blocks[bi], w, b, s)), store))
    return np.concatenate(ups, axis=0)


def head_to_oracle_layout(head_hwc):
    return np.asarray(head_hwc, dtype=np.float64).transpose(2, 0, 1)


def check_nms(dec, out, thr, band=1e-4):
    """Rotated NMS parity on the GPU's own input boxes: the output is a
    subsequence of them copied bit for bit, and each keep/drop decision, taken
    against the boxes the GPU kept before it, matches the oracle's float64 IoU
    test -- except where that IoU lies within `band` of the threshold (the
    kernel decides in float32).  Returns the kept positions."""
    pos = {int(a): i for i, a in enumerate(dec["anchor"])}
    assert len(pos) == len(dec), "anchors identify the boxes"
    kept = [pos[int(a)] for a in out["anchor"]]
    assert kept == sorted(kept) and len(set(kept)) == len(kept)
    assert out.tobytes() == dec[kept].tobytes()
    bev = np.stack([dec[f] for f in ("x", "y", "l", "w", "yaw")], axis=1).astype(np.float64)
    ks = set(kept)
    before = []
    for i in range(len(dec)):
        worst = max((onms.rotated_iou(bev[i], bev[j]) for j in before), default=-1.0)
        if (worst > thr) == (i in ks):                  # the decisions differ
            assert abs(worst - thr) < band, (i, worst, thr)
        if i in ks:
            before.append(i)
    return kept

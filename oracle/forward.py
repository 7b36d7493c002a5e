"""Plain forward pass of the fork-join intermediate-fusion detector (oracle).

TEST INFRASTRUCTURE ONLY -- see ``oracle/__init__.py``.

The paper's DNN (Sec. III-B, Sec. V-A-1) is a PointPillars-based intermediate
fusion detector: K independent per-agent encoder branches E_k, then a shared
post-join subgraph (fusion and the classification/regression heads).  The paper
states the structure but not the layer arithmetic, so each step below is the
textbook definition of the named PointPillars operation; where the paper is
silent, each function's docstring states the reading it takes.

All arithmetic is float64, except where a floating-point value decides an
integer (the pillar index of a point), which is taken in float32 as the CUDA
path does.  ``store`` selects the storage-rounded mode: weights and every
stored activation are rounded to "fp16" or "bf16" (round to nearest even),
matching the points where the GPU path stores 16-bit values; accumulation stays
float64.  ``store=None`` is the pure float64 forward.
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence

import numpy as np

from . import nms

# --------------------------------------------------------------------------
# storage rounding
# --------------------------------------------------------------------------


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round to bfloat16 (8-bit significand), nearest-even, via float32 bits."""
    f = np.asarray(x, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    return r.astype(np.uint32).view(np.float32).astype(np.float64)


def store_round(x: np.ndarray, store: Optional[str]) -> np.ndarray:
    """Round a float64 array to the storage type (identity when store is None)."""
    x = np.asarray(x, dtype=np.float64)
    if store is None:
        return x
    if store == "fp16":
        return x.astype(np.float16).astype(np.float64)
    if store == "bf16":
        return round_bf16(x)
    raise ValueError(store)


def relu(v: np.ndarray) -> np.ndarray:
    """max(v, 0) with a canonical +0 for every non-positive input."""
    return np.where(v > 0.0, v, 0.0)


# --------------------------------------------------------------------------
# O1 pillarisation
# --------------------------------------------------------------------------


def point_cells(points: np.ndarray, cfg) -> tuple:
    """Pillar coordinates of each point, decided in float32.

    ix = floor((x - x_min) / v), iy likewise, each subtraction and division an
    IEEE float32 operation with round-to-nearest.  A point is in range iff
    z_min <= z < z_max, 0 <= ix < W and 0 <= iy < H (half-open boxes).
    Returns (ix, iy, in_range) as int64, int64, bool arrays.
    """
    p = np.asarray(points, dtype=np.float32)
    v = np.float32(cfg.pillar)
    fx = (p[:, 0] - np.float32(cfg.x_min)) / v
    fy = (p[:, 1] - np.float32(cfg.y_min)) / v
    assert fx.dtype == np.float32 and fy.dtype == np.float32
    ix = np.floor(fx).astype(np.int64)
    iy = np.floor(fy).astype(np.int64)
    z = p[:, 2]
    ok = (z >= np.float32(cfg.z_min)) & (z < np.float32(cfg.z_max))
    ok &= (ix >= 0) & (ix < cfg.grid_w) & (iy >= 0) & (iy < cfg.grid_h)
    return ix, iy, ok


def pillarise(points: np.ndarray, cfg, max_pillars: Optional[int] = None,
              max_pts: Optional[int] = None) -> Dict[str, np.ndarray]:
    """Group points into pillars, sequentially in point order.

    Points are visited i = 0..n-1.  An out-of-range point is dropped.  A point
    whose cell has no pillar yet opens the next pillar id, unless P_max pillars
    exist already (then it is dropped); a point whose pillar already holds N_max
    points is dropped.  Pillar ids are therefore the ranks of the kept cells'
    first occurrences, and each pillar keeps its first N_max points in order.

    Returns cell2pillar [H*W] (-1 = empty), pillar_cell [P], count [P],
    members [P][N_max] point indices (-1 pad), pts [P][N_max][4] float32 (0
    pad), n_pillars, and drop counters.
    """
    P = cfg.max_pillars if max_pillars is None else max_pillars
    N = cfg.max_pts if max_pts is None else max_pts
    W, H = cfg.grid_w, cfg.grid_h
    ix, iy, ok = point_cells(points, cfg)
    cell2pillar = np.full(W * H, -1, dtype=np.int64)
    pillar_cell: List[int] = []
    members: List[List[int]] = []
    drop_range = drop_pcap = drop_ncap = 0
    for i in range(points.shape[0]):
        if not ok[i]:
            drop_range += 1
            continue
        c = int(iy[i]) * W + int(ix[i])
        p = int(cell2pillar[c])
        if p < 0:
            if len(pillar_cell) == P:
                drop_pcap += 1
                continue
            p = len(pillar_cell)
            cell2pillar[c] = p
            pillar_cell.append(c)
            members.append([])
        if len(members[p]) == N:
            drop_ncap += 1
            continue
        members[p].append(i)
    n_p = len(pillar_cell)
    mem = np.full((P, N), -1, dtype=np.int64)
    cnt = np.zeros(P, dtype=np.int64)
    for p, m in enumerate(members):
        mem[p, :len(m)] = m
        cnt[p] = len(m)
    pts = np.zeros((P, N, 4), dtype=np.float32)
    valid = mem >= 0
    pts[valid] = np.asarray(points, dtype=np.float32)[mem[valid]]
    pc = np.full(P, -1, dtype=np.int64)
    pc[:n_p] = pillar_cell
    return {
        "cell2pillar": cell2pillar, "pillar_cell": pc, "count": cnt,
        "members": mem, "pts": pts, "n_pillars": n_p,
        "drop_range": drop_range, "drop_pcap": drop_pcap, "drop_ncap": drop_ncap,
    }


# --------------------------------------------------------------------------
# O2 pillar feature net, O3 scatter
# --------------------------------------------------------------------------


def pfn_features(pill: Dict[str, np.ndarray], cfg) -> np.ndarray:
    """Augmented 9-d point features [P][N][9] (float64, 0 on padding slots).

    f = (x, y, z, i, x - mean_x, y - mean_y, z - mean_z, x - x_c, y - y_c):
    the means run over the pillar's kept points; (x_c, y_c) is the centre of
    the pillar's cell, x_c = x_min + (ix + 0.5) v.
    """
    pts = pill["pts"].astype(np.float64)
    cnt = pill["count"]
    P, N, _ = pts.shape
    valid = np.arange(N)[None, :] < cnt[:, None]
    safe = np.maximum(cnt, 1)[:, None]
    mean = (pts[:, :, :3] * valid[:, :, None]).sum(axis=1) / safe
    cell = np.maximum(pill["pillar_cell"], 0)
    cix = cell % cfg.grid_w
    ciy = cell // cfg.grid_w
    xc = cfg.x_min + (cix + 0.5) * cfg.pillar
    yc = cfg.y_min + (ciy + 0.5) * cfg.pillar
    f = np.zeros((P, N, 9))
    f[:, :, 0:4] = pts
    f[:, :, 4:7] = pts[:, :, :3] - mean[:, None, :]
    f[:, :, 7] = pts[:, :, 0] - xc[:, None]
    f[:, :, 8] = pts[:, :, 1] - yc[:, None]
    f[~valid] = 0.0
    return f


def pfn(pill: Dict[str, np.ndarray], w: np.ndarray, b: np.ndarray, cfg,
        store: Optional[str] = None) -> np.ndarray:
    """Pillar feature net: h_j = max over kept points of ReLU(sum_d W_jd f_d + b_j).

    A linear layer (BatchNorm folded into the bias), ReLU, and a max over the
    pillar's kept points only; padding slots never enter the max.  Returns
    [P][C] (rows of empty pillar ids are 0), rounded to the storage type.
    """
    f = pfn_features(pill, cfg)
    W = store_round(w, store)
    B = store_round(b, store)
    lin = relu(f @ W.T + B)                      # [P][N][C]
    N = f.shape[1]
    valid = np.arange(N)[None, :] < pill["count"][:, None]
    lin = np.where(valid[:, :, None], lin, -np.inf)
    h = lin.max(axis=1)
    h[pill["count"] == 0] = 0.0
    return store_round(h, store)


def scatter(h: np.ndarray, pill: Dict[str, np.ndarray], cfg) -> np.ndarray:
    """BEV pseudo-image [C][H][W]: pillar p's vector at its cell, zero elsewhere."""
    C = h.shape[1]
    img = np.zeros((C, cfg.grid_h, cfg.grid_w))
    n = pill["n_pillars"]
    cell = pill["pillar_cell"][:n]
    img.reshape(C, -1)[:, cell] = h[:n].T
    return img


# --------------------------------------------------------------------------
# O4 backbone: 3x3 convolutions and deconvolutions
# --------------------------------------------------------------------------


def conv3x3(x: np.ndarray, w: np.ndarray, b: np.ndarray, stride: int) -> np.ndarray:
    """Cross-correlation with a 3x3 kernel, zero padding 1, given stride, + bias.

    y[co, oy, ox] = b[co] + sum_{ci,dy,dx} w[co,ci,dy,dx] x[ci, s*oy+dy-1, s*ox+dx-1]
    (x is 0 outside the image).  One matrix product per kernel tap.  No ReLU.
    """
    ci, H, W = x.shape
    co = w.shape[0]
    Ho = (H + 2 - 3) // stride + 1
    Wo = (W + 2 - 3) // stride + 1
    xp = np.zeros((ci, H + 2, W + 2))
    xp[:, 1:H + 1, 1:W + 1] = x
    y = np.zeros((co, Ho, Wo))
    for dy in range(3):
        for dx in range(3):
            patch = xp[:, dy:dy + stride * (Ho - 1) + 1:stride,
                       dx:dx + stride * (Wo - 1) + 1:stride]
            y += np.tensordot(w[:, :, dy, dx], patch, axes=(1, 0))
    return y + b[:, None, None]


def deconv(x: np.ndarray, w: np.ndarray, b: np.ndarray, s: int) -> np.ndarray:
    """Transposed convolution with kernel = stride = s, no padding, + bias.

    y[co, oy, ox] = b[co] + sum_ci w[ci, co, oy mod s, ox mod s] x[ci, oy // s, ox // s].
    Output windows do not overlap.  No ReLU.
    """
    ci, H, W = x.shape
    co = w.shape[1]
    y = np.zeros((co, H * s, W * s))
    for sy in range(s):
        for sx in range(s):
            y[:, sy::s, sx::s] = np.tensordot(w[:, :, sy, sx], x, axes=(0, 0))
    return y + b[:, None, None]


def encoder(points: np.ndarray, weights: Dict[str, np.ndarray], cfg,
            store: Optional[str] = None) -> Dict[str, np.ndarray]:
    """Encoder branch E_k: pillarise -> PFN -> scatter -> backbone -> neck.

    Backbone block b: n 3x3 convs of C_b channels, the first with the block's
    stride, each followed by ReLU.  Neck: per block a deconv (kernel = stride =
    up_strides[b]) to up_ch channels + ReLU, concatenated in block order.  With
    no neck, the feature map is the last block's output.  Every conv/deconv
    output is rounded to the storage type.
    """
    pill = pillarise(points, cfg)
    h = pfn(pill, weights["pfn.w"], weights["pfn.b"], cfg, store)
    image = scatter(h, pill, cfg)
    x = image
    outs = []
    for bi, (n, _ch, st) in enumerate(cfg.blocks):
        for li in range(n):
            w = store_round(weights[f"b{bi}.c{li}.w"], store)
            bb = store_round(weights[f"b{bi}.c{li}.b"], store)
            x = store_round(relu(conv3x3(x, w, bb, st if li == 0 else 1)), store)
        outs.append(x)
    feat = neck(outs, weights, cfg, store) if cfg.up_strides else outs[-1]
    return {"pillars": pill, "pfn": h, "image": image, "blocks": outs, "feat": feat}


def neck(blocks: Sequence[np.ndarray], weights: Dict[str, np.ndarray], cfg,
         store: Optional[str] = None) -> np.ndarray:
    """Per block a deconv (kernel = stride = up_strides[b]) to up_ch channels
    + ReLU, outputs rounded to the storage type, concatenated in block order."""
    ups = []
    for bi, s in enumerate(cfg.up_strides):
        w = store_round(weights[f"up{bi}.w"], store)
        bb = store_round(weights[f"up{bi}.b"], store)
        ups.append(store_round(relu(deconv(blocks[bi], w, bb, s)), store))
    return np.concatenate(ups, axis=0)


# --------------------------------------------------------------------------
# O5 fusion, O6 head, O7 decode
# --------------------------------------------------------------------------


def fuse_max(feats: Sequence[Optional[np.ndarray]]) -> np.ndarray:
    """Elementwise max over the present agents' feature maps, in index order.

    F = X_first; then F = X_k where X_k > F, for the remaining present k.
    """
    present = [f for f in feats if f is not None]
    F = present[0].copy()
    for X in present[1:]:
        F = np.where(X > F, X, F)
    return F


def fuse_attn(feats: Sequence[Optional[np.ndarray]]) -> np.ndarray:
    """Per-cell scaled dot-product attention with the ego agent (index 0) as query.

    For each cell, s_k = <X_0, X_k> / sqrt(C) over present agents k (absent
    agents are masked out), w = softmax(s), F = sum_k w_k X_k.  No learned
    projections.
    """
    assert feats[0] is not None, "the ego agent must be present"
    C = feats[0].shape[0]
    present = [k for k, f in enumerate(feats) if f is not None]
    X0 = feats[0]
    s = np.stack([(X0 * feats[k]).sum(axis=0) / math.sqrt(C) for k in present])
    m = s.max(axis=0)
    e = np.exp(s - m)
    w = e / e.sum(axis=0)
    F = np.zeros_like(X0)
    for j, k in enumerate(present):
        F += w[j] * feats[k]
    return F


def head(F: np.ndarray, w: np.ndarray, b: np.ndarray) -> np.ndarray:
    """1x1 convolution: out[o, y, x] = b[o] + sum_c w[o, c] F[c, y, x] (no ReLU)."""
    return np.tensordot(w, F, axes=(1, 0)) + b[:, None, None]


ANCHOR_LWH = (3.9, 1.6, 1.56)
ANCHOR_Z = -1.0
EXP_CLAMP = 10.0


def decode(hd: np.ndarray, cfg, cls_thresh: Optional[float] = None,
           max_boxes: Optional[int] = None) -> Dict[str, np.ndarray]:
    """Anchor decode, threshold and deterministic top-K of the head output.

    Channels: [0, A) are the per-anchor class logits, [A + 7a, A + 7a + 7) the
    regression (dx, dy, dz, dl, dw, dh, dyaw) of anchor a.  Anchor index
    idx = (iy * W' + ix) * A + a; anchor a sits at the cell centre, z = -1,
    size (3.9, 1.6, 1.56), yaw = a * pi / A.  A candidate is kept iff its
    logit >= cls_thresh (i.e. score >= sigmoid(cls_thresh)); candidates are
    ordered by logit descending, then index ascending, and cut to max_boxes.
    Box: x = x_a + dx d_a, y = y_a + dy d_a (d_a = sqrt(l_a^2 + w_a^2)),
    z = z_a + dz h_a, l = l_a exp(min(dl, 10)) (w, h likewise),
    yaw = yaw_a + dyaw, score = 1 / (1 + exp(-logit)).
    """
    thr = cfg.cls_thresh if cls_thresh is None else cls_thresh
    kmax = cfg.max_boxes if max_boxes is None else max_boxes
    A = cfg.anchors
    _, Hf, Wf = hd.shape
    cls = hd[:A].transpose(1, 2, 0).reshape(-1)            # idx order
    keep = np.nonzero(cls >= thr)[0]
    order = sorted(keep.tolist(), key=lambda i: (-cls[i], i))[:kmax]
    idx = np.array(order, dtype=np.int64)
    a = idx % A
    cell = idx // A
    ix = cell % Wf
    iy = cell // Wf
    sx = (cfg.x_max - cfg.x_min) / Wf
    sy = (cfg.y_max - cfg.y_min) / Hf
    xa = cfg.x_min + (ix + 0.5) * sx
    ya = cfg.y_min + (iy + 0.5) * sy
    la, wa, ha = ANCHOR_LWH
    da = math.sqrt(la * la + wa * wa)
    reg = np.zeros((len(idx), 7))
    for j in range(7):
        reg[:, j] = hd[A + 7 * a + j, iy, ix]
    boxes = np.zeros((len(idx), 8))
    boxes[:, 0] = xa + reg[:, 0] * da
    boxes[:, 1] = ya + reg[:, 1] * da
    boxes[:, 2] = ANCHOR_Z + reg[:, 2] * ha
    boxes[:, 3] = la * np.exp(np.minimum(reg[:, 3], EXP_CLAMP))
    boxes[:, 4] = wa * np.exp(np.minimum(reg[:, 4], EXP_CLAMP))
    boxes[:, 5] = ha * np.exp(np.minimum(reg[:, 5], EXP_CLAMP))
    boxes[:, 6] = a * math.pi / A + reg[:, 6]
    boxes[:, 7] = 1.0 / (1.0 + np.exp(-cls[idx]))
    return {"idx": idx, "boxes": boxes}


def detect(hd: np.ndarray, cfg) -> Dict[str, np.ndarray]:
    """The final detections: the decode's top-K, then greedy rotated BEV NMS
    at ``cfg.nms_iou`` (see :mod:`oracle.nms`); ``nms_iou <= 0`` skips it.

    The paper's T^det ends after box decoding, score thresholding and rotated
    NMS (Sec. V-A-3).
    """
    det = decode(hd, cfg)
    thr = getattr(cfg, "nms_iou", 0.0)
    if thr > 0 and len(det["idx"]):
        keep = nms.nms(nms.bev(det["boxes"]), thr)
        det = {"idx": det["idx"][keep], "boxes": det["boxes"][keep]}
    return det


# --------------------------------------------------------------------------
# whole frame
# --------------------------------------------------------------------------


def forward_multiscale(points: Sequence[Optional[np.ndarray]], weights: Dict[str, np.ndarray],
                       cfg, store: Optional[str] = None) -> Dict[str, object]:
    """The paper's placement of the fusion (Sec. IV-A; Sec. IV-D): every
    present agent's encoder runs up to its backbone blocks; each block's
    output is fused across the agents (the same per-cell max, or ego-query
    attention at that block's channel count), rounded to the storage type;
    the deconv neck and the concatenation then run once, after the join, on
    the fused maps; then the head and the detections.  Parity unpinned
    against the GPU (no kernel yet); pinned by the reductions in
    tests/test_oracle_layers.py.
    """
    enc = [None if p is None else encoder(p, weights, cfg, store) for p in points]
    fuse = fuse_max if cfg.fusion == "max" else fuse_attn
    fused = [store_round(fuse([None if e is None else e["blocks"][bi] for e in enc]), store)
             for bi in range(len(cfg.blocks))]
    F = neck(fused, weights, cfg, store) if cfg.up_strides else fused[-1]
    hw = store_round(weights["head.w"], store)
    hb = store_round(weights["head.b"], store)
    hd = head(F, hw, hb)
    return {"enc": enc, "fused_blocks": fused, "fused": F, "head": hd, "det": detect(hd, cfg)}


def forward(points: Sequence[Optional[np.ndarray]], weights: Dict[str, np.ndarray], cfg,
            store: Optional[str] = None) -> Dict[str, object]:
    """One frame: every present agent's encoder, then fusion, head, decode and NMS.

    ``points[k] is None`` marks agent k absent (masked out of the fusion).  The
    result does not depend on the order or time at which encoders run: each
    writes the slot of its own agent index (Sec. IV-D), which is why RTCC and
    Barrier produce identical outputs.
    """
    enc = [None if p is None else encoder(p, weights, cfg, store) for p in points]
    feats = [None if e is None else e["feat"] for e in enc]
    F = fuse_max(feats) if cfg.fusion == "max" else fuse_attn(feats)
    hw = store_round(weights["head.w"], store)
    hb = store_round(weights["head.b"], store)
    hd = head(F, hw, hb)
    det = detect(hd, cfg)
    return {"enc": enc, "fused": F, "head": hd, "det": det}

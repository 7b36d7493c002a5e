"""Rotated bird's-eye-view non-maximum suppression (oracle).

TEST INFRASTRUCTURE ONLY -- see ``oracle/__init__.py``.

The paper's primary latency endpoint T^det ends when the final detections
exist: box decoding, score thresholding and rotated NMS (Sec. V-A-3).  The
paper names the step but not its arithmetic, so this is the textbook greedy
NMS over rotated BEV rectangles, in float64:

* a box (x, y, l, w, yaw) is the rectangle centred at (x, y) whose length l
  runs along the unit vector (cos yaw, sin yaw) (yaw counter-clockwise from
  +x, the decode's heading) and whose width w runs along (-sin yaw, cos yaw);
* IoU = area(A n B) / (area(A) + area(B) - area(A n B)); the intersection of
  the two convex rectangles is rectangle A clipped by the four half-planes of
  rectangle B (Sutherland-Hodgman), its area by the shoelace formula;
* greedy: boxes are visited in the given order (the decode's rank order, score
  descending); a box is kept iff its IoU with every box kept before it is at
  most the threshold, i.e. a box is suppressed only by kept boxes.
"""
from __future__ import annotations

import math
from typing import List, Sequence

import numpy as np


def box_corners(x: float, y: float, l: float, w: float, yaw: float) -> List[tuple]:
    """Corners of the rectangle in counter-clockwise order (front-left first)."""
    c, s = math.cos(yaw), math.sin(yaw)
    out = []
    for dl, dw in ((0.5, 0.5), (-0.5, 0.5), (-0.5, -0.5), (0.5, -0.5)):
        px, py = dl * l, dw * w
        out.append((x + c * px - s * py, y + s * px + c * py))
    return out


def _cross(ax, ay, bx, by):
    return ax * by - ay * bx


def clip_halfplane(poly: Sequence[tuple], a: tuple, b: tuple) -> List[tuple]:
    """Part of the polygon on the left of (or on) the directed line a -> b."""
    out = []
    n = len(poly)
    ex, ey = b[0] - a[0], b[1] - a[1]
    for k in range(n):
        p, q = poly[k], poly[(k + 1) % n]
        sp = _cross(ex, ey, p[0] - a[0], p[1] - a[1])
        sq = _cross(ex, ey, q[0] - a[0], q[1] - a[1])
        if sp >= 0:
            out.append(p)
        if (sp >= 0) != (sq >= 0):
            t = sp / (sp - sq)
            out.append((p[0] + t * (q[0] - p[0]), p[1] + t * (q[1] - p[1])))
    return out


def polygon_area(poly: Sequence[tuple]) -> float:
    """Shoelace area (positive for counter-clockwise vertices)."""
    n = len(poly)
    s = 0.0
    for k in range(n):
        p, q = poly[k], poly[(k + 1) % n]
        s += p[0] * q[1] - q[0] * p[1]
    return 0.5 * s


def intersection_area(b1: Sequence[float], b2: Sequence[float]) -> float:
    """Area of the intersection of two rotated rectangles (x, y, l, w, yaw)."""
    poly = box_corners(*b1)
    q = box_corners(*b2)
    for k in range(4):
        poly = clip_halfplane(poly, q[k], q[(k + 1) % 4])
        if not poly:
            return 0.0
    return max(polygon_area(poly), 0.0)


def rotated_iou(b1: Sequence[float], b2: Sequence[float]) -> float:
    """IoU of two rotated BEV rectangles given as (x, y, l, w, yaw)."""
    inter = intersection_area(b1, b2)
    union = b1[2] * b1[3] + b2[2] * b2[3] - inter
    return inter / union if union > 0 else 0.0


def bev(boxes: np.ndarray) -> np.ndarray:
    """(x, y, l, w, yaw) columns of decode-format boxes (x, y, z, l, w, h, yaw, ...)."""
    b = np.asarray(boxes, dtype=np.float64)
    return b[:, [0, 1, 3, 4, 6]]


def nms(boxes_bev: np.ndarray, iou_thresh: float) -> List[int]:
    """Greedy NMS in the given order: the indices of the kept boxes, in order."""
    kept: List[int] = []
    for i in range(len(boxes_bev)):
        if all(rotated_iou(boxes_bev[i], boxes_bev[j]) <= iou_thresh for j in kept):
            kept.append(i)
    return kept

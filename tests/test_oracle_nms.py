"""Pins of the oracle's rotated BEV IoU and greedy NMS.

Closed forms (axis-aligned overlaps, the regular octagon of two squares at
45 degrees), corners derived by hand from the heading convention, a brute-force
area count on a fine grid (point-in-rectangle in the box's own frame, written
here independently of the clipping code), invariances of the definition, and
hand-built suppression chains for the greedy rule.
"""
import math

import numpy as np
import pytest

from oracle import nms as N


def test_corners_follow_the_heading_convention():
    # l = 4 along (cos 30deg, sin 30deg), w = 2 along (-sin 30deg, cos 30deg)
    got = N.box_corners(0.0, 0.0, 4.0, 2.0, math.pi / 6)
    want = [(1.2320508075688772, 1.8660254037844386), (-2.2320508075688772, -0.1339745962155614),
            (-1.2320508075688772, -1.8660254037844386), (2.2320508075688772, 0.1339745962155614)]
    np.testing.assert_allclose(np.array(got), np.array(want), atol=1e-12)
    # counter-clockwise: positive shoelace area = l * w
    assert N.polygon_area(got) == pytest.approx(8.0, abs=1e-12)


def test_axis_aligned_iou_is_the_overlap_product():
    rng = np.random.default_rng(0)
    for _ in range(300):
        b = []
        for _k in range(2):
            x, y = rng.uniform(-2, 2, size=2)
            l, w = rng.uniform(0.2, 3, size=2)
            along_y = rng.random() < 0.5
            yaw = (math.pi / 2 if along_y else 0.0) + (math.pi if rng.random() < 0.5 else 0.0)
            ex, ey = (w, l) if along_y else (l, w)              # extents along x and y
            b.append(((x, y, l, w, yaw), (x - ex / 2, x + ex / 2, y - ey / 2, y + ey / 2)))
        (b1, r1), (b2, r2) = b
        ox = max(0.0, min(r1[1], r2[1]) - max(r1[0], r2[0]))
        oy = max(0.0, min(r1[3], r2[3]) - max(r1[2], r2[2]))
        inter = ox * oy
        want = inter / (b1[2] * b1[3] + b2[2] * b2[3] - inter)
        assert N.rotated_iou(b1, b2) == pytest.approx(want, abs=1e-12)


def test_squares_at_45_degrees_meet_in_a_regular_octagon():
    # side-2 squares about one centre, one turned by 45 degrees: the overlap is
    # the regular octagon of inradius 1, area 8 (sqrt 2 - 1); IoU = 1 / sqrt 2
    a, b = (0.3, -0.7, 2.0, 2.0, 0.0), (0.3, -0.7, 2.0, 2.0, math.pi / 4)
    assert N.intersection_area(a, b) == pytest.approx(8 * (math.sqrt(2) - 1), abs=1e-12)
    assert N.rotated_iou(a, b) == pytest.approx(1 / math.sqrt(2), abs=1e-12)


def test_identical_disjoint_and_touching():
    a = (1.0, 2.0, 3.9, 1.6, 0.7)
    assert N.rotated_iou(a, a) == pytest.approx(1.0, abs=1e-12)
    assert N.rotated_iou(a, (40.0, 2.0, 3.9, 1.6, 0.7)) == 0.0
    assert N.rotated_iou((0.5, 0.5, 1.0, 1.0, 0.0), (1.5, 0.5, 1.0, 1.0, 0.0)) == 0.0


def _grid_area(b1, b2, n=700):
    """Brute-force intersection area: count grid points inside both boxes
    (inside = within the half extents in the box's own frame)."""
    def inside(b, px, py):
        x, y, l, w, yaw = b
        c, s = math.cos(yaw), math.sin(yaw)
        u = (px - x) * c + (py - y) * s
        v = -(px - x) * s + (py - y) * c
        return (np.abs(u) <= l / 2) & (np.abs(v) <= w / 2)
    r = max(math.hypot(b1[2], b1[3]), math.hypot(b2[2], b2[3]))
    lo_x, hi_x = min(b1[0], b2[0]) - r, max(b1[0], b2[0]) + r
    lo_y, hi_y = min(b1[1], b2[1]) - r, max(b1[1], b2[1]) + r
    hx, hy = (hi_x - lo_x) / n, (hi_y - lo_y) / n
    px, py = np.meshgrid(lo_x + (np.arange(n) + 0.5) * hx, lo_y + (np.arange(n) + 0.5) * hy)
    cnt = np.count_nonzero(inside(b1, px, py) & inside(b2, px, py))
    # each cell the boundary crosses can be miscounted: bound by perimeters
    bound = 2 * (b1[2] + b1[3] + b2[2] + b2[3]) * math.hypot(hx, hy)
    return cnt * hx * hy, bound


def test_intersection_area_matches_a_grid_count():
    rng = np.random.default_rng(1)
    for _ in range(25):
        b1 = (0.0, 0.0, rng.uniform(1, 5), rng.uniform(0.5, 2), rng.uniform(-math.pi, math.pi))
        b2 = (rng.uniform(-2, 2), rng.uniform(-2, 2), rng.uniform(1, 5), rng.uniform(0.5, 2),
              rng.uniform(-math.pi, math.pi))
        area, bound = _grid_area(b1, b2)
        assert abs(N.intersection_area(b1, b2) - area) <= bound


def test_heading_turns_counter_clockwise():
    # a thin box turned by +0.5 rad reaches a square placed along that heading
    # (and would miss it if the heading turned clockwise)
    a = (0.0, 0.0, 6.0, 0.5, 0.5)
    b = (2.5 * math.cos(0.5), 2.5 * math.sin(0.5), 1.0, 1.0, 0.0)
    area, bound = _grid_area(a, b)
    assert area > 0.3 and abs(N.intersection_area(a, b) - area) <= bound
    assert N.intersection_area(a, (b[0], -b[1], 1.0, 1.0, 0.0)) == 0.0


def test_iou_invariances():
    rng = np.random.default_rng(2)
    for _ in range(50):
        b1 = tuple(rng.uniform([-2, -2, 0.5, 0.5, -4], [2, 2, 5, 3, 4]))
        b2 = tuple(rng.uniform([-2, -2, 0.5, 0.5, -4], [2, 2, 5, 3, 4]))
        v = N.rotated_iou(b1, b2)
        assert 0.0 <= v <= 1.0
        assert N.rotated_iou(b2, b1) == pytest.approx(v, abs=1e-12)
        flipped = b1[:4] + (b1[4] + math.pi,)
        assert N.rotated_iou(flipped, b2) == pytest.approx(v, abs=1e-12)
        # one rigid motion of both boxes
        th, tx, ty = rng.uniform(-3, 3), rng.uniform(-5, 5), rng.uniform(-5, 5)
        c, s = math.cos(th), math.sin(th)
        mv = lambda b: (c * b[0] - s * b[1] + tx, s * b[0] + c * b[1] + ty, b[2], b[3], b[4] + th)
        assert N.rotated_iou(mv(b1), mv(b2)) == pytest.approx(v, abs=1e-10)


def _unit(x):
    return (x, 0.0, 1.0, 1.0, 0.0)


def test_nms_suppresses_only_by_kept_boxes():
    # A-B and B-C overlap with IoU 1/2, A-C with IoU 1/5: B falls to A, and C
    # stays because its only strong overlap is the suppressed B
    boxes = np.array([_unit(0.0), _unit(1 / 3), _unit(2 / 3)])
    assert N.rotated_iou(boxes[0], boxes[1]) == pytest.approx(0.5, abs=1e-12)
    assert N.rotated_iou(boxes[0], boxes[2]) == pytest.approx(0.2, abs=1e-12)
    assert N.nms(boxes, 0.3) == [0, 2]
    assert N.nms(boxes, 0.49) == [0, 2]
    assert N.nms(boxes, 0.51) == [0, 1, 2]
    assert N.nms(boxes, 0.1) == [0]


def test_nms_edge_cases():
    assert N.nms(np.zeros((0, 5)), 0.5) == []
    assert N.nms(np.array([_unit(0.0)]), 0.5) == [0]
    rng = np.random.default_rng(3)
    boxes = np.column_stack([rng.uniform(-3, 3, 20), rng.uniform(-3, 3, 20), rng.uniform(1, 4, 20),
                             rng.uniform(0.5, 2, 20), rng.uniform(-3, 3, 20)])
    assert N.nms(boxes, 1.0) == list(range(20))          # IoU never exceeds 1
    assert N.nms(boxes, -1.0) == [0]                     # every pair exceeds -1


@pytest.mark.parametrize("seed", range(6))
def test_nms_result_is_the_greedy_fixed_point(seed):
    # the kept set S is characterised by: i in S iff no j in S with j < i
    # overlaps i above the threshold
    rng = np.random.default_rng(10 + seed)
    n = 30
    boxes = np.column_stack([rng.uniform(-4, 4, n), rng.uniform(-4, 4, n), rng.uniform(1, 4, n),
                             rng.uniform(0.5, 2, n), rng.uniform(-3, 3, n)])
    thr = 0.15
    S = set(N.nms(boxes, thr))
    assert 0 in S
    for i in range(n):
        hit = any(N.rotated_iou(boxes[i], boxes[j]) > thr for j in S if j < i)
        assert (i in S) == (not hit)

"""GPU rotated BEV NMS (rtcc_nms) against the oracle's float64 IoU and greedy
rule, on constructed box sets: ragged and full 32-box chunks, the largest
list (512), duplicates, disjoint sets, suppression chains, and thresholds 0
and 1."""
import math

import numpy as np
import pytest

from tests import gpu_util as U

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def R():
    return U.load()


def _boxes(rows):
    b = np.zeros(len(rows), dtype=U.R.BOX_DTYPE)
    for i, (x, y, l, w, yaw) in enumerate(rows):
        b[i] = (x, y, -1.0, l, w, 1.5, yaw, 1.0 - i * 1e-3, i)
    return b


def _crowd(n, seed, spread=12.0):
    """n car-sized boxes around a few centres, so many pairs overlap."""
    rng = np.random.default_rng(seed)
    centres = rng.uniform(-spread, spread, size=(max(1, n // 24), 2))
    c = centres[rng.integers(0, len(centres), n)]
    xy = c + rng.normal(scale=1.0, size=(n, 2))
    l = 3.9 * np.exp(rng.normal(scale=0.2, size=n))
    w = 1.6 * np.exp(rng.normal(scale=0.2, size=n))
    yaw = rng.choice([0.0, math.pi / 2], n) + rng.normal(scale=0.3, size=n)
    return _boxes(np.column_stack([xy[:, 0], xy[:, 1], l, w, yaw]))


@pytest.mark.parametrize("n,seed", [(1, 0), (31, 1), (32, 2), (33, 3), (200, 4), (512, 5)])
@pytest.mark.parametrize("thr", [0.15, 0.5])
def test_nms_crowded_sets(R, n, seed, thr):
    b = _crowd(n, seed)
    out = R.rtcc_nms(b, thr)
    kept = U.check_nms(b, out, thr)
    assert kept[0] == 0
    if n >= 200:
        assert len(kept) < n                           # the crowd does overlap


def test_nms_edge_cases(R):
    assert len(R.rtcc_nms(np.zeros(0, dtype=R.BOX_DTYPE), 0.15)) == 0
    same = _boxes([(5.0, -3.0, 3.9, 1.6, 0.4)] * 40)
    same["anchor"] = np.arange(40)
    assert R.rtcc_nms(same, 0.15)["anchor"].tolist() == [0]
    far = _boxes([(10.0 * i, 0.0, 3.9, 1.6, 0.1 * i) for i in range(64)])
    assert R.rtcc_nms(far, 0.0)["anchor"].tolist() == list(range(64))
    # A-B and B-C at IoU 1/2, A-C at 1/5: B falls to A, C survives
    chain = _boxes([(0.0, 0.0, 1.0, 1.0, 0.0), (1 / 3, 0.0, 1.0, 1.0, 0.0), (2 / 3, 0.0, 1.0, 1.0, 0.0)])
    assert R.rtcc_nms(chain, 0.3)["anchor"].tolist() == [0, 2]
    assert R.rtcc_nms(chain, 0.1)["anchor"].tolist() == [0]
    crowd = _crowd(128, 9)
    assert R.rtcc_nms(crowd, 1.0)["anchor"].tolist() == list(range(128))
    out = R.rtcc_nms(crowd, 0.0)                         # any overlap suppresses
    U.check_nms(crowd, out, 0.0)

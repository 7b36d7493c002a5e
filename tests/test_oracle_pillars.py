"""Pins of the oracle's pillarisation, pillar feature net and scatter.

Each check is independent of the oracle's own formulation: points built inside
known cells, an O(n^2) brute force over "first occurrence" and "earlier points
of the same cell", conservation laws, hand-derivable special cases.
"""
import numpy as np
import pytest

import synth
from oracle import forward as of

TINY = synth.get_config("tiny")


def _cfg(**kw):
    return synth.get_config("tiny", **kw)


def _brute(points, cfg, P, N, cells):
    """O(n^2) restatement: a cell is kept iff fewer than P distinct cells occur
    before its first point; a point is kept iff its cell is kept and fewer than
    N in-range points of that cell precede it."""
    n = len(points)
    inr = cells >= 0
    first = {}
    for i in range(n):
        if inr[i] and cells[i] not in first:
            first[cells[i]] = i
    firsts = sorted(first.values())
    pid_of = {}
    for c, f in first.items():
        rank = sum(1 for g in firsts if g < f)
        if rank < P:
            pid_of[c] = rank
    members = {p: [] for p in pid_of.values()}
    for i in range(n):
        if not inr[i] or cells[i] not in pid_of:
            continue
        earlier = int(np.sum(cells[:i] == cells[i]))
        if earlier < N:
            members[pid_of[cells[i]]].append(i)
    return pid_of, members


def _patch(n, cells, seed):
    return synth.points_cap_patch(n=n, cells=cells, seed=seed)


def test_point_cells_known_construction():
    pts = _patch(500, 8, 1)
    ix, iy, ok = of.point_cells(pts, TINY)
    # by construction x = -12.8 + (cx + frac) * 0.4 with frac in [0.05, 0.95]
    cx = np.floor((pts[:, 0].astype(np.float64) + 12.8) / 0.4 + 1e-9).astype(int)
    cy = np.floor((pts[:, 1].astype(np.float64) + 12.8) / 0.4 + 1e-9).astype(int)
    assert ok.all()
    assert (ix == cx).all() and (iy == cy).all()


@pytest.mark.parametrize("seed,P,N", [(0, 10, 3), (1, 5, 1), (2, 64, 64), (3, 1, 4), (4, 20, 7)])
def test_pillarise_matches_bruteforce(seed, P, N):
    rng = np.random.default_rng(seed)
    cfg = _cfg(grid_w=6, grid_h=5, x_min=0.0, y_min=0.0, x_max=2.4, y_max=2.0, pillar=0.4)
    n = 400
    pts = np.empty((n, 4), dtype=np.float32)
    pts[:, 0] = rng.uniform(-0.5, 2.9, n)          # some out of range in x
    pts[:, 1] = rng.uniform(-0.3, 2.3, n)
    pts[:, 2] = rng.uniform(-3.5, 1.5, n)          # some out of range in z
    pts[:, 3] = rng.uniform(0, 1, n)
    ix, iy, ok = of.point_cells(pts, cfg)
    cells = np.where(ok, iy * cfg.grid_w + ix, -1)
    pid_of, members = _brute(pts, cfg, P, N, cells)
    got = of.pillarise(pts, cfg, max_pillars=P, max_pts=N)
    assert got["n_pillars"] == len(pid_of)
    for c, p in pid_of.items():
        assert got["cell2pillar"][c] == p
        assert got["pillar_cell"][p] == c
        assert got["count"][p] == len(members[p])
        assert list(got["members"][p, :got["count"][p]]) == members[p]
    assert (got["cell2pillar"] >= 0).sum() == len(pid_of)


def test_pillarise_conservation_and_caps():
    cfg = _cfg()
    pts = _patch(2048, 8, 3)
    got = of.pillarise(pts, cfg, max_pillars=16, max_pts=8)
    kept = int(got["count"].sum())
    assert kept + got["drop_range"] + got["drop_pcap"] + got["drop_ncap"] == len(pts)
    assert got["drop_pcap"] > 0 and got["drop_ncap"] > 0     # both caps bind
    assert got["n_pillars"] == 16
    pc = got["pillar_cell"][:16]
    assert len(set(pc.tolist())) == 16
    firsts = [int(got["members"][p, 0]) for p in range(16)]
    assert firsts == sorted(firsts)                          # ids follow first occurrence


def test_pillarise_single_cell_and_single_pillar():
    cfg = _cfg()
    pts = np.zeros((50, 4), dtype=np.float32)
    pts[:, 0] = -12.8 + 5.5 * 0.4
    pts[:, 1] = -12.8 + 7.5 * 0.4
    pts[:, 2] = -1.0
    got = of.pillarise(pts, cfg, max_pillars=4, max_pts=16)
    assert got["n_pillars"] == 1 and got["count"][0] == 16 and got["drop_ncap"] == 34
    assert got["pillar_cell"][0] == 7 * 64 + 5
    many = _patch(300, 8, 5)
    one = of.pillarise(many, cfg, max_pillars=1, max_pts=1000)
    assert one["n_pillars"] == 1
    ix, iy, _ = of.point_cells(many[:1], cfg)
    assert one["pillar_cell"][0] == iy[0] * 64 + ix[0]


def test_pillarise_half_open_boundaries():
    cfg = _cfg()
    pts = np.array([
        [-12.8, -12.8, -3.0, 0.5],     # lower corners: kept, cell (0, 0)
        [12.8, 0.0, 0.0, 0.5],         # x == x_max: dropped
        [0.0, 12.8, 0.0, 0.5],         # y == y_max: dropped
        [0.0, 0.0, 1.0, 0.5],          # z == z_max: dropped
        [0.0, 0.0, -3.0001, 0.5],      # z < z_min: dropped
        [-12.80001, 0.0, 0.0, 0.5],    # x < x_min: dropped
    ], dtype=np.float32)
    got = of.pillarise(pts, cfg)
    assert got["n_pillars"] == 1 and got["pillar_cell"][0] == 0 and got["drop_range"] == 5


def _two_point_pillar():
    cfg = _cfg(pfn_ch=9)
    cx, cy = 10, 20
    xc, yc = -12.8 + (cx + 0.5) * 0.4, -12.8 + (cy + 0.5) * 0.4
    p1 = np.array([xc - 0.1, yc + 0.15, -1.0, 0.25], dtype=np.float32)
    p2 = np.array([xc + 0.05, yc - 0.05, -2.0, 0.75], dtype=np.float32)
    pts = np.stack([p1, p2])
    return cfg, pts, (xc, yc)


def test_pfn_features_two_point_by_hand():
    cfg, pts, (xc, yc) = _two_point_pillar()
    pill = of.pillarise(pts, cfg)
    w = np.eye(9)
    h_pos = of.pfn(pill, w, np.zeros(9), cfg)[0]
    h_neg = of.pfn(pill, -w, np.zeros(9), cfg)[0]
    p = pts.astype(np.float64)
    half = np.abs(p[0, :3] - p[1, :3]) / 2.0
    # max_j ReLU(f_j) and max_j ReLU(-f_j) over the two points, derived by hand
    exp_pos = [max(p[0, 0], p[1, 0], 0), max(p[0, 1], p[1, 1], 0), 0.0, 0.75,
               half[0], half[1], half[2],
               max(p[0, 0] - xc, p[1, 0] - xc, 0), max(p[0, 1] - yc, p[1, 1] - yc, 0)]
    exp_neg = [max(-p[0, 0], -p[1, 0], 0), max(-p[0, 1], -p[1, 1], 0), 2.0, 0.0,
               half[0], half[1], half[2],
               max(xc - p[0, 0], xc - p[1, 0], 0), max(yc - p[0, 1], yc - p[1, 1], 0)]
    np.testing.assert_allclose(h_pos, exp_pos, rtol=0, atol=1e-6)
    np.testing.assert_allclose(h_neg, exp_neg, rtol=0, atol=1e-6)


def test_pfn_single_point_offsets_vanish():
    cfg = _cfg(pfn_ch=9)
    pts = np.array([[1.01, -2.03, -0.5, 0.3]], dtype=np.float32)
    pill = of.pillarise(pts, cfg)
    f = of.pfn_features(pill, cfg)[0, 0]
    assert np.all(f[4:7] == 0.0)
    np.testing.assert_allclose(f[:4], pts[0].astype(np.float64))


def test_pfn_point_order_within_pillar_is_irrelevant():
    cfg = _cfg()
    w = synth.weights_for(cfg)
    pts = _patch(400, 4, 9)
    pill = of.pillarise(pts, cfg)
    h = of.pfn(pill, w["pfn.w"], w["pfn.b"], cfg)
    perm = pill["pts"].copy()
    rng = np.random.default_rng(0)
    for p in range(pill["n_pillars"]):
        c = pill["count"][p]
        perm[p, :c] = perm[p, rng.permutation(c)]
    pill2 = dict(pill, pts=perm)
    h2 = of.pfn(pill2, w["pfn.w"], w["pfn.b"], cfg)
    np.testing.assert_allclose(h, h2, rtol=1e-12, atol=1e-12)


def test_scatter_occupancy_equals_pillar_map():
    cfg = _cfg()
    w = synth.weights_for(cfg)
    pts = synth.points_for(cfg, 0, 0)
    pill = of.pillarise(pts, cfg)
    h = of.pfn(pill, w["pfn.w"], np.full(cfg.pfn_ch, 1.0), cfg)   # strictly positive
    img = of.scatter(h, pill, cfg)
    occ = (img != 0).any(axis=0).reshape(-1)
    assert (occ == (pill["cell2pillar"] >= 0)).all()
    p = 5
    c = pill["pillar_cell"][p]
    np.testing.assert_array_equal(img[:, c // cfg.grid_w, c % cfg.grid_w], h[p])


def test_store_round_matches_torch_casts():
    torch = pytest.importorskip("torch")
    x = np.random.default_rng(0).normal(0, 30, 10000)
    x[:10] = [0.0, -0.0, 1e-8, 65504.0, 1.0 + 2**-11, 1.0 + 3 * 2**-11, 255.5, -3.75, 1e5, 7e-6]
    h = torch.tensor(x, dtype=torch.float64).to(torch.float16).double().numpy()
    bf = torch.tensor(x, dtype=torch.float64).float().to(torch.bfloat16).double().numpy()
    np.testing.assert_array_equal(of.store_round(x, "fp16"), h)
    np.testing.assert_array_equal(of.store_round(x, "bf16"), bf)

"""Host-side checks of the backbone's tile plan (rtcc_plan_conv; no GPU).

The backbone cuts each 3x3 conv layer into work items: K slices (split-K),
an N tile, and a pixel tile of 8 x 16, 8 x 32 (tall), 16 x 8 (wide), or
8 x 16 / 8 x 32 walked with the image's rows as x (transposed).  What the
kernel computes per pixel must not depend on that choice, so these tests
hold the plan to the properties its correctness rests on:

* the K slices (which fix the fp32 summation order) are the same for every
  batch size, so a branch's bytes do not depend on the launch that ran it;
* every shape flag is one the kernel supports for that layer (tall and
  transposed tiles only on halo layers without split-K, wide tiles only on
  layers that load one box per tap);
* the pixel tiles cover every output pixel exactly once, with the tile
  origins and the pixel index the kernel uses for that orientation;
* the item count is what a launch deals out, and no other legal choice has
  a lower modelled cost.
"""
import itertools

import numpy as np
import pytest

import synth
from paper_2608_08330_gb300 import build as B

GRIDS = (144, 152)          # CTAs of a launch with and without clusters of 4


@pytest.fixture(scope="module")
def R():
    B.build()
    from paper_2608_08330_gb300 import rtcc
    rtcc.load()
    return rtcc


def conv_layers(cfg):
    """(kind, cin, cout, out_w, out_h) of every conv layer of the backbone:
    the first layer of a stride-2 block is kind 1."""
    out = []
    w, h, cin = cfg.grid_w, cfg.grid_h, cfg.pfn_ch
    for n_layers, ch, st in cfg.blocks:
        ow, oh = w // st, h // st
        for li in range(n_layers):
            out.append((1 if (li == 0 and st == 2) else 0, cin if li == 0 else ch, ch, ow, oh))
        w, h, cin = ow, oh, ch
    return out


def is_halo(kind, cin, splits):
    return kind == 0 and cin >= 64 and (cin // 64) % splits == 0


def tile_shape(p):
    tw = 16 if p["wide"] else 8
    th = 32 if p["tall"] else (8 if p["wide"] else 16)
    return tw, th


def coverage(p, out_w, out_h):
    """Output pixels each covered how many times by the plan's tiles, with the
    kernel's tile origins (x0, y0) and pixel rows (row % tw, row / tw, the
    tall tile's lower block TH rows further), and its pixel index (h * W + w,
    h and w swapped for transposed tiles)."""
    tw, th = tile_shape(p)
    gx, gy = (out_h, out_w) if p["transposed"] else (out_w, out_h)
    tiles_x = -(-gx // tw)
    hits = np.zeros(out_w * out_h, dtype=np.int32)
    rows = np.arange(128)
    for mt in range(p["m_tiles"]):
        x0, y0 = (mt % tiles_x) * tw, (mt // tiles_x) * th
        for half in range(2 if p["tall"] else 1):
            px = x0 + rows % tw
            py = y0 + half * 16 + rows // tw
            ok = (px < gx) & (py < gy)
            pix = np.where(p["transposed"], px * out_w + py, py * out_w + px)[ok]
            np.add.at(hits, pix, 1)
    return hits


def model_cost(kind, cin, cout, out_w, out_h, grid, nb, splits, bn, tall, tr, wide):
    """The cost the tile picker minimises: rounds of items over the grid x
    k-blocks per item x the k-block's MMA time at that N (x 1.6 for tall)."""
    tw = 16 if wide else 8
    th = 32 if tall else (8 if wide else 16)
    gx, gy = (out_h, out_w) if tr else (out_w, out_h)
    m_tiles = -(-gx // tw) * -(-gy // th)
    items = nb * m_tiles * (cout // bn) * splits
    rounds = -(-items // grid)
    total_kb = 9 * (cin // (64 if cin >= 64 else 32))
    kb = {32: 0.70, 64: 0.75, 128: 1.0}[bn]
    return rounds * -(-total_kb // splits) * kb * (1.6 if tall else 1.0)


def legal_choices(kind, cin, cout, splits):
    halo = is_halo(kind, cin, splits)
    for bn, tall, orient in itertools.product((32, 64, 128), (0, 1), (0, 1)):
        if bn > cout or cout % bn:
            continue
        if tall and (not halo or splits != 1):
            continue
        tr, wide = (orient, 0) if halo else (0, orient)
        if orient and splits != 1:
            continue
        yield bn, tall, tr, wide


@pytest.mark.parametrize("name", list(synth.CONFIGS))
def test_plan_properties_on_every_workload(R, name):
    cfg = synth.get_config(name)
    for layer in conv_layers(cfg):
        kind, cin, cout, out_w, out_h = layer
        for grid in GRIDS:
            plans = [R.rtcc_plan_conv(kind, cin, cout, out_w, out_h, grid, nb)
                     for nb in range(1, cfg.n_agents + 1)]
            # the K slices are the one-agent choice for every batch size
            assert len({p["splits"] for p in plans}) == 1, (layer, plans)
            for nb, p in enumerate(plans, start=1):
                where = (name, layer, grid, nb, p)
                halo = is_halo(kind, cin, p["splits"])
                assert p["splits"] in (1, 4) and p["bn"] in (32, 64, 128) and cout % p["bn"] == 0, where
                assert not (p["tall"] and p["wide"]) and not (p["transposed"] and p["wide"]), where
                if p["tall"] or p["transposed"]:
                    assert halo and p["splits"] == 1, where
                if p["wide"]:
                    assert not halo and p["splits"] == 1, where
                assert p["items"] == nb * p["m_tiles"] * (cout // p["bn"]) * p["splits"], where
                hits = coverage(p, out_w, out_h)
                assert hits.min() == 1 and hits.max() == 1, where
                # no legal choice (same K slices) has a lower modelled cost; a
                # split layer whose items fit the grid keeps 64-wide tiles
                need64 = p["splits"] > 1 and nb * (-(-out_w // 8) * -(-out_h // 16)) * (cout // 64) * 4 <= grid
                best = min(model_cost(kind, cin, cout, out_w, out_h, grid, nb, p["splits"], *c)
                           for c in legal_choices(kind, cin, cout, p["splits"])
                           if not need64 or c[0] == 64)
                got = model_cost(kind, cin, cout, out_w, out_h, grid, nb, p["splits"], p["bn"],
                                 p["tall"], p["transposed"], p["wide"])
                assert got <= best + 1e-9, (where, got, best)


def test_block0_of_the_704x200_grid_uses_the_orientation_with_fewer_rounds(R):
    # 352 x 100 in 8 x 16 tiles is 44 x 7 = 308 tiles, 3 rounds on 152 CTAs;
    # 16 x 8 tiles (stride-2 layer) need 22 x 13 = 286, and tall tiles walked
    # transposed (halo layers) 13 x 11 = 143, one round
    s2 = R.rtcc_plan_conv(1, 64, 64, 352, 100, 152, 1)
    assert (s2["wide"], s2["transposed"], s2["tall"], s2["bn"], s2["items"]) == (1, 0, 0, 64, 286)
    halo = R.rtcc_plan_conv(0, 64, 64, 352, 100, 152, 1)
    assert (halo["tall"], halo["transposed"], halo["wide"], halo["bn"], halo["items"]) == (1, 1, 0, 64, 143)
    # an 8-agent launch: 8 x 143 tall transposed items (8 rounds) against
    # 8 x 176 tall ones (10 rounds)
    halo8 = R.rtcc_plan_conv(0, 64, 64, 352, 100, 152, 8)
    assert (halo8["tall"], halo8["transposed"], halo8["items"]) == (1, 1, 1144)


def test_square_grids_keep_the_plain_orientation(R):
    # pp3's maps (128, 64, 32 pixels square) divide into 8 x 16 tiles either
    # way round, so ties keep the plain orientation
    for layer in conv_layers(synth.get_config("pp3")):
        p = R.rtcc_plan_conv(*layer, 152, 1)
        assert p["transposed"] == 0 and p["wide"] == 0, (layer, p)


@pytest.mark.parametrize("args", [
    (2, 64, 64, 64, 64, 152, 1),        # not a 3x3 conv kind
    (0, 96, 64, 64, 64, 152, 1),        # cin not a power of two
    (0, 64, 48, 64, 64, 152, 1),        # cout not a multiple of 32
    (0, 64, 512, 64, 64, 152, 1),       # cout above 256
    (0, 64, 64, 0, 64, 152, 1),         # empty output
    (0, 64, 64, 64, 64, 0, 1),          # no CTAs
    (0, 64, 64, 64, 64, 152, 0),        # no agents
    (0, 64, 64, 64, 64, 152, 9),        # more agents than RTCC_MAX_AGENTS
])
def test_plan_rejects_bad_arguments(R, args):
    with pytest.raises(R.RTCCError) as e:
        R.rtcc_plan_conv(*args)
    assert e.value.status == R.E_ARG

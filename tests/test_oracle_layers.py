"""Pins of the oracle's conv/deconv backbone, fusion, head and decode.

Library special cases (torch CPU conv2d / conv_transpose2d / scaled dot-product
attention, NumPy max), brute-force loops on tiny tensors, and invariants the
definitions imply (agent-order invariance of max fusion, ego-only attention).
"""
import math

import numpy as np
import pytest

import synth
from oracle import forward as of

torch = pytest.importorskip("torch")
F = torch.nn.functional


def _t(x):
    return torch.tensor(x, dtype=torch.float64)


@pytest.mark.parametrize("ci,co,h,w,s", [(3, 4, 7, 5, 1), (3, 4, 8, 6, 2), (16, 8, 12, 10, 2), (8, 8, 9, 9, 1)])
def test_conv3x3_matches_torch(ci, co, h, w, s):
    rng = np.random.default_rng(ci * 100 + h)
    x = rng.normal(size=(ci, h, w))
    wt = rng.normal(size=(co, ci, 3, 3))
    b = rng.normal(size=co)
    ref = F.conv2d(_t(x)[None], _t(wt), _t(b), stride=s, padding=1)[0].numpy()
    np.testing.assert_allclose(of.conv3x3(x, wt, b, s), ref, rtol=1e-12, atol=1e-12)


def test_conv3x3_bruteforce_tiny():
    rng = np.random.default_rng(5)
    ci, co, h, w = 2, 3, 5, 4
    x = rng.normal(size=(ci, h, w))
    wt = rng.normal(size=(co, ci, 3, 3))
    b = rng.normal(size=co)
    for s in (1, 2):
        ho, wo = (h - 1) // s + 1, (w - 1) // s + 1
        ref = np.zeros((co, ho, wo))
        for o in range(co):
            for oy in range(ho):
                for ox in range(wo):
                    acc = b[o]
                    for c in range(ci):
                        for dy in range(3):
                            for dx in range(3):
                                yy, xx = s * oy + dy - 1, s * ox + dx - 1
                                if 0 <= yy < h and 0 <= xx < w:
                                    acc += wt[o, c, dy, dx] * x[c, yy, xx]
                    ref[o, oy, ox] = acc
        np.testing.assert_allclose(of.conv3x3(x, wt, b, s), ref, rtol=1e-12, atol=1e-12)


def test_conv3x3_identity_kernel():
    x = np.random.default_rng(1).normal(size=(4, 6, 7))
    wt = np.zeros((4, 4, 3, 3))
    for c in range(4):
        wt[c, c, 1, 1] = 1.0
    np.testing.assert_array_equal(of.conv3x3(x, wt, np.zeros(4), 1), x)


@pytest.mark.parametrize("s", [1, 2, 4])
def test_deconv_matches_torch(s):
    rng = np.random.default_rng(s)
    x = rng.normal(size=(6, 5, 3))
    wt = rng.normal(size=(6, 4, s, s))
    b = rng.normal(size=4)
    ref = F.conv_transpose2d(_t(x)[None], _t(wt), _t(b), stride=s)[0].numpy()
    np.testing.assert_allclose(of.deconv(x, wt, b, s), ref, rtol=1e-12, atol=1e-12)


def test_fuse_max_library_and_permutation():
    rng = np.random.default_rng(2)
    X = [of.relu(rng.normal(size=(8, 5, 6))) for _ in range(4)]
    Fm = of.fuse_max(X)
    np.testing.assert_array_equal(Fm, np.max(np.stack(X), axis=0))
    for perm in ([3, 1, 0, 2], [2, 3, 1, 0]):
        got = of.fuse_max([X[i] for i in perm])
        assert got.tobytes() == Fm.tobytes()                  # bit-exact, +0 canonical
    np.testing.assert_array_equal(of.fuse_max([X[0]]), X[0])
    np.testing.assert_array_equal(of.fuse_max([X[0], None, X[2], None]), np.maximum(X[0], X[2]))


def test_fuse_attn_matches_torch_sdpa():
    rng = np.random.default_rng(3)
    C, H, W, K = 16, 4, 5, 5
    X = [rng.normal(size=(C, H, W)) for _ in range(K)]
    present = [True, True, False, True, False]
    feats = [x if p else None for x, p in zip(X, present)]
    got = of.fuse_attn(feats)
    q = _t(np.stack(X)[0]).permute(1, 2, 0).reshape(-1, 1, 1, C)
    kv = _t(np.stack(X)).permute(2, 3, 0, 1).reshape(-1, 1, K, C)
    mask = torch.tensor(present).reshape(1, 1, 1, K)
    ref = F.scaled_dot_product_attention(q, kv, kv, attn_mask=mask)
    ref = ref.reshape(H, W, C).permute(2, 0, 1).numpy()
    np.testing.assert_allclose(got, ref, rtol=1e-10, atol=1e-10)


def test_fuse_attn_special_cases():
    rng = np.random.default_rng(4)
    X0 = rng.normal(size=(8, 3, 3))
    np.testing.assert_allclose(of.fuse_attn([X0, None, None]), X0, rtol=0, atol=0)
    np.testing.assert_allclose(of.fuse_attn([X0, X0.copy(), X0.copy()]), X0, rtol=1e-14, atol=1e-14)
    # constant feature vectors c_k: weights are softmax_k(c_0 c_k sqrt(C)) by hand
    cs = [0.5, -0.2, 0.3]
    C = 8
    Xc = [np.full((C, 2, 2), c) for c in cs]
    s = np.array([cs[0] * c * C / math.sqrt(C) for c in cs])
    wgt = np.exp(s - s.max()) / np.exp(s - s.max()).sum()
    np.testing.assert_allclose(of.fuse_attn(Xc), np.full((C, 2, 2), (wgt * cs).sum()), rtol=1e-13)


def test_head_matches_torch_1x1():
    rng = np.random.default_rng(6)
    Fm = rng.normal(size=(12, 4, 7))
    w = rng.normal(size=(16, 12))
    b = rng.normal(size=16)
    ref = F.conv2d(_t(Fm)[None], _t(w)[:, :, None, None], _t(b))[0].numpy()
    np.testing.assert_allclose(of.head(Fm, w, b), ref, rtol=1e-12, atol=1e-12)


def test_decode_zero_regression_gives_anchors():
    cfg = synth.get_config("tiny")
    A, Hf, Wf = cfg.anchors, cfg.feat_h, cfg.feat_w
    hd = np.zeros((8 * A, Hf, Wf))
    det = of.decode(hd, cfg, cls_thresh=0.0, max_boxes=10 ** 9)
    assert len(det["idx"]) == A * Hf * Wf                 # cls = 0 >= 0 keeps all
    np.testing.assert_array_equal(det["idx"], np.arange(A * Hf * Wf))   # ties -> index order
    b = det["boxes"]
    assert np.all(b[:, 7] == 0.5)
    np.testing.assert_allclose(b[:, 3:6], np.tile([3.9, 1.6, 1.56], (len(b), 1)))
    i = 2 * 37 + 1                                          # cell 37, anchor 1
    assert b[i, 0] == pytest.approx(-12.8 + (37 % Wf + 0.5) * 0.4)
    assert b[i, 1] == pytest.approx(-12.8 + (37 // Wf + 0.5) * 0.4)
    assert b[i, 6] == pytest.approx(math.pi / 2)
    assert b[i, 2] == pytest.approx(-1.0)


def test_decode_threshold_order_and_cut():
    cfg = synth.get_config("tiny")
    A, Hf, Wf = cfg.anchors, cfg.feat_h, cfg.feat_w
    hd = np.full((8 * A, Hf, Wf), 0.0)
    hd[:A] = -5.0
    hd[0, 3, 4] = 2.0          # idx (3*64+4)*2 + 0 = 392
    hd[1, 0, 0] = 2.0          # idx 1 (same logit: smaller index first)
    hd[1, 9, 9] = 3.0          # idx (9*64+9)*2 + 1 = 1171
    hd[0, 1, 1] = -0.5         # below threshold 0
    hd[A + 7 * 0 + 3, 3, 4] = 50.0    # dl clamps at 10
    det = of.decode(hd, cfg, cls_thresh=0.0, max_boxes=2)
    assert det["idx"].tolist() == [1171, 1]
    det = of.decode(hd, cfg, cls_thresh=0.0, max_boxes=10)
    assert det["idx"].tolist() == [1171, 1, 392]
    assert det["boxes"][2, 3] == pytest.approx(3.9 * math.exp(10.0))
    assert det["boxes"][0, 7] == pytest.approx(1 / (1 + math.exp(-3.0)))


def test_forward_tiny_invariances():
    cfg = synth.get_config("tiny")
    w = synth.weights_for(cfg)
    p0, p1 = synth.points_for(cfg, 0, 0), synth.points_for(cfg, 0, 1)
    out = of.forward([p0, p1], w, cfg, store="fp16")
    swapped = of.forward([p1, p0], w, cfg, store="fp16")
    assert out["fused"].tobytes() == swapped["fused"].tobytes()   # max fusion: order-free
    assert out["head"].shape == (16, 64, 64)
    e = out["enc"][0]
    assert e["pillars"]["n_pillars"] > 1000 and e["pillars"]["drop_pcap"] == 0
    # storage-rounded and pure float64 forwards agree to the 16-bit rounding level
    pure = of.forward([p0, p1], w, cfg, store=None)
    assert np.max(np.abs(pure["head"] - out["head"])) < 2e-2 + 1e-2 * np.max(np.abs(pure["head"]))


def _small_neck_cfg(fusion="max", n_agents=2):
    import dataclasses
    base = synth.get_config("pp3")
    return dataclasses.replace(base, n_agents=n_agents, grid_w=32, grid_h=32, x_min=-6.4, x_max=6.4,
                               y_min=-6.4, y_max=6.4, pts_x=(-7.0, 7.0), pts_y=(-7.0, 7.0),
                               n_uniform=1500, n_clusters=2, cluster_pts=100, max_pillars=1024,
                               fusion=fusion, anchors=2)


@pytest.mark.parametrize("fusion", ["max", "attn"])
def test_multiscale_fusion_of_one_agent_is_the_single_scale_path(fusion):
    # one present agent: every per-scale fusion is the identity, so fusing
    # before or after the neck gives the same head, exactly
    cfg = _small_neck_cfg(fusion, n_agents=1)
    w = synth.weights_for(cfg)
    pts = [synth.points_for(cfg, 0, 0)]
    a = of.forward(pts, w, cfg, store="fp16")
    b = of.forward_multiscale(pts, w, cfg, store="fp16")
    np.testing.assert_array_equal(a["head"], b["head"])
    assert a["det"]["idx"].tolist() == b["det"]["idx"].tolist()


def test_multiscale_attention_of_identical_agents_is_one_agent():
    # identical agents have equal scores: uniform weights return the map
    cfg = _small_neck_cfg("attn", n_agents=3)
    w = synth.weights_for(cfg)
    p = synth.points_for(cfg, 0, 0)
    one = of.forward_multiscale([p], w, dataclasses_replace(cfg, n_agents=1))
    three = of.forward_multiscale([p, p, p], w, cfg)
    np.testing.assert_allclose(three["head"], one["head"], rtol=1e-12, atol=1e-12)


def test_multiscale_max_is_agent_order_invariant_and_differs_from_late_fusion():
    cfg = _small_neck_cfg("max", n_agents=3)
    w = synth.weights_for(cfg)
    pts = [synth.points_for(cfg, 0, k) for k in range(3)]
    a = of.forward_multiscale(pts, w, cfg, store="fp16")
    b = of.forward_multiscale(pts[::-1], w, cfg, store="fp16")
    np.testing.assert_array_equal(a["head"], b["head"])
    for bi, fb in enumerate(a["fused_blocks"]):             # each scale: max of the agents'
        np.testing.assert_array_equal(fb, np.maximum.reduce([e["blocks"][bi] for e in a["enc"]]))
    # the deconvs do not commute with the max: the placement changes the result
    late = of.forward(pts, w, cfg, store="fp16")
    assert not np.allclose(late["head"], a["head"])


def dataclasses_replace(cfg, **kw):
    import dataclasses
    return dataclasses.replace(cfg, **kw)


def test_multiscale_attention_is_a_convex_mix_per_scale():
    # attention weights are a softmax: each fused cell lies between the
    # agents' values, and (unlike max fusion) strictly inside somewhere
    cfg = _small_neck_cfg("attn", n_agents=2)
    w = synth.weights_for(cfg)
    pts = [synth.points_for(cfg, 0, k) for k in range(2)]
    r = of.forward_multiscale(pts, w, cfg)
    for bi, fb in enumerate(r["fused_blocks"]):
        xs = np.stack([e["blocks"][bi] for e in r["enc"]])
        assert (fb >= xs.min(0) - 1e-12).all() and (fb <= xs.max(0) + 1e-12).all()
        assert (fb < xs.max(0) - 1e-9).any()


def test_decode_regression_hand_worked():
    # Two anchors with every regression term non-zero and distinct, so that
    # each term is forced to its own channel and scale.  Expected values were
    # worked out by hand from the anchor definition (tiny grid: 64 x 64 cells
    # of 0.4 m from -12.8 m; car anchor l, w, h = 3.9, 1.6, 1.56 at z = -1,
    # yaw a * pi / 2; d_a = sqrt(3.9^2 + 1.6^2) = sqrt(17.77) = 4.2154478).
    #   anchor 0, cell (ix 10, iy 20): centre (-8.6, -4.6)
    #     reg (0.5, -0.25, 0.2, 0.1, -0.2, 0.3, 0.1)
    #     x = -8.6 + 0.5 d_a = -6.4922761    y = -4.6 - 0.25 d_a = -5.6538619
    #     z = -1 + 0.2 * 1.56 = -0.688        l = 3.9 e^0.1 = 4.3101666
    #     w = 1.6 e^-0.2 = 1.3099692          h = 1.56 e^0.3 = 2.1057797
    #     yaw = 0 + 0.1
    #   anchor 1, cell (ix 3, iy 5): centre (-11.4, -10.6)
    #     reg (-0.1, 0.4, -0.5, -0.3, 0.25, -0.1, -0.2)
    #     x = -11.4 - 0.1 d_a = -11.8215448   y = -10.6 + 0.4 d_a = -8.9138209
    #     z = -1 - 0.5 * 1.56 = -1.78         l = 3.9 e^-0.3 = 2.8891911
    #     w = 1.6 e^0.25 = 2.0544407          h = 1.56 e^-0.1 = 1.4115464
    #     yaw = pi / 2 - 0.2 = 1.3707963
    # A wrong diagonal (d_a = l_a), dz scaled by d_a, or a channel read one
    # term off each move at least one of these numbers by more than 1e-3.
    cfg = synth.get_config("tiny")
    A, Hf, Wf = cfg.anchors, cfg.feat_h, cfg.feat_w
    hd = np.zeros((8 * A, Hf, Wf))
    hd[:A] = -5.0
    hd[0, 20, 10] = 2.0
    hd[1, 5, 3] = 1.0
    hd[A + 0:A + 7, 20, 10] = (0.5, -0.25, 0.2, 0.1, -0.2, 0.3, 0.1)
    hd[A + 7:A + 14, 5, 3] = (-0.1, 0.4, -0.5, -0.3, 0.25, -0.1, -0.2)
    # decoy regression on the other anchor of each cell (must not be read)
    hd[A + 7:A + 14, 20, 10] = 9.0
    hd[A + 0:A + 7, 5, 3] = -9.0
    det = of.decode(hd, cfg, cls_thresh=0.0, max_boxes=10)
    assert det["idx"].tolist() == [(20 * Wf + 10) * A + 0, (5 * Wf + 3) * A + 1]
    want = np.array([
        [-6.4922761, -5.6538619, -0.688, 4.3101666, 1.3099692, 2.1057797, 0.1,
         1.0 / (1.0 + math.exp(-2.0))],
        [-11.8215448, -8.9138209, -1.78, 2.8891911, 2.0544407, 1.4115464, 1.3707963,
         1.0 / (1.0 + math.exp(-1.0))]])
    np.testing.assert_allclose(det["boxes"], want, rtol=0, atol=2e-7)

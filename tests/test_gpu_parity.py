"""GPU path vs the CPU oracle, through the C ABI.

Bar: pillar indices, counts and drop counters bit-exact; every floating-point
tensor within |gpu - oracle| <= 2e-2 + 1e-2 |oracle| (fp16/bf16 storage, fp32
accumulation) against the oracle in storage-rounded mode; the decode's
selection and order exact given the GPU head; RTCC and Barrier outputs
bit-identical (Sec. III-C last paragraph, Sec. V-F).

Stages are also checked in isolation (the oracle's next stage applied to the
GPU's own input of that stage) so that a kernel is judged on its own error.
"""
import dataclasses
import time

import numpy as np
import pytest

import synth
from oracle import forward as of
from tests import gpu_util as U

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def R():
    return U.load()


def _small_pp(name="pp3", grid=(96, 64), n_uniform=6000, clusters=4, **kw):
    base = synth.get_config(name)
    return dataclasses.replace(base, grid_w=grid[0], grid_h=grid[1],
                               x_min=-grid[0] * 0.2, x_max=grid[0] * 0.2,
                               y_min=-grid[1] * 0.2, y_max=grid[1] * 0.2,
                               pts_x=(-grid[0] * 0.2 - 1, grid[0] * 0.2 + 1),
                               pts_y=(-grid[1] * 0.2 - 1, grid[1] * 0.2 + 1),
                               n_uniform=n_uniform, n_clusters=clusters, **kw)


def _check_frame(R, ctx, cfg, w, pts, absent=()):
    """Compare every stage of the frame just run against the oracle."""
    store = cfg.dtype
    K = cfg.n_agents
    feats_gpu = []
    for k in range(K):
        if k in absent:
            feats_gpu.append(None)
            continue
        # pillars: bit-exact
        op = of.pillarise(pts[k], cfg)
        gp = R.rtcc_get_pillars(ctx, k, cfg.grid_h, cfg.grid_w, cfg.max_pillars)
        assert gp["n_pillars"] == op["n_pillars"]
        np.testing.assert_array_equal(gp["cell2pillar"], op["cell2pillar"])
        n = op["n_pillars"]
        np.testing.assert_array_equal(gp["pillar_cell"][:n], op["pillar_cell"][:n])
        np.testing.assert_array_equal(gp["count"][:n], op["count"][:n])
        assert gp["drop_range"] == op["drop_range"]
        assert gp["drop_pcap"] == op["drop_pcap"]
        assert gp["drop_ncap"] == op["drop_ncap"]
        # PFN + scatter
        h = of.pfn(op, w["pfn.w"], w["pfn.b"], cfg, store)
        img_o = of.scatter(h, op, cfg)
        img_g = U.gpu_tensor(ctx, cfg, k, 0, (cfg.pfn_ch, cfg.grid_h, cfg.grid_w))
        occ_g = (img_g != 0).any(axis=0).reshape(-1)
        assert not (occ_g & (op["cell2pillar"] < 0)).any()        # nonzero only on pillars
        U.assert_close(img_g, img_o, f"pseudo-image agent {k}")
        # every conv layer, isolated on the GPU's own input of that layer
        x_g = img_g
        layers = U.conv_layers(cfg)
        last_of_block = {}
        for i, (bi, li, st, shape) in enumerate(layers):
            y_o = U.oracle_conv_layer(x_g, w, bi, li, st, store)
            y_g = U.gpu_tensor(ctx, cfg, k, 16 + i, shape)
            U.assert_close(y_g, y_o, f"conv b{bi}.c{li} agent {k}")
            x_g = y_g
            last_of_block[bi] = y_g
        blocks_g = [last_of_block[bi] for bi in range(len(cfg.blocks))]
        shapes = U.block_shapes(cfg)
        for bi in range(len(cfg.blocks)):                       # block read-back = last layer
            np.testing.assert_array_equal(U.gpu_tensor(ctx, cfg, k, bi + 1, shapes[bi]), blocks_g[bi])
        # neck, isolated on the GPU's own block outputs
        feat_o = U.oracle_neck(blocks_g, w, cfg, store)
        feat_g = U.gpu_tensor(ctx, cfg, k, 8, (cfg.feat_ch, cfg.feat_h, cfg.feat_w))
        U.assert_close(feat_g, feat_o, f"features agent {k}")
        feats_gpu.append(feat_g)
    # fusion + head, isolated on the GPU's own feature slots
    F_o = of.fuse_max(feats_gpu) if cfg.fusion == "max" else of.fuse_attn(feats_gpu)
    F_g = U.gpu_tensor(ctx, cfg, 0, 9, (cfg.feat_ch, cfg.feat_h, cfg.feat_w))
    if cfg.fusion == "max":
        np.testing.assert_array_equal(F_g, F_o)                 # max is exact
    else:
        U.assert_close(F_g, F_o, "fused (attention)")
    hd_o = of.head(F_o, of.store_round(w["head.w"], store), of.store_round(w["head.b"], store))
    hd_g = U.head_to_oracle_layout(R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w))
    U.assert_close(hd_g, hd_o, "head (isolated)")
    return hd_g


_BOX_FIELDS = ("x", "y", "z", "l", "w", "h", "yaw", "score")


def _check_decode(cfg, hd_g, boxes, R=None, ctx=None):
    """The decode's selection and order exact given the GPU head, its boxes
    within tolerance; with NMS, the decoded list comes from the read-back and
    the result must be its NMS (see gpu_util.check_nms)."""
    det = of.decode(hd_g, cfg)
    nms_on = getattr(cfg, "nms_iou", 0.0) > 0
    dec = R.rtcc_get_decoded(ctx) if nms_on else boxes
    assert dec["anchor"].tolist() == det["idx"].tolist()        # exact selection + order
    got = np.stack([dec[f] for f in _BOX_FIELDS], axis=1)
    U.assert_close(got, det["boxes"], "boxes")
    if nms_on:
        U.check_nms(dec, boxes, cfg.nms_iou)
        assert 0 < len(boxes) <= len(dec) or len(dec) == 0


def _end_to_end(R, cfg, frame=0, absent=(), flags=None, arrivals=None):
    ctx, w = U.make_ctx(cfg) if flags is None else U.make_ctx(cfg, flags=flags)
    try:
        pts = [synth.points_for(cfg, frame, k) for k in range(cfg.n_agents)]
        a = synth.arrivals_for(cfg, frame) if arrivals is None else arrivals
        boxes = U.run_frame(ctx, cfg, pts, a, R.MODE_RTCC, absent=absent)
        hd_g = _check_frame(R, ctx, cfg, w, pts, absent=absent)
        _check_decode(cfg, hd_g, boxes, R, ctx)
        # whole-path parity: the oracle forward from the points
        full = of.forward([None if k in absent else pts[k] for k in range(cfg.n_agents)], w, cfg,
                          store=cfg.dtype)
        U.assert_close(hd_g, full["head"], "head (end to end)")
        return ctx, w, pts, a
    except Exception:
        R.rtcc_destroy(ctx)
        raise


def test_tiny_end_to_end(R):
    cfg = synth.get_config("tiny")
    ctx, *_ = _end_to_end(R, cfg)
    info = R.rtcc_get_frame_info(ctx)
    assert info.n_dispatched == 2 and info.gpu_backbone_ms[0] > 0 and info.gpu_fusion_ms > 0
    # the fusion kernel's own global-timer span sits inside its event-node span
    assert 0 < info.gpu_fusion_kernel_ms <= info.gpu_fusion_ms + 1e-3
    # completions reported back to back share a backbone launch (or, if the
    # host was slow, agent 0 ran alone and agent 1 as its own branch graph)
    assert all(info.gpu_pfn_kernel_ms[k] > 0 for k in range(2))
    assert all(info.gpu_pfn_kernel_ms[k] < info.gpu_branch_ms[k] for k in range(2)
               if info.gpu_branch_ms[k] > 0)
    assert sum(info.backbone_batch[j] for j in range(info.n_backbone_launches)) == 2
    R.rtcc_destroy(ctx)


def test_release_hold_gathers_a_burst_and_lets_a_lone_branch_go(R):
    # A release that does not resolve the last branch leaves its backbone
    # batch open for a short hold.  Completions reported back to back then
    # share one backbone launch; a branch released alone gets its own launch
    # once the hold runs out, and the last branch, released onto a free GPU,
    # runs as its own branch graph (pillar chain and backbone in one graph).
    # The outputs are the same bytes either way (Sec. III-C: the schedule
    # changes when work runs, not what it computes).
    cfg = synth.get_config("tiny")
    ctx, _ = U.make_ctx(cfg)
    try:
        pts = [synth.points_for(cfg, 0, k) for k in range(cfg.n_agents)]
        U.run_frame(ctx, cfg, pts, [0.0, 0.0], R.MODE_BARRIER, frame_id=1)
        ref = R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w).tobytes()
        info = R.rtcc_get_frame_info(ctx)
        assert list(info.backbone_batch)[:info.n_backbone_launches] == [2]
        # back to back (resident payloads, so the calls are short): the second
        # completion joins the first one's launch when it comes within the
        # hold.  A slow host can miss the hold, so the library's release stamps
        # decide what to expect: a second release less than 30 us after the
        # first was inside the hold and must have shared the launch
        for k in range(cfg.n_agents):
            assert R.rtcc_stage_resident(ctx, k, pts[k]) == R.OK
        burst = []
        for f in range(5):
            assert R.rtcc_set_mode(ctx, R.MODE_RTCC) == R.OK
            assert R.rtcc_frame_begin(ctx, 2 + f, 0.0) == R.OK
            for k in range(cfg.n_agents):
                assert R.rtcc_payload_resident(ctx, k, 0.0) == R.OK
            s, _, _ = R.rtcc_wait_detection(ctx, 60000)
            assert s == R.OK, R.rtcc_status_str(s)
            assert R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w).tobytes() == ref
            info = R.rtcc_get_frame_info(ctx)
            sizes = list(info.backbone_batch)[:info.n_backbone_launches]
            gap_us = (info.t_release_ms[1] - info.t_release_ms[0]) * 1e3
            burst.append((sizes, round(gap_us, 1)))
            assert sizes in ([2], [1, 1]), burst
            if gap_us < 30.0:
                assert sizes == [2], burst
        # 20 ms apart: agent 0's backbone runs alone after the hold and has
        # ended when agent 1 arrives
        assert R.rtcc_frame_begin(ctx, 9, 0.0) == R.OK
        assert R.rtcc_payload_complete(ctx, 0, pts[0], 0.0) == R.OK
        time.sleep(0.02)
        assert R.rtcc_payload_complete(ctx, 1, pts[1], 20.0) == R.OK
        s, _, _ = R.rtcc_wait_detection(ctx, 60000)
        assert s == R.OK, R.rtcc_status_str(s)
        assert R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w).tobytes() == ref
        info = R.rtcc_get_frame_info(ctx)
        assert list(info.backbone_batch)[:info.n_backbone_launches] == [1, 1]
        assert list(info.dispatch_order)[:2] == [0, 1]
        assert info.gpu_branch_ms[0] < 0 < info.gpu_branch_ms[1]
        assert info.gpu_backbone_ms[0] > 0 and info.gpu_backbone_ms[1] > 0
    finally:
        R.rtcc_destroy(ctx)


def test_pointpillars_small_grid_ragged_tiles(R):
    # 96x64 grid: block maps 48x32, 24x16, 12x8 -- none a multiple of the
    # 32x4 tile in x except the first; deconvs s = 1, 2, 4 into 384 channels
    cfg = _small_pp()
    ctx, *_ = _end_to_end(R, cfg)
    R.rtcc_destroy(ctx)


def test_attention_bf16_with_absent_agent(R):
    cfg = _small_pp("lr5", grid=(88, 40), n_uniform=5000)
    ctx, *_ = _end_to_end(R, cfg, absent=(3,))
    R.rtcc_destroy(ctx)


def test_caps_bind_bit_exact(R):
    cfg = dataclasses.replace(synth.get_config("tiny"), max_pillars=16, max_pts=8)
    ctx, w = U.make_ctx(cfg, max_points=4096)
    pts = [synth.points_cap_patch(2048, 8, seed=3), synth.points_cap_patch(4096, 6, seed=4)]
    U.run_frame(ctx, cfg, pts, [0.0, 1.0], R.MODE_RTCC)
    hd = _check_frame(R, ctx, cfg, w, pts)
    full = of.forward(pts, w, cfg, store="fp16")
    U.assert_close(hd, full["head"], "head (caps)")
    gp = R.rtcc_get_pillars(ctx, 1, cfg.grid_h, cfg.grid_w, cfg.max_pillars)
    assert gp["drop_pcap"] > 0 and gp["drop_ncap"] > 0
    R.rtcc_destroy(ctx)


def test_large_payload_scan_takes_several_tiles_per_block(R):
    # 1.6 million points per branch: the pillar scan runs 4,096-point tiles,
    # more tiles than the cooperative grid has blocks, so each block takes
    # several in order; pillars, drops and every later stage as in any frame
    cfg = dataclasses.replace(synth.get_config("tiny"), max_pillars=2048, max_pts=16)
    rng = np.random.default_rng(5)
    pts = []
    for n in (1_600_000, 700_001):
        p = np.zeros((n, 4), dtype=np.float32)
        p[:, 0] = rng.uniform(-14.0, 14.0, n)
        p[:, 1] = rng.uniform(-14.0, 14.0, n)
        p[:, 2] = rng.uniform(-3.2, 1.2, n)
        p[:, 3] = rng.uniform(0.0, 1.0, n)
        pts.append(p)
    ctx, w = U.make_ctx(cfg, max_points=1_600_000)
    try:
        for fid, mode in ((1, R.MODE_RTCC), (2, R.MODE_BARRIER)):
            U.run_frame(ctx, cfg, pts, [0.0, 1.0], mode, frame_id=fid)
            _check_frame(R, ctx, cfg, w, pts)
    finally:
        R.rtcc_destroy(ctx)


def test_empty_and_out_of_range_payloads(R):
    cfg = synth.get_config("tiny")
    ctx, w = U.make_ctx(cfg)
    far = synth.points_for(cfg, 0, 1).copy()
    far[:, 0] += 100.0                                  # every point out of range
    pts = [np.zeros((0, 4), dtype=np.float32), far]
    U.run_frame(ctx, cfg, pts, [0.0, 0.0], R.MODE_RTCC)
    for k in range(2):
        gp = R.rtcc_get_pillars(ctx, k, cfg.grid_h, cfg.grid_w, cfg.max_pillars)
        assert gp["n_pillars"] == 0 and (gp["cell2pillar"] == -1).all()
    hd = _check_frame(R, ctx, cfg, w, pts)
    full = of.forward(pts, w, cfg, store="fp16")
    U.assert_close(hd, full["head"], "head (empty)")
    R.rtcc_destroy(ctx)


@pytest.mark.parametrize("grid", [(96, 64), (256, 256)])
def test_decode_all_equal_logits(R, grid):
    # Zero head weights: every logit of anchor a equals its bias, so the keys
    # of an anchor are one value repeated over all cells.  The selection is
    # then decided by anchor index alone (ties), and at 256x256 the threshold
    # bin holds 16384 keys, more than the decode's shared-memory list takes
    # (its radix-select fallback); at 96x64 it holds 1536 (the list path).
    cfg = dataclasses.replace(_small_pp(grid=grid), cls_thresh=-1.0, nms_iou=0.0)
    w = dict(synth.weights_for(cfg))
    w["head.w"] = np.zeros_like(w["head.w"])
    ctx = R.rtcc_init(R.model_config(cfg, flags=U.DEBUG_FLAGS), synth.weight_blob(w))
    try:
        pts = [synth.points_for(cfg, 0, k) for k in range(cfg.n_agents)]
        boxes = U.run_frame(ctx, cfg, pts, [0.0] * cfg.n_agents, R.MODE_RTCC)
        hd = U.head_to_oracle_layout(R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w))
        assert len(boxes) == cfg.max_boxes
        _check_decode(cfg, hd, boxes, R, ctx)
    finally:
        R.rtcc_destroy(ctx)


def _decode_path_sizes(hd, cls_thresh, max_boxes):
    """The decode's list sizes for a head output, recomputed on the host: the
    count below0 of keys in level-0 bins below the bin b0 that holds the K-th
    key, that bin's size nb0, and the size nb1 of the level-1 bin (next 10 key
    bits) that holds it.  Keys order the class logits descending as 32-bit
    unsigned integers (the fusion kernel's encoding)."""
    A = 2
    logit = (hd[:A].transpose(1, 2, 0).reshape(-1).astype(np.float32) + np.float32(0.0))
    u = logit.view(np.uint32)
    asc = np.where(u & np.uint32(0x80000000), ~u, u | np.uint32(0x80000000))
    key = (~asc)[logit >= np.float32(cls_thresh)]
    need = min(max_boxes, key.size)
    cum = np.cumsum(np.bincount(key >> 20, minlength=4096))
    b0 = int(np.searchsorted(cum, need))
    below0 = int(cum[b0 - 1]) if b0 > 0 else 0
    inb = key[(key >> 20) == b0]
    cum1 = np.cumsum(np.bincount((inb >> 10) & 1023, minlength=1024))
    b1 = int(np.searchsorted(cum1, need - below0))
    return below0, inb.size, int(cum1[b1] - (cum1[b1 - 1] if b1 > 0 else 0))


def test_decode_level1_list_path(R):
    # Class logits crowded into one level-0 key bin (logits about 1.03 +- 0.02)
    # but spread over its next 10 bits: more candidates than the decode's
    # threads, so it takes the level-1 histogram and warp-sort path instead of
    # ranking by counting (which the other workloads take).
    cfg = dataclasses.replace(_small_pp(grid=(96, 64)), cls_thresh=-1.0, max_boxes=500, nms_iou=0.0)
    w = dict(synth.weights_for(cfg))
    pts = [synth.points_for(cfg, 0, k) for k in range(cfg.n_agents)]
    F = of.forward(pts, w, cfg, store=cfg.dtype)["fused"]
    z = np.tensordot(of.store_round(w["head.w"], cfg.dtype)[:2], F, axes=(1, 0))
    hw = w["head.w"].copy()
    hw[:2] *= np.float32(0.02 / max(float(z.std()), 1e-6))
    hb = w["head.b"].copy()
    hb[:2] = 1.03
    w["head.w"], w["head.b"] = hw, hb
    ctx = R.rtcc_init(R.model_config(cfg, flags=U.DEBUG_FLAGS), synth.weight_blob(w))
    try:
        boxes = U.run_frame(ctx, cfg, pts, [0.0] * cfg.n_agents, R.MODE_RTCC)
        hd = U.head_to_oracle_layout(R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w))
        below0, nb0, nb1 = _decode_path_sizes(hd, cfg.cls_thresh, cfg.max_boxes)
        assert below0 + nb0 > 1024 and nb0 <= 4096 and nb1 <= 64, (below0, nb0, nb1)
        assert len(boxes) == cfg.max_boxes
        _check_decode(cfg, hd, boxes, R, ctx)
    finally:
        R.rtcc_destroy(ctx)


def test_split_k_without_clusters_bit_identical(R):
    # The deepest block's 4-way split-K reduces through distributed shared
    # memory when the backbone runs in clusters of four CTAs, and through
    # global memory without clusters; both sum the slices in slice order, so
    # the outputs must match bit for bit (and the oracle within tolerance).
    cfg = _small_pp()
    pts = [synth.points_for(cfg, 0, k) for k in range(cfg.n_agents)]
    heads = []
    for flags in (U.DEBUG_FLAGS, U.DEBUG_FLAGS | R.FLAG_NO_CLUSTERS):
        ctx, w = U.make_ctx(cfg, flags=flags)
        try:
            U.run_frame(ctx, cfg, pts, [0.0, 1.0, 2.0], R.MODE_RTCC)
            heads.append(R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w).copy())
            if flags & R.FLAG_NO_CLUSTERS:
                hd = _check_frame(R, ctx, cfg, w, pts)
                full = of.forward(pts, w, cfg, store=cfg.dtype)
                U.assert_close(hd, full["head"], "head (no clusters)")
        finally:
            R.rtcc_destroy(ctx)
    assert heads[0].tobytes() == heads[1].tobytes()


@pytest.mark.parametrize("name", ["tiny", "small_pp", "small_attn"])
def test_rtcc_and_barrier_bit_identical(R, name):
    if name == "tiny":
        cfg = synth.get_config("tiny")
    elif name == "small_pp":
        cfg = _small_pp()
    else:
        cfg = _small_pp("lr5", grid=(88, 40), n_uniform=5000)
    ctx, w = U.make_ctx(cfg)
    outs = {}
    for frame in range(2):
        pts = [synth.points_for(cfg, frame, k) for k in range(cfg.n_agents)]
        a = synth.arrivals_for(cfg, frame) if cfg.arrival != "fixed" else [0.0, 5.0]
        for mode in (R.MODE_RTCC, R.MODE_BARRIER, R.MODE_RTCC):
            boxes = U.run_frame(ctx, cfg, pts, a, mode, frame_id=frame)
            hd = R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w)
            feats = b"".join(R.rtcc_get_tensor(ctx, k, 8).tobytes() for k in range(cfg.n_agents))
            key = (frame, mode)
            cur = (hd.tobytes(), boxes.tobytes(), feats)
            if key in outs:
                assert outs[key] == cur                       # run-to-run deterministic
            outs[key] = cur
        assert outs[(frame, R.MODE_RTCC)] == outs[(frame, R.MODE_BARRIER)]
    R.rtcc_destroy(ctx)


def test_resident_input_release_matches_staged(R):
    cfg = synth.get_config("tiny")
    ctx, w = U.make_ctx(cfg)
    pts = [synth.points_for(cfg, 3, k) for k in range(2)]
    b1 = U.run_frame(ctx, cfg, pts, [1.0, 2.0], R.MODE_RTCC)
    h1 = R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w).tobytes()
    for k in range(2):
        assert R.rtcc_stage_resident(ctx, k, pts[k]) == R.OK
    assert R.rtcc_frame_begin(ctx, 9, 0.0) == R.OK
    assert R.rtcc_payload_resident(ctx, 1, 1.0) == R.OK
    assert R.rtcc_payload_resident(ctx, 0, 2.0) == R.OK
    s, b2, _ = R.rtcc_wait_detection(ctx, 60000)
    assert s == R.OK
    assert R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w).tobytes() == h1
    assert b1.tobytes() == b2.tobytes()
    R.rtcc_destroy(ctx)


def test_abort_is_infeasible_and_next_frame_clean(R):
    cfg = synth.get_config("tiny")
    ctx, w = U.make_ctx(cfg)
    pts = [synth.points_for(cfg, 0, k) for k in range(2)]
    assert R.rtcc_frame_begin(ctx, 1, 0.0) == R.OK
    assert R.rtcc_payload_complete(ctx, 0, pts[0], 1.0) == R.OK
    assert R.rtcc_wait_detection(ctx, 100)[0] == R.E_STATE        # branch 1 still missing
    assert R.rtcc_frame_abort(ctx) == R.OK
    assert R.rtcc_wait_detection(ctx, 100)[0] == R.E_INFEASIBLE
    boxes = U.run_frame(ctx, cfg, pts, [0.0, 5.0], R.MODE_RTCC, frame_id=2)
    hd = _check_frame(R, ctx, cfg, w, pts)
    _check_decode(cfg, hd, boxes, R, ctx)
    R.rtcc_destroy(ctx)


def test_pointpillars_full_size(R):
    cfg = synth.get_config("pp3")
    ctx, *_ = _end_to_end(R, cfg, frame=1)
    R.rtcc_destroy(ctx)


def test_layer_spans_follow_dependencies(R):
    # With layer stamps on, the backbone records when each layer's first item
    # passed its wait and when its last item was counted.  Every conv reads
    # the conv before it and the neck deconv of block b reads that block's
    # last conv, so no layer may start before the layers it reads have ended
    # (up to the global timer's resolution).  The stamps must not change the
    # results.
    cfg = synth.get_config("pp3")
    pts = [synth.points_for(cfg, 2, k) for k in range(cfg.n_agents)]
    heads, spans = [], None
    for flags in (U.DEBUG_FLAGS, U.DEBUG_FLAGS | R.FLAG_LAYER_TIMES):
        ctx, _ = U.make_ctx(cfg, flags=flags)
        try:
            U.run_frame(ctx, cfg, pts, [0.0, 1.0, 2.0], R.MODE_RTCC)
            heads.append(R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w).copy())
            if flags & R.FLAG_LAYER_TIMES:
                spans = [R.rtcc_get_layer_spans(ctx, k) for k in range(cfg.n_agents)]
                dur = R.rtcc_get_layer_times(ctx, 0)
        finally:
            R.rtcc_destroy(ctx)
    assert heads[0].tobytes() == heads[1].tobytes()
    last_of_block, n_conv = [], 0
    for n, _, _ in cfg.blocks:
        n_conv += n
        last_of_block.append(n_conv - 1)
    deps = [[l - 1] if 0 < l < n_conv else [] for l in range(n_conv)]
    deps += [[last_of_block[b]] for b in range(len(cfg.up_strides))]
    tol = 2e-3                                  # ms
    for start, end in spans:
        assert len(start) == len(deps)
        assert np.all(start >= 0) and np.all(end >= start)
        assert np.min(start) == 0.0
        for l, dl in enumerate(deps):
            for d in dl:
                assert start[l] >= end[d] - tol, (l, d, start[l], end[d])
    np.testing.assert_allclose(dur, spans[0][1] - spans[0][0], rtol=0, atol=1e-6)


def test_long_range_attention_bf16_full_size(R):
    # 5 agents, 704x200 grid, 120k points each, per-cell attention fusion with
    # the ego agent as query, bf16 storage; one agent masked out
    cfg = synth.get_config("lr5")
    ctx, *_ = _end_to_end(R, cfg, frame=1, absent=(2,))
    R.rtcc_destroy(ctx)


def test_eight_agent_stress_full_size(R):
    # 8 agents, 704x200 grid, 150k points each, max fusion; all eight payloads
    # complete at once (branches contend for the GPU)
    cfg = synth.get_config("stress8")
    ctx, *_ = _end_to_end(R, cfg, frame=1, arrivals=[0.0] * cfg.n_agents)
    R.rtcc_destroy(ctx)


def _production_frame(R, ctx, cfg, pts, a, mode, absent=()):
    boxes = U.run_frame(ctx, cfg, pts, a, mode, absent=absent)
    hd = R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w).copy()
    feats = b"".join(b"" if k in absent else R.rtcc_get_tensor(ctx, k, 8).tobytes()
                     for k in range(cfg.n_agents))
    dec = R.rtcc_get_decoded(ctx)
    return hd, boxes, feats, dec


@pytest.mark.parametrize("name,absent,spread", [("pp3", (), None), ("lr5", (2,), None),
                                                ("stress8", (), "zero"),
                                                ("stress8", (), "lognormal")])
def test_production_context_full_size(R, name, absent, spread):
    # The context the bench times: flags = 0, i.e. two ping-pong activation
    # buffers per block (layer l + 1 overwrites what layer l - 1 wrote), the
    # neck deconvs reading a block's last buffer while the next block runs,
    # split-K through distributed shared memory, no per-layer buffers, no
    # event nodes.  Checked end to end against the oracle (pillars bit-exact,
    # pseudo-image, head, decode selection, NMS decisions), then the same
    # frame in Barrier mode and again in RTCC mode must give byte-identical
    # head, boxes and feature slots (Sec. III-C; Sec. V-F), and the debug
    # context (per-layer buffers, checked layer by layer elsewhere) must give
    # the same head byte for byte.
    cfg = synth.get_config(name)
    frame = 1
    pts = [synth.points_for(cfg, frame, k) for k in range(cfg.n_agents)]
    a = synth.arrivals_for(cfg, frame, spread)
    ctx, w = U.make_ctx(cfg, flags=0)
    try:
        hd, boxes, feats, dec = _production_frame(R, ctx, cfg, pts, a, R.MODE_RTCC, absent)
        for k in range(cfg.n_agents):
            if k in absent:
                continue
            op = of.pillarise(pts[k], cfg)
            gp = R.rtcc_get_pillars(ctx, k, cfg.grid_h, cfg.grid_w, cfg.max_pillars)
            n = op["n_pillars"]
            assert gp["n_pillars"] == n
            np.testing.assert_array_equal(gp["cell2pillar"], op["cell2pillar"])
            np.testing.assert_array_equal(gp["pillar_cell"][:n], op["pillar_cell"][:n])
            np.testing.assert_array_equal(gp["count"][:n], op["count"][:n])
            img_g = U.gpu_tensor(ctx, cfg, k, 0, (cfg.pfn_ch, cfg.grid_h, cfg.grid_w))
            img_o = of.scatter(of.pfn(op, w["pfn.w"], w["pfn.b"], cfg, cfg.dtype), op, cfg)
            U.assert_close(img_g, img_o, f"pseudo-image agent {k}")
        hd_o = U.head_to_oracle_layout(hd)
        full = of.forward([None if k in absent else pts[k] for k in range(cfg.n_agents)], w, cfg,
                          store=cfg.dtype)
        U.assert_close(hd_o, full["head"], "head (end to end, production context)")
        _check_decode(cfg, hd_o, boxes, R, ctx)
        ref = (hd.tobytes(), boxes.tobytes(), feats, dec.tobytes())
        for mode in (R.MODE_BARRIER, R.MODE_RTCC):
            h2, b2, f2, d2 = _production_frame(R, ctx, cfg, pts, a, mode, absent)
            assert (h2.tobytes(), b2.tobytes(), f2, d2.tobytes()) == ref, f"mode {mode} differs"
            info = R.rtcc_get_frame_info(ctx)
            n_present = cfg.n_agents - len(absent)
            sizes = list(info.backbone_batch)[:info.n_backbone_launches]
            assert sum(sizes) == n_present
            if mode == R.MODE_BARRIER:                 # all released at A: one launch
                assert sizes == [n_present], sizes
    finally:
        R.rtcc_destroy(ctx)
    # the debug context runs every branch in its own backbone launch
    dctx, _ = U.make_ctx(cfg, flags=U.DEBUG_FLAGS | R.FLAG_NO_BATCH)
    try:
        U.run_frame(dctx, cfg, pts, a, R.MODE_BARRIER, absent=absent)
        info = R.rtcc_get_frame_info(dctx)
        assert info.n_backbone_launches == cfg.n_agents - len(absent)
        assert R.rtcc_get_head(dctx, cfg.feat_h, cfg.feat_w).tobytes() == ref[0]
    finally:
        R.rtcc_destroy(dctx)


def test_bounded_wait_runs_out_and_next_frame_is_clean(R):
    # A backbone launch made to wait for a work item that never comes: the
    # wait gives up after the short limit, the kernel sets its error word and
    # winds down (no trap, no hang), rtcc_wait_detection reports
    # RTCC_E_DEVICE, and the next frame runs clean with the same outputs as
    # before and passes parity (Sec. IV-C: a frame that cannot complete is
    # reported, not waited on forever).
    cfg = synth.get_config("tiny")
    ctx, w = U.make_ctx(cfg, flags=U.DEBUG_FLAGS | R.FLAG_SHORT_WAITS)
    plain, _ = U.make_ctx(cfg, flags=0)
    try:
        assert R.rtcc_test_unreachable_wait(plain) == R.E_STATE
        pts = [synth.points_for(cfg, 0, k) for k in range(cfg.n_agents)]
        b0 = U.run_frame(ctx, cfg, pts, [0.0, 5.0], R.MODE_RTCC, frame_id=1)
        h0 = R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w).tobytes()
        assert R.rtcc_test_unreachable_wait(ctx) == R.OK
        assert R.rtcc_frame_begin(ctx, 2, 0.0) == R.OK
        for k, t in ((0, 0.0), (1, 5.0)):
            assert R.rtcc_payload_complete(ctx, k, pts[k], t) == R.OK
        s, _, _ = R.rtcc_wait_detection(ctx, 60000)
        assert s == R.E_DEVICE, R.rtcc_status_str(s)
        for mode in (R.MODE_RTCC, R.MODE_BARRIER):
            b1 = U.run_frame(ctx, cfg, pts, [0.0, 5.0], mode, frame_id=3 + mode)
            assert b1.tobytes() == b0.tobytes()
            assert R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w).tobytes() == h0
        hd = _check_frame(R, ctx, cfg, w, pts)
        _check_decode(cfg, hd, b1, R, ctx)
    finally:
        R.rtcc_destroy(ctx)
        R.rtcc_destroy(plain)


@pytest.mark.parametrize("name", ["tiny", "pp3"])
def test_copy_engine_release_matches_zero_copy(R, name):
    # Host payloads through a copy-engine transfer and a cross-stream event
    # (the release path as Sec. IV-F writes it) give the same bytes as the
    # default path, whose first kernel reads the pinned staging buffer.
    cfg = synth.get_config(name)
    pts = [synth.points_for(cfg, 2, k) for k in range(cfg.n_agents)]
    a = synth.arrivals_for(cfg, 2) if cfg.arrival != "fixed" else [0.0, 5.0]
    outs = []
    for flags in (0, R.FLAG_H2D_COPY):
        ctx, _ = U.make_ctx(cfg, flags=flags)
        try:
            for mode in (R.MODE_RTCC, R.MODE_BARRIER):
                boxes = U.run_frame(ctx, cfg, pts, a, mode)
                outs.append((R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w).tobytes(), boxes.tobytes()))
        finally:
            R.rtcc_destroy(ctx)
    assert all(o == outs[0] for o in outs)

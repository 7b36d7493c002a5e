"""The paper's multi-scale fusion placement on the GPU (RTCC_FLAG_MULTISCALE;
Sec. IV-A's shared subgraph of fusion, upsampling and concatenation; the
agent-indexed slots of Sec. IV-D) against oracle.forward.forward_multiscale:
each branch ends at its backbone blocks; after the join every block's map is
fused across the present agents, the deconv neck runs once on the fused maps,
then the head, decode and rotated NMS.

Each stage is also checked on the GPU's own input of that stage: max fusion
bit-exact, attention within the tolerance, the neck and the head within the
tolerance; RTCC and Barrier byte-identical (Sec. III-C, Sec. V-F); and the
branches' block outputs byte-identical to those of the single-scale context
(the branch computation up to the blocks is the same)."""
import numpy as np
import pytest

import synth
from oracle import forward as of
from tests import gpu_util as U
from tests.test_gpu_parity import _check_decode, _small_pp

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def R():
    return U.load()


def _frame(R, ctx, cfg, pts, a, mode, absent):
    boxes = U.run_frame(ctx, cfg, pts, a, mode, absent=absent)
    hd = R.rtcc_get_head(ctx, cfg.feat_h, cfg.feat_w).copy()
    fb = b"".join(R.rtcc_get_tensor(ctx, 0, R.TENSOR_FUSED_BLOCK0 + bi).tobytes()
                  for bi in range(len(cfg.blocks)))
    return hd, boxes, fb


def _multiscale(R, cfg, absent=(), frame=1, arrivals=None):
    K = cfg.n_agents
    store = cfg.dtype
    pts = [synth.points_for(cfg, frame, k) for k in range(K)]
    a = arrivals if arrivals is not None else synth.arrivals_for(cfg, frame)
    shapes = U.block_shapes(cfg)
    ctx, w = U.make_ctx(cfg, flags=R.FLAG_MULTISCALE)
    try:
        hd, boxes, fbytes = _frame(R, ctx, cfg, pts, a, R.MODE_RTCC, absent)
        blocks_raw = {(k, bi): R.rtcc_get_tensor(ctx, k, bi + 1).tobytes()
                      for k in range(K) if k not in absent for bi in range(len(cfg.blocks))}
        blocks = [[None if k in absent else U.gpu_tensor(ctx, cfg, k, bi + 1, shapes[bi])
                   for k in range(K)] for bi in range(len(cfg.blocks))]
        fused = [U.gpu_tensor(ctx, cfg, 0, R.TENSOR_FUSED_BLOCK0 + bi, shapes[bi])
                 for bi in range(len(cfg.blocks))]
        for bi in range(len(cfg.blocks)):
            if cfg.fusion == "max":
                np.testing.assert_array_equal(fused[bi], of.fuse_max(blocks[bi]),
                                              err_msg=f"max fusion of block {bi}")
            else:
                U.assert_close(fused[bi], of.store_round(of.fuse_attn(blocks[bi]), store),
                               f"attention fusion of block {bi}")
        neck = U.gpu_tensor(ctx, cfg, 0, R.TENSOR_FUSED, (cfg.feat_ch, cfg.feat_h, cfg.feat_w))
        U.assert_close(neck, U.oracle_neck(fused, w, cfg, store), "neck on the fused blocks")
        hd_o = U.head_to_oracle_layout(hd)
        U.assert_close(hd_o, of.head(neck, of.store_round(w["head.w"], store),
                                     of.store_round(w["head.b"], store)), "head on the GPU neck")
        full = of.forward_multiscale([None if k in absent else pts[k] for k in range(K)], w, cfg,
                                     store=store)
        U.assert_close(hd_o, full["head"], "head (end to end)")
        _check_decode(cfg, hd_o, boxes, R, ctx)
        ref = (hd.tobytes(), boxes.tobytes(), fbytes)
        for mode in (R.MODE_BARRIER, R.MODE_RTCC):
            h2, b2, f2 = _frame(R, ctx, cfg, pts, a, mode, absent)
            assert (h2.tobytes(), b2.tobytes(), f2) == ref, f"mode {mode} differs"
    finally:
        R.rtcc_destroy(ctx)
    sctx, _ = U.make_ctx(cfg, flags=0)
    try:
        U.run_frame(sctx, cfg, pts, a, R.MODE_RTCC, absent=absent)
        for (k, bi), raw in blocks_raw.items():
            assert R.rtcc_get_tensor(sctx, k, bi + 1).tobytes() == raw, (k, bi)
    finally:
        R.rtcc_destroy(sctx)


def test_multiscale_small_grid_ragged_tiles(R):
    # 96 x 64 pillars: block grids 48 x 32, 24 x 16, 12 x 8 (ragged 8 x 16 tiles)
    _multiscale(R, _small_pp())


def test_multiscale_small_attention_absent_agent(R):
    cfg = _small_pp("lr5", grid=(128, 48))
    _multiscale(R, cfg, absent=(3,))


@pytest.mark.parametrize("name,absent", [("pp3", ()), ("lr5", (2,))])
def test_multiscale_full_size(R, name, absent):
    _multiscale(R, synth.get_config(name), absent=absent)


def test_multiscale_rejected_without_neck(R):
    cfg = synth.get_config("tiny")
    w = synth.weights_for(cfg)
    with pytest.raises(R.RTCCError):
        R.rtcc_init(R.model_config(cfg, flags=R.FLAG_MULTISCALE), synth.weight_blob(w))

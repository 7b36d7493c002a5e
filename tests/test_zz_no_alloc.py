"""The allocation-free pillarisation entry point.

rtcc_pillarise_noalloc serves callers that cannot allocate device memory
where they need the pass (inside a stream capture, in a plugin host with no
allocator, in a latency-bound loop).  Its scratch is a fixed array the library
reserves on load.  This test runs two different point clouds through it, one
call after the other, and requires for each:

- the pillars (cell map, pillar cells, kept counts, drop counters) bit-exact
  against the oracle's pillarisation;
- the pseudo-image within the parity tolerance of the oracle's PFN + scatter;
- the pseudo-image byte for byte equal to what the existing entry point
  (rtcc_payload_complete on a full-size 3-agent context) writes for the same
  points.

The second call also shows that leftovers of the first call in the shared
array do not leak into the next result.  Oversized and misaligned requests
must be refused before any work is enqueued.  The file is named to be
collected last.
"""
import numpy as np
import pytest

import synth
from oracle import forward as of
from tests import gpu_util as U

pytestmark = pytest.mark.gpu


def test_noalloc_matches_oracle_and_context_on_two_calls():
    torch = pytest.importorskip("torch")
    R = U.load()
    cfg = synth.get_config("pp3")
    ctx, w = U.make_ctx(cfg, flags=0)
    pts = [synth.points_for(cfg, 5, k) for k in range(cfg.n_agents)]
    U.run_frame(ctx, cfg, pts, [0.0, 1.0, 2.0], R.MODE_RTCC)
    ctx_img = {k: R.rtcc_get_tensor(ctx, k, R.TENSOR_IMAGE).copy() for k in (0, 1)}
    R.rtcc_destroy(ctx)

    dev = torch.device("cuda")
    # the PFN weights as rtcc_init stores them: rounded once to the storage type
    pw = torch.tensor(of.store_round(w["pfn.w"], cfg.dtype).astype(np.float32), device=dev)
    pb = torch.tensor(of.store_round(w["pfn.b"], cfg.dtype).astype(np.float32), device=dev)
    cells = cfg.grid_w * cfg.grid_h
    c2p = torch.empty(cells, dtype=torch.int32, device=dev)
    pcell = torch.empty(cfg.max_pillars, dtype=torch.int32, device=dev)
    cnt = torch.empty(cfg.max_pillars, dtype=torch.int32, device=dev)
    stats = torch.empty(8, dtype=torch.int32, device=dev)
    img = torch.empty(cells * cfg.pfn_ch, dtype=torch.int16, device=dev)
    c = R.model_config(cfg)
    for k in (0, 1):                                   # two calls in a row
        d_pts = torch.from_numpy(pts[k]).to(dev)
        for t in (c2p, pcell, cnt, img):
            t.fill_(-7)
        stats.fill_(12345)                             # must be cleared by the call
        torch.cuda.synchronize()
        s = R.rtcc_pillarise_noalloc(c, d_pts.data_ptr(), pts[k].shape[0], pw.data_ptr(),
                                     pb.data_ptr(), c2p.data_ptr(), pcell.data_ptr(),
                                     cnt.data_ptr(), stats.data_ptr(), img.data_ptr(), 0)
        assert s == R.OK, R.rtcc_status_str(s)
        torch.cuda.synchronize()
        op = of.pillarise(pts[k], cfg)
        n = op["n_pillars"]
        st = stats.cpu().numpy()
        assert st[0] == pts[k].shape[0] and st[2] == n and st[3] == op["count"][:n].sum()
        assert st[0] - st[1] == op["drop_range"]
        assert st[1] - st[7] == op["drop_pcap"] and st[6] == op["drop_ncap"]
        np.testing.assert_array_equal(c2p.cpu().numpy(), op["cell2pillar"])
        np.testing.assert_array_equal(pcell.cpu().numpy()[:n], op["pillar_cell"][:n])
        np.testing.assert_array_equal(cnt.cpu().numpy()[:n], op["count"][:n])
        raw = img.cpu().numpy().view(np.uint16)
        got = U.u16_to_f64(raw, cfg.dtype).reshape(cfg.grid_h, cfg.grid_w, cfg.pfn_ch)
        want = of.scatter(of.pfn(op, w["pfn.w"], w["pfn.b"], cfg, cfg.dtype), op, cfg)
        U.assert_close(got.transpose(2, 0, 1), want, f"pseudo-image call {k}")
        assert raw.tobytes() == ctx_img[k].tobytes(), f"call {k}: image differs from the context's"

    big = R.model_config(cfg)
    big.grid_w, big.grid_h = 512, 512                  # 262,144 cells > the 65,536 limit
    s = R.rtcc_pillarise_noalloc(big, d_pts.data_ptr(), pts[1].shape[0], pw.data_ptr(),
                                 pb.data_ptr(), c2p.data_ptr(), pcell.data_ptr(), cnt.data_ptr(),
                                 stats.data_ptr(), img.data_ptr(), 0)
    assert s == R.E_ARG
    s = R.rtcc_pillarise_noalloc(c, d_pts.data_ptr(), 200000, pw.data_ptr(), pb.data_ptr(),
                                 c2p.data_ptr(), pcell.data_ptr(), cnt.data_ptr(),
                                 stats.data_ptr(), img.data_ptr(), 0)
    assert s == R.E_ARG
    # sub-views that are not 16-byte aligned are refused (nothing is launched)
    s = R.rtcc_pillarise_noalloc(c, d_pts.data_ptr() + 4, 1000, pw.data_ptr(), pb.data_ptr(),
                                 c2p.data_ptr(), pcell.data_ptr(), cnt.data_ptr(),
                                 stats.data_ptr(), img.data_ptr(), 0)
    assert s == R.E_ARG
    s = R.rtcc_pillarise_noalloc(c, d_pts.data_ptr(), 1000, pw.data_ptr(), pb.data_ptr(),
                                 c2p.data_ptr(), pcell.data_ptr(), cnt.data_ptr(),
                                 stats.data_ptr(), img.data_ptr() + 8, 0)
    assert s == R.E_ARG

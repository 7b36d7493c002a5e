"""Seeded synthetic inputs for the cooperative-perception workloads.

This module is shared by the CUDA path's tests/benchmark and by the CPU oracle.
It holds only workload descriptions (grid sizes, channel counts, ranges) and
seeded random draws: point clouds, fp32 master weights and uplink-completion
traces (or the raw channel draws a slot simulator consumes).  It contains none
of the method's arithmetic: no pillarisation, no network layer, no scheduling.

The paper evaluates a trained PointPillars-style attentive-fusion detector on
OPV2V frames with OFDMA uplink traces (Sec. V-A, Table II).  Neither the
dataset nor the checkpoint is available, so every input here is a synthetic
stand-in with the shapes of those workloads: uniform ground clutter plus
Gaussian object clusters, He-normal weights, and seeded arrival times.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence, Tuple

import numpy as np

__all__ = [
    "ModelConfig", "CONFIGS", "get_config", "points_for", "weights_for",
    "weight_layout", "arrivals_for", "channel_draws", "points_cap_patch",
]


@dataclasses.dataclass(frozen=True)
class ModelConfig:
    """Shape of one workload.  Units: metres, milliseconds."""

    name: str
    n_agents: int
    grid_w: int                   # pillars along x
    grid_h: int                   # pillars along y
    x_min: float
    y_min: float
    z_min: float
    x_max: float
    y_max: float
    z_max: float
    pillar: float                 # pillar edge length
    max_pillars: int              # P_max
    max_pts: int                  # N_max, points kept per pillar
    pfn_ch: int                   # C_p
    blocks: Tuple[Tuple[int, int, int], ...]   # (n_conv, channels, first stride)
    up_strides: Tuple[int, ...]   # deconv kernel = stride per block; () = no neck
    up_ch: int                    # channels of each deconv output
    fusion: str                   # "max" or "attn"
    anchors: int                  # anchors per BEV cell
    dtype: str                    # storage type on the GPU: "fp16" or "bf16"
    max_boxes: int                # top-K after thresholding
    cls_thresh: float             # logit threshold (score >= sigmoid(cls_thresh))
    # synthetic point recipe
    n_uniform: int
    n_clusters: int
    cluster_pts: int
    cluster_sigma: float
    pts_x: Tuple[float, float]
    pts_y: Tuple[float, float]
    pts_z: Tuple[float, float]
    weight_seed: int
    point_seed: int
    arrival: str                  # "fixed", "uniform", "lognormal", "slots", "zero"
    arrival_args: Tuple[float, ...] = ()
    nms_iou: float = 0.15         # rotated BEV NMS: suppress IoU > nms_iou (0: no NMS)

    # ---- derived shapes (no arithmetic of the method, only bookkeeping) ----
    @property
    def max_points_per_agent(self) -> int:
        return self.n_uniform + self.n_clusters * self.cluster_pts

    @property
    def feat_stride(self) -> int:
        """Downsampling of the fused BEV map relative to the pillar grid."""
        s = 1
        for (_, _, st) in self.blocks[:1]:
            s *= st
        return s

    @property
    def feat_w(self) -> int:
        return self.grid_w // self.feat_stride

    @property
    def feat_h(self) -> int:
        return self.grid_h // self.feat_stride

    @property
    def feat_ch(self) -> int:
        if self.up_strides:
            return self.up_ch * len(self.up_strides)
        return self.blocks[-1][1]

    @property
    def head_ch(self) -> int:
        return self.anchors * 8


def _cfg(**kw) -> ModelConfig:
    return ModelConfig(**kw)


_PP_BLOCKS = ((3, 64, 2), (5, 128, 2), (5, 256, 2))

CONFIGS = {
    # 2 agents, 64x64 grid, three 3x3 convs of 32 channels, max fusion.
    "tiny": _cfg(
        name="tiny", n_agents=2, grid_w=64, grid_h=64,
        x_min=-12.8, y_min=-12.8, z_min=-3.0, x_max=12.8, y_max=12.8, z_max=1.0,
        pillar=0.4, max_pillars=2048, max_pts=16, pfn_ch=32,
        blocks=((3, 32, 1),), up_strides=(), up_ch=0, fusion="max", anchors=2,
        dtype="fp16", max_boxes=128, cls_thresh=0.0,
        n_uniform=2048, n_clusters=0, cluster_pts=0, cluster_sigma=0.0,
        pts_x=(-12.8, 12.8), pts_y=(-12.8, 12.8), pts_z=(-3.0, 1.0),
        weight_seed=0, point_seed=0, arrival="fixed", arrival_args=(0.0, 5.0)),
    # 3-agent PointPillars intermediate fusion, 256x256 grid, max fusion.
    "pp3": _cfg(
        name="pp3", n_agents=3, grid_w=256, grid_h=256,
        x_min=-51.2, y_min=-51.2, z_min=-3.0, x_max=51.2, y_max=51.2, z_max=1.0,
        pillar=0.4, max_pillars=12000, max_pts=32, pfn_ch=64,
        blocks=_PP_BLOCKS, up_strides=(1, 2, 4), up_ch=128, fusion="max", anchors=2,
        dtype="fp16", max_boxes=256, cls_thresh=0.0,
        n_uniform=100000, n_clusters=20, cluster_pts=500, cluster_sigma=0.5,
        pts_x=(-51.2, 51.2), pts_y=(-51.2, 51.2), pts_z=(-3.0, 1.0),
        weight_seed=1, point_seed=1, arrival="uniform", arrival_args=(0.0, 30.0)),
    # 5-agent attention fusion on a long-range 704x200 grid, bf16.
    "lr5": _cfg(
        name="lr5", n_agents=5, grid_w=704, grid_h=200,
        x_min=-140.8, y_min=-40.0, z_min=-3.0, x_max=140.8, y_max=40.0, z_max=1.0,
        pillar=0.4, max_pillars=16000, max_pts=32, pfn_ch=64,
        blocks=_PP_BLOCKS, up_strides=(1, 2, 4), up_ch=128, fusion="attn", anchors=2,
        dtype="bf16", max_boxes=256, cls_thresh=0.0,
        n_uniform=120000, n_clusters=20, cluster_pts=500, cluster_sigma=0.5,
        pts_x=(-140.8, 140.8), pts_y=(-40.0, 40.0), pts_z=(-3.0, 1.0),
        weight_seed=2, point_seed=2, arrival="lognormal",
        arrival_args=(math.log(10.0), 0.8)),
    # 4 agents on the pp3 network; arrivals from a slot-level uplink simulator.
    "sweep4": _cfg(
        name="sweep4", n_agents=4, grid_w=256, grid_h=256,
        x_min=-51.2, y_min=-51.2, z_min=-3.0, x_max=51.2, y_max=51.2, z_max=1.0,
        pillar=0.4, max_pillars=12000, max_pts=32, pfn_ch=64,
        blocks=_PP_BLOCKS, up_strides=(1, 2, 4), up_ch=128, fusion="max", anchors=2,
        dtype="fp16", max_boxes=256, cls_thresh=0.0,
        n_uniform=100000, n_clusters=20, cluster_pts=500, cluster_sigma=0.5,
        pts_x=(-51.2, 51.2), pts_y=(-51.2, 51.2), pts_z=(-3.0, 1.0),
        weight_seed=1, point_seed=3, arrival="slots", arrival_args=()),
    # 8-agent stress on the long-range grid with max fusion.
    "stress8": _cfg(
        name="stress8", n_agents=8, grid_w=704, grid_h=200,
        x_min=-140.8, y_min=-40.0, z_min=-3.0, x_max=140.8, y_max=40.0, z_max=1.0,
        pillar=0.4, max_pillars=16000, max_pts=32, pfn_ch=64,
        blocks=_PP_BLOCKS, up_strides=(1, 2, 4), up_ch=128, fusion="max", anchors=2,
        dtype="fp16", max_boxes=256, cls_thresh=0.0,
        n_uniform=150000, n_clusters=20, cluster_pts=500, cluster_sigma=0.5,
        pts_x=(-140.8, 140.8), pts_y=(-40.0, 40.0), pts_z=(-3.0, 1.0),
        weight_seed=2, point_seed=4, arrival="lognormal",
        arrival_args=(math.log(10.0), 0.8)),
}


def get_config(name: str, **overrides) -> ModelConfig:
    """Preset by name, optionally with fields replaced (for small test cases)."""
    cfg = CONFIGS[name]
    if overrides:
        cfg = dataclasses.replace(cfg, **overrides)
    return cfg


# --------------------------------------------------------------------------
# point clouds
# --------------------------------------------------------------------------

def points_for(cfg: ModelConfig, frame: int, agent: int) -> np.ndarray:
    """float32 [n, 4] = (x, y, z, intensity) for one agent of one frame.

    Uniform clutter over the configured box, then ``n_clusters`` isotropic
    Gaussian blobs (object stand-ins), concatenated and shuffled by one seeded
    permutation so that the point order (which decides which pillars survive
    the caps) does not favour either population.
    """
    rng = np.random.default_rng([cfg.point_seed, frame, agent])
    n_u = cfg.n_uniform
    pts = np.empty((n_u, 4), dtype=np.float64)
    pts[:, 0] = rng.uniform(cfg.pts_x[0], cfg.pts_x[1], n_u)
    pts[:, 1] = rng.uniform(cfg.pts_y[0], cfg.pts_y[1], n_u)
    pts[:, 2] = rng.uniform(cfg.pts_z[0], cfg.pts_z[1], n_u)
    pts[:, 3] = rng.uniform(0.0, 1.0, n_u)
    parts = [pts]
    for _ in range(cfg.n_clusters):
        c = np.array([rng.uniform(cfg.pts_x[0], cfg.pts_x[1]),
                      rng.uniform(cfg.pts_y[0], cfg.pts_y[1]),
                      rng.uniform(-2.0, 0.0)])
        blob = np.empty((cfg.cluster_pts, 4))
        blob[:, :3] = c + rng.normal(0.0, cfg.cluster_sigma, (cfg.cluster_pts, 3))
        blob[:, 3] = rng.uniform(0.0, 1.0, cfg.cluster_pts)
        parts.append(blob)
    allp = np.concatenate(parts, axis=0)
    allp = allp[rng.permutation(allp.shape[0])]
    out = allp.astype(np.float32)
    assert np.isfinite(out).all()
    return np.ascontiguousarray(out)


def points_cap_patch(n: int = 2048, cells: int = 8, pillar: float = 0.4,
                     x0: float = -12.8, y0: float = -12.8, seed: int = 7) -> np.ndarray:
    """Dense points inside a small ``cells`` x ``cells`` patch of the grid.

    Used with small pillar/point caps so that both caps bind.  Points are drawn
    strictly inside cell interiors (a 5 % margin) so that no coordinate sits on
    a cell edge.
    """
    rng = np.random.default_rng(seed)
    cx = rng.integers(0, cells, n)
    cy = rng.integers(0, cells, n)
    fx = rng.uniform(0.05, 0.95, n)
    fy = rng.uniform(0.05, 0.95, n)
    pts = np.empty((n, 4))
    pts[:, 0] = x0 + (cx + fx) * pillar
    pts[:, 1] = y0 + (cy + fy) * pillar
    pts[:, 2] = rng.uniform(-3.0, 1.0, n)
    pts[:, 3] = rng.uniform(0.0, 1.0, n)
    return pts.astype(np.float32)


# --------------------------------------------------------------------------
# weights
# --------------------------------------------------------------------------

def weight_layout(cfg: ModelConfig) -> List[Tuple[str, Tuple[int, ...], int]]:
    """Ordered (name, shape, fan_in) of every tensor in the weight blob.

    Order: PFN W [C_p][9], b; every 3x3 conv of every block W [Co][Ci][3][3],
    b; every deconv W [Ci][Co][s][s], b; head W [A*8][C_feat], b.
    """
    out = [("pfn.w", (cfg.pfn_ch, 9), 9), ("pfn.b", (cfg.pfn_ch,), 0)]
    cin = cfg.pfn_ch
    for bi, (n, ch, _st) in enumerate(cfg.blocks):
        for li in range(n):
            out.append((f"b{bi}.c{li}.w", (ch, cin, 3, 3), 9 * cin))
            out.append((f"b{bi}.c{li}.b", (ch,), 0))
            cin = ch
    for bi, s in enumerate(cfg.up_strides):
        ci = cfg.blocks[bi][1]
        out.append((f"up{bi}.w", (ci, cfg.up_ch, s, s), ci))
        out.append((f"up{bi}.b", (cfg.up_ch,), 0))
    out.append(("head.w", (cfg.head_ch, cfg.feat_ch), cfg.feat_ch))
    out.append(("head.b", (cfg.head_ch,), 0))
    return out


def pfn_feature_stats(cfg: ModelConfig) -> Tuple[np.ndarray, np.ndarray]:
    """Population mean and variance of the 9 PFN input features under the
    synthetic point recipe (x, y, z, intensity uniform over their ranges;
    offsets to the pillar mean and centre spread over one pillar)."""
    v = cfg.pillar
    ux = lambda lo, hi: ((lo + hi) / 2.0, (hi - lo) ** 2 / 12.0)
    mx, vx = ux(*cfg.pts_x)
    my, vy = ux(*cfg.pts_y)
    mz, vz = ux(*cfg.pts_z)
    mean = np.array([mx, my, mz, 0.5, 0.0, 0.0, 0.0, 0.0, 0.0])
    var = np.array([vx, vy, vz, 1.0 / 12.0, v * v / 12.0, v * v / 12.0, vz / 2.0,
                    v * v / 12.0, v * v / 12.0])
    return mean, var


def weights_for(cfg: ModelConfig) -> dict:
    """fp32 master weights: He-normal std sqrt(2/fan_in), biases U(-0.1, 0.1).

    The PFN's linear layer is followed by BatchNorm in PointPillars; here a
    BatchNorm with the synthetic inputs' population statistics (gamma = 1,
    beta = the drawn bias) is folded into the PFN weight and bias, so that the
    PFN output -- and with He-normal layers after it, every activation -- has
    unit scale as in a trained, normalised network.

    Returns an ordered dict name -> float32 array; ``np.concatenate`` of the
    flattened values in order is the blob the C library takes.
    """
    rng = np.random.default_rng(cfg.weight_seed)
    out = {}
    for name, shape, fan_in in weight_layout(cfg):
        if name.endswith(".w"):
            v = rng.normal(0.0, math.sqrt(2.0 / fan_in), shape)
        else:
            v = rng.uniform(-0.1, 0.1, shape)
        out[name] = v
    mean, var = pfn_feature_stats(cfg)
    w = out["pfn.w"]
    sigma = np.sqrt((w * w * var[None, :]).sum(axis=1))
    mu = w @ mean
    out["pfn.w"] = w / sigma[:, None]
    out["pfn.b"] = out["pfn.b"] - mu / sigma
    return {k: v.astype(np.float32) for k, v in out.items()}


def weight_blob(weights: dict) -> np.ndarray:
    return np.ascontiguousarray(np.concatenate([v.reshape(-1) for v in weights.values()]))


# --------------------------------------------------------------------------
# uplink-completion traces
# --------------------------------------------------------------------------

def arrivals_for(cfg: ModelConfig, frame: int, spread: Optional[str] = None) -> np.ndarray:
    """Per-agent uplink completion times a_k in ms (float64 [K]) for one frame.

    ``spread`` overrides the preset recipe ("zero" = all simultaneous).  The
    "slots" recipe is produced by a slot-level uplink simulator from
    :func:`channel_draws`; it is not drawn here.
    """
    kind = spread or cfg.arrival
    rng = np.random.default_rng([cfg.point_seed, 1_000_003, frame])
    K = cfg.n_agents
    if kind == "fixed":
        a = np.array(cfg.arrival_args[:K], dtype=np.float64)
    elif kind == "uniform":
        lo, hi = cfg.arrival_args
        a = rng.uniform(lo, hi, K)
    elif kind == "lognormal":
        mu, sigma = cfg.arrival_args
        a = np.exp(rng.normal(mu, sigma, K))
    elif kind == "zero":
        a = np.zeros(K)
    else:
        raise ValueError(f"arrival recipe {kind!r} is not a direct draw")
    return a


def channel_draws(n_agents: int, n_slots: int, n_rb: int, frame: int, seed: int = 3,
                  snr_db: Tuple[float, float] = (0.0, 25.0)) -> dict:
    """Random draws of one frame of a slot-level uplink.

    Returns mean SNR per agent (linear, drawn once per frame from U[snr_db] in
    dB) and small-scale fading power |h|^2 ~ Exp(1), i.i.d. per slot, agent and
    resource block, shaped [n_slots][n_agents][n_rb].
    """
    rng = np.random.default_rng([seed, 77, frame])
    snr = 10.0 ** (rng.uniform(snr_db[0], snr_db[1], n_agents) / 10.0)
    h2 = rng.exponential(1.0, (n_slots, n_agents, n_rb))
    return {"snr": snr, "h2": h2}

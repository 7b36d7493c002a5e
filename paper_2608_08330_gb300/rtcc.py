"""Thin ctypes binding of ``include/rtcc.h`` (argument marshalling only).

Every function here has the name of the C entry point it wraps and only
converts arguments; all work runs in the compiled library.  The library is
loaded on first use from ``paper_2608_08330_gb300/_build/librtcc.so`` and a
missing library raises -- there is no fallback.
"""
from __future__ import annotations

import ctypes as C
import math
import os
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "librtcc.so")

MAX_AGENTS = 8
MAX_BLOCKS = 3

# status codes (rtcc_status)
OK, E_ARG, E_AGENT, E_DUPLICATE, E_PREMATURE, E_MALFORMED, E_STATE, E_TIMEOUT, \
    E_INFEASIBLE, E_CUDA, E_NOMEM, E_DEVICE = range(12)
MODE_RTCC, MODE_BARRIER = 0, 1
FUSE_MAX, FUSE_ATTN = 0, 1
FP16, BF16 = 0, 1
WAITING, RELEASED, RUNNING, FINISHED, ABSENT = range(5)
FLAG_TIMELINE, FLAG_KEEP_FUSED, FLAG_KEEP_LAYERS, FLAG_LAYER_TIMES = 1, 2, 4, 8
FLAG_NO_CLUSTERS, FLAG_SHORT_WAITS, FLAG_NO_BATCH, FLAG_H2D_COPY = 16, 32, 64, 128
FLAG_MULTISCALE = 256
TENSOR_IMAGE, TENSOR_FEAT, TENSOR_FUSED, TENSOR_LAYER0 = 0, 8, 9, 16
TENSOR_FUSED_BLOCK0 = 10


class rtcc_model_config(C.Structure):
    _fields_ = [
        ("n_agents", C.c_int32), ("grid_w", C.c_int32), ("grid_h", C.c_int32),
        ("x_min", C.c_float), ("y_min", C.c_float), ("z_min", C.c_float),
        ("x_max", C.c_float), ("y_max", C.c_float), ("z_max", C.c_float),
        ("pillar", C.c_float), ("max_pillars", C.c_int32), ("max_pts", C.c_int32),
        ("pfn_ch", C.c_int32), ("n_blocks", C.c_int32),
        ("block_layers", C.c_int32 * MAX_BLOCKS), ("block_ch", C.c_int32 * MAX_BLOCKS),
        ("block_stride", C.c_int32 * MAX_BLOCKS), ("up_stride", C.c_int32 * MAX_BLOCKS),
        ("up_ch", C.c_int32), ("fusion", C.c_int32), ("anchors", C.c_int32),
        ("dtype", C.c_int32), ("max_points", C.c_int32), ("max_boxes", C.c_int32),
        ("cls_thresh", C.c_float), ("nms_iou", C.c_float), ("flags", C.c_int32),
    ]


class rtcc_box(C.Structure):
    _fields_ = [("x", C.c_float), ("y", C.c_float), ("z", C.c_float), ("l", C.c_float),
                ("w", C.c_float), ("h", C.c_float), ("yaw", C.c_float), ("score", C.c_float),
                ("anchor", C.c_int32)]


class rtcc_frame_info(C.Structure):
    _fields_ = [
        ("t_last_event_ms", C.c_double), ("t_ready_ms", C.c_double),
        ("t_release_ms", C.c_double * MAX_AGENTS),
        ("gpu_backbone_ms", C.c_float * MAX_AGENTS), ("gpu_branch_ms", C.c_float * MAX_AGENTS),
        ("gpu_fusion_ms", C.c_float), ("gpu_post_ms", C.c_float),
        ("dispatch_order", C.c_int32 * MAX_AGENTS), ("n_dispatched", C.c_int32),
        ("gpu_fusion_kernel_ms", C.c_float), ("gpu_pfn_kernel_ms", C.c_float * MAX_AGENTS),
        ("n_backbone_launches", C.c_int32), ("backbone_batch", C.c_int32 * MAX_AGENTS),
        ("gpu_launch_ms", C.c_float * MAX_AGENTS),
    ]


class rtcc_conv_plan(C.Structure):
    _fields_ = [("splits", C.c_int32), ("bn", C.c_int32), ("tall", C.c_int32),
                ("transposed", C.c_int32), ("wide", C.c_int32), ("m_tiles", C.c_int32),
                ("items", C.c_int32)]


BOX_DTYPE = np.dtype([("x", "<f4"), ("y", "<f4"), ("z", "<f4"), ("l", "<f4"), ("w", "<f4"),
                      ("h", "<f4"), ("yaw", "<f4"), ("score", "<f4"), ("anchor", "<i4")])

_ctx_p = C.c_void_p
_ctrl_p = C.c_void_p
_lib = None


class RTCCError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {rtcc_status_str(status)} ({status})")


def load(path: Optional[str] = None) -> C.CDLL:
    """Load the compiled library (raises if it was not built)."""
    global _lib
    if _lib is not None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"RTCC library not built: {p} (run paper_2608_08330_gb300.build)")
    lib = C.CDLL(p)
    S = C.c_int
    sig = {
        "rtcc_init": (S, [C.POINTER(rtcc_model_config), C.POINTER(C.c_float), C.c_size_t,
                          C.POINTER(_ctx_p)]),
        "rtcc_destroy": (None, [_ctx_p]),
        "rtcc_set_mode": (S, [_ctx_p, C.c_int]),
        "rtcc_staging_buffer": (S, [_ctx_p, C.c_int32, C.POINTER(C.POINTER(C.c_float)),
                                    C.POINTER(C.c_int32)]),
        "rtcc_stage_resident": (S, [_ctx_p, C.c_int32, C.c_void_p, C.c_int32]),
        "rtcc_frame_begin": (S, [_ctx_p, C.c_uint64, C.c_double]),
        "rtcc_payload_complete": (S, [_ctx_p, C.c_int32, C.c_void_p, C.c_int32, C.c_double]),
        "rtcc_payload_resident": (S, [_ctx_p, C.c_int32, C.c_double]),
        "rtcc_payload_absent": (S, [_ctx_p, C.c_int32, C.c_double]),
        "rtcc_frame_abort": (S, [_ctx_p]),
        "rtcc_wait_detection": (S, [_ctx_p, C.c_int32, C.c_void_p, C.c_int32,
                                    C.POINTER(C.c_int32), C.POINTER(C.c_double)]),
        "rtcc_get_frame_info": (S, [_ctx_p, C.POINTER(rtcc_frame_info)]),
        "rtcc_get_branch_state": (S, [_ctx_p, C.c_int32, C.POINTER(C.c_int32),
                                      C.POINTER(C.c_double)]),
        "rtcc_get_layer_times": (S, [_ctx_p, C.c_int32, C.c_void_p, C.c_int32,
                                     C.POINTER(C.c_int32)]),
        "rtcc_get_layer_spans": (S, [_ctx_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_int32,
                                     C.POINTER(C.c_int32)]),
        "rtcc_get_head": (S, [_ctx_p, C.c_void_p, C.c_size_t]),
        "rtcc_get_decoded": (S, [_ctx_p, C.c_void_p, C.c_int32, C.POINTER(C.c_int32)]),
        "rtcc_nms": (S, [C.c_void_p, C.c_int32, C.c_float, C.c_void_p, C.POINTER(C.c_int32)]),
        "rtcc_get_pillars": (S, [_ctx_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p,
                                 C.c_void_p]),
        "rtcc_get_tensor": (S, [_ctx_p, C.c_int32, C.c_int32, C.c_void_p, C.c_size_t,
                                C.POINTER(C.c_size_t)]),
        "rtcc_ctrl_create": (S, [C.c_int32, C.c_int32, C.c_int32, C.POINTER(_ctrl_p)]),
        "rtcc_ctrl_destroy": (None, [_ctrl_p]),
        "rtcc_ctrl_set_mode": (S, [_ctrl_p, C.c_int]),
        "rtcc_ctrl_begin": (S, [_ctrl_p, C.c_uint64, C.c_double]),
        "rtcc_ctrl_complete": (S, [_ctrl_p, C.c_int32, C.c_void_p, C.c_int32, C.c_double,
                                   C.POINTER(C.c_int32), C.POINTER(C.c_int32)]),
        "rtcc_ctrl_absent": (S, [_ctrl_p, C.c_int32, C.c_double, C.POINTER(C.c_int32),
                                 C.POINTER(C.c_int32)]),
        "rtcc_ctrl_mark": (S, [_ctrl_p, C.c_int32, C.c_int32]),
        "rtcc_ctrl_abort": (S, [_ctrl_p]),
        "rtcc_ctrl_join_ready": (C.c_int32, [_ctrl_p]),
        "rtcc_ctrl_state": (S, [_ctrl_p, C.c_int32, C.POINTER(C.c_int32),
                                C.POINTER(C.c_double)]),
        "rtcc_ctrl_end": (S, [_ctrl_p]),
        "rtcc_status_str": (C.c_char_p, [C.c_int]),
        "rtcc_now_ms": (C.c_double, []),
        "rtcc_kernels_per_frame": (C.c_int32, [_ctx_p, C.c_int32]),
        "rtcc_test_unreachable_wait": (S, [_ctx_p]),
        "rtcc_uplink_simulate": (S, [C.c_int32, C.c_int32, C.c_int32, C.c_void_p, C.c_void_p,
                                     C.c_void_p, C.c_double, C.c_int32, C.c_void_p, C.c_void_p,
                                     C.POINTER(C.c_int32)]),
        "rtcc_plan_conv": (S, [C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_int32,
                               C.c_int32, C.POINTER(rtcc_conv_plan)]),
        "rtcc_pillarise_noalloc": (S, [C.POINTER(rtcc_model_config), C.c_void_p, C.c_int32,
                                       C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                       C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


def _chk(status: int, where: str) -> int:
    if status != OK:
        raise RTCCError(status, where)
    return status


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


# --------------------------------------------------------------------------
# config marshalling
# --------------------------------------------------------------------------

def model_config(cfg, max_points: Optional[int] = None, flags: int = 0) -> rtcc_model_config:
    """Fill the C config from any object with the workload fields
    (n_agents, grid_w, grid_h, ranges, pillar, max_pillars, max_pts, pfn_ch,
    blocks = [(n_conv, channels, stride)], up_strides, up_ch, fusion, anchors,
    dtype, max_boxes, cls_thresh; nms_iou, absent = 0, no NMS)."""
    c = rtcc_model_config()
    c.n_agents = cfg.n_agents
    c.grid_w, c.grid_h = cfg.grid_w, cfg.grid_h
    c.x_min, c.y_min, c.z_min = cfg.x_min, cfg.y_min, cfg.z_min
    c.x_max, c.y_max, c.z_max = cfg.x_max, cfg.y_max, cfg.z_max
    c.pillar = cfg.pillar
    c.max_pillars, c.max_pts, c.pfn_ch = cfg.max_pillars, cfg.max_pts, cfg.pfn_ch
    c.n_blocks = len(cfg.blocks)
    for i, (n, ch, st) in enumerate(cfg.blocks):
        c.block_layers[i], c.block_ch[i], c.block_stride[i] = n, ch, st
    for i, s in enumerate(cfg.up_strides):
        c.up_stride[i] = s
    c.up_ch = cfg.up_ch
    c.fusion = FUSE_ATTN if cfg.fusion == "attn" else FUSE_MAX
    c.anchors = cfg.anchors
    c.dtype = BF16 if cfg.dtype == "bf16" else FP16
    c.max_points = cfg.max_points_per_agent if max_points is None else max_points
    c.max_boxes = cfg.max_boxes
    c.cls_thresh = cfg.cls_thresh
    c.nms_iou = float(getattr(cfg, "nms_iou", 0.0))
    c.flags = flags
    return c


# --------------------------------------------------------------------------
# context API (same names as the C entry points)
# --------------------------------------------------------------------------

def rtcc_init(cfg: rtcc_model_config, weights: np.ndarray) -> C.c_void_p:
    lib = load()
    w = np.ascontiguousarray(weights, dtype=np.float32)
    out = _ctx_p()
    _chk(lib.rtcc_init(C.byref(cfg), w.ctypes.data_as(C.POINTER(C.c_float)), w.size,
                       C.byref(out)), "rtcc_init")
    return out


def rtcc_destroy(ctx) -> None:
    load().rtcc_destroy(ctx)


def rtcc_set_mode(ctx, mode: int) -> int:
    return load().rtcc_set_mode(ctx, mode)


def rtcc_staging_buffer(ctx, agent: int) -> np.ndarray:
    """The agent's pinned staging buffer as a float32 [cap][4] array view."""
    ptr = C.POINTER(C.c_float)()
    cap = C.c_int32()
    _chk(load().rtcc_staging_buffer(ctx, agent, C.byref(ptr), C.byref(cap)), "rtcc_staging_buffer")
    return np.ctypeslib.as_array(ptr, shape=(max(cap.value, 1), 4))


def rtcc_stage_resident(ctx, agent: int, points: Optional[np.ndarray]) -> int:
    n = 0 if points is None else int(points.shape[0])
    return load().rtcc_stage_resident(ctx, agent, _ptr(points), n)


def rtcc_frame_begin(ctx, frame_id: int, t0_ms: float) -> int:
    return load().rtcc_frame_begin(ctx, frame_id, t0_ms)


def rtcc_payload_complete(ctx, agent: int, points: Optional[np.ndarray], t_ms: float,
                          n_points: Optional[int] = None) -> int:
    if points is not None:
        assert points.dtype == np.float32 and points.flags.c_contiguous
    n = (0 if points is None else int(points.shape[0])) if n_points is None else n_points
    return load().rtcc_payload_complete(ctx, agent, _ptr(points), n, t_ms)


def rtcc_payload_resident(ctx, agent: int, t_ms: float) -> int:
    return load().rtcc_payload_resident(ctx, agent, t_ms)


def rtcc_payload_absent(ctx, agent: int, t_ms: float) -> int:
    return load().rtcc_payload_absent(ctx, agent, t_ms)


def rtcc_frame_abort(ctx) -> int:
    return load().rtcc_frame_abort(ctx)


def rtcc_wait_detection(ctx, timeout_ms: int = -1, cap: int = 512):
    """Returns (status, boxes structured array, t_ready_ms)."""
    out = np.zeros(cap, dtype=BOX_DTYPE)
    n = C.c_int32(0)
    t = C.c_double(0.0)
    s = load().rtcc_wait_detection(ctx, timeout_ms, _ptr(out), cap, C.byref(n), C.byref(t))
    return s, out[:min(n.value, cap)], t.value


def rtcc_get_frame_info(ctx) -> rtcc_frame_info:
    info = rtcc_frame_info()
    _chk(load().rtcc_get_frame_info(ctx, C.byref(info)), "rtcc_get_frame_info")
    return info


def rtcc_get_layer_times(ctx, agent: int) -> np.ndarray:
    """Per-layer ms (first input-ready to last item counted) of the agent's
    conv/deconv layers in the last frame."""
    lib = load()
    n = C.c_int32(0)
    _chk(lib.rtcc_get_layer_times(ctx, agent, None, 0, C.byref(n)), "rtcc_get_layer_times")
    out = np.empty(n.value, dtype=np.float32)
    _chk(lib.rtcc_get_layer_times(ctx, agent, _ptr(out), out.size, C.byref(n)),
         "rtcc_get_layer_times")
    return out


def rtcc_get_layer_spans(ctx, agent: int):
    """(start_ms, end_ms) of each conv/deconv layer of the agent's backbone in
    the last frame, from the earliest layer start."""
    lib = load()
    n = C.c_int32(0)
    _chk(lib.rtcc_get_layer_spans(ctx, agent, None, None, 0, C.byref(n)), "rtcc_get_layer_spans")
    a = np.empty(n.value, dtype=np.float32)
    e = np.empty(n.value, dtype=np.float32)
    _chk(lib.rtcc_get_layer_spans(ctx, agent, _ptr(a), _ptr(e), a.size, C.byref(n)),
         "rtcc_get_layer_spans")
    return a, e


def rtcc_get_branch_state(ctx, agent: int):
    st = C.c_int32()
    r = C.c_double()
    s = load().rtcc_get_branch_state(ctx, agent, C.byref(st), C.byref(r))
    return s, st.value, r.value


def rtcc_get_head(ctx, feat_h: int, feat_w: int) -> np.ndarray:
    out = np.empty((feat_h, feat_w, 16), dtype=np.float32)
    _chk(load().rtcc_get_head(ctx, _ptr(out), out.size), "rtcc_get_head")
    return out


def rtcc_get_decoded(ctx, cap: int = 512) -> np.ndarray:
    """The decode's top-K boxes before NMS, in rank order."""
    out = np.zeros(cap, dtype=BOX_DTYPE)
    n = C.c_int32(0)
    _chk(load().rtcc_get_decoded(ctx, _ptr(out), cap, C.byref(n)), "rtcc_get_decoded")
    return out[:min(n.value, cap)]


def rtcc_nms(boxes: np.ndarray, iou: float) -> np.ndarray:
    """Rotated BEV NMS of boxes (BOX_DTYPE, rank order) on the GPU."""
    b = np.ascontiguousarray(boxes, dtype=BOX_DTYPE)
    out = np.zeros(max(len(b), 1), dtype=BOX_DTYPE)
    n = C.c_int32(0)
    _chk(load().rtcc_nms(_ptr(b) if len(b) else None, len(b), iou, _ptr(out), C.byref(n)), "rtcc_nms")
    return out[:n.value]


def rtcc_get_pillars(ctx, agent: int, grid_h: int, grid_w: int, max_pillars: int) -> dict:
    c2p = np.empty(grid_h * grid_w, dtype=np.int32)
    pc = np.empty(max_pillars, dtype=np.int32)
    cnt = np.empty(max_pillars, dtype=np.int32)
    st = np.empty(8, dtype=np.int32)
    _chk(load().rtcc_get_pillars(ctx, agent, _ptr(c2p), _ptr(pc), _ptr(cnt), _ptr(st)),
         "rtcc_get_pillars")
    return {"cell2pillar": c2p, "pillar_cell": pc, "count": cnt, "n_points": int(st[0]),
            "n_in_range": int(st[1]), "n_pillars": int(st[2]), "n_kept": int(st[3]),
            "drop_range": int(st[4]), "drop_pcap": int(st[5]), "drop_ncap": int(st[6])}


def rtcc_get_tensor(ctx, agent: int, which: int) -> np.ndarray:
    """Raw 16-bit tensor as uint16 (reinterpret per the config's dtype)."""
    lib = load()
    n = C.c_size_t(0)
    _chk(lib.rtcc_get_tensor(ctx, agent, which, None, 0, C.byref(n)), "rtcc_get_tensor")
    out = np.empty(n.value, dtype=np.uint16)
    _chk(lib.rtcc_get_tensor(ctx, agent, which, _ptr(out), out.size, C.byref(n)), "rtcc_get_tensor")
    return out


def rtcc_status_str(s: int) -> str:
    return load().rtcc_status_str(s).decode()


def rtcc_now_ms() -> float:
    return load().rtcc_now_ms()


def rtcc_kernels_per_frame(ctx, n_present: int) -> int:
    return load().rtcc_kernels_per_frame(ctx, n_present)


SCHED_MAXRATE, SCHED_ROUNDROBIN, SCHED_MAXWEIGHT, SCHED_EARLIEST, SCHED_WEIGHTED = range(5)


def rtcc_uplink_simulate(payload_bits, first_slot, rates: np.ndarray, slot_s: float, policy: int,
                         weight=None):
    """Completion slots of one frame's uploads (see rtcc.h); rates [T][K][F]
    bit/s.  Returns (completion slots int32 [K], 0 = not within T; slots used)."""
    r = np.ascontiguousarray(rates, dtype=np.float64)
    T, K, F = r.shape
    b = np.ascontiguousarray(payload_bits, dtype=np.float64)
    l = np.ascontiguousarray(first_slot, dtype=np.int32)
    wt = None if weight is None else np.ascontiguousarray(weight, dtype=np.float64)
    out = np.zeros(K, dtype=np.int32)
    used = C.c_int32(0)
    _chk(load().rtcc_uplink_simulate(K, F, T, _ptr(b), _ptr(l), _ptr(r), float(slot_s), int(policy),
                                     None if wt is None else _ptr(wt), _ptr(out), C.byref(used)),
         "rtcc_uplink_simulate")
    return out, used.value


def rtcc_plan_conv(kind: int, cin: int, cout: int, out_w: int, out_h: int, grid: int,
                   n_batch: int) -> dict:
    """The backbone's tile choice for one 3x3 conv layer (see rtcc.h)."""
    p = rtcc_conv_plan()
    _chk(load().rtcc_plan_conv(int(kind), int(cin), int(cout), int(out_w), int(out_h), int(grid),
                               int(n_batch), C.byref(p)), "rtcc_plan_conv")
    return {f: int(getattr(p, f)) for f, _ in rtcc_conv_plan._fields_}


def rtcc_test_unreachable_wait(ctx) -> int:
    """Arm the wait-limit test hook for the next frame (see rtcc.h)."""
    return load().rtcc_test_unreachable_wait(ctx)


def rtcc_pillarise_noalloc(cfg: rtcc_model_config, d_points: int, n_points: int, d_pfn_w: int,
                           d_pfn_b: int, d_cell2pillar: int, d_pillar_cell: int, d_count: int,
                           d_stats: int, d_image: int, stream: int = 0) -> int:
    """Allocation-free pillarise/PFN/scatter; every d_* is a device address."""
    return load().rtcc_pillarise_noalloc(C.byref(cfg), d_points, n_points, d_pfn_w, d_pfn_b,
                                         d_cell2pillar, d_pillar_cell, d_count, d_stats,
                                         d_image, stream or None)


# --------------------------------------------------------------------------
# controller API
# --------------------------------------------------------------------------

def rtcc_ctrl_create(n_agents: int, cap_points: int, attn_ego: bool = False):
    out = _ctrl_p()
    _chk(load().rtcc_ctrl_create(n_agents, cap_points, int(attn_ego), C.byref(out)),
         "rtcc_ctrl_create")
    return out


def rtcc_ctrl_destroy(c) -> None:
    load().rtcc_ctrl_destroy(c)


def rtcc_ctrl_set_mode(c, mode: int) -> int:
    return load().rtcc_ctrl_set_mode(c, mode)


def rtcc_ctrl_begin(c, frame_id: int, t0_ms: float) -> int:
    return load().rtcc_ctrl_begin(c, frame_id, t0_ms)


def rtcc_ctrl_complete(c, agent: int, payload_nonnull: bool, n_points: int, t_ms: float):
    """Returns (status, released agents in dispatch order)."""
    rel = (C.c_int32 * MAX_AGENTS)()
    nrel = C.c_int32(0)
    payload = C.c_void_p(1) if payload_nonnull else None
    s = load().rtcc_ctrl_complete(c, agent, payload, n_points, t_ms, rel, C.byref(nrel))
    return s, [rel[i] for i in range(nrel.value)]


def rtcc_ctrl_absent(c, agent: int, t_ms: float):
    rel = (C.c_int32 * MAX_AGENTS)()
    nrel = C.c_int32(0)
    s = load().rtcc_ctrl_absent(c, agent, t_ms, rel, C.byref(nrel))
    return s, [rel[i] for i in range(nrel.value)]


def rtcc_ctrl_mark(c, agent: int, state: int) -> int:
    return load().rtcc_ctrl_mark(c, agent, state)


def rtcc_ctrl_abort(c) -> int:
    return load().rtcc_ctrl_abort(c)


def rtcc_ctrl_join_ready(c) -> bool:
    return bool(load().rtcc_ctrl_join_ready(c))


def rtcc_ctrl_state(c, agent: int):
    st = C.c_int32()
    r = C.c_double()
    s = load().rtcc_ctrl_state(c, agent, C.byref(st), C.byref(r))
    return s, st.value, (None if math.isnan(r.value) else r.value)


def rtcc_ctrl_end(c) -> int:
    return load().rtcc_ctrl_end(c)

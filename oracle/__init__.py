"""CPU oracle for the RTCC cooperative-perception path.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The product path
(the CUDA library and its Python binding) never calls it and shares no code
with it; the two meet only through the seeded generators in ``synth``.

* :mod:`oracle.forward` -- the plain forward pass of the fork-join detector
  (pillarisation, pillar feature net, BEV scatter, conv backbone with deconv
  neck, cross-agent fusion, 1x1 head, anchor decode), in float64 with an
  optional storage-rounding mode that rounds weights and every stored
  activation to the GPU's 16-bit storage type.
* :mod:`oracle.nms` -- rotated bird's-eye-view IoU (Sutherland-Hodgman
  clipping, shoelace area) and greedy NMS, the last step of the detections
  that end T^det (Sec. V-A-3).
* :mod:`oracle.schedule` -- the single-stream execution model of RTCC and
  Barrier (Sec. III-B/C, Eqs. 17-19, the second phase of Algorithm 1) and the
  slot-level OFDMA uplink with causal schedulers (Eqs. 1-6, 13-16, 20-21, the
  first phase of Algorithm 1).

Every function says which passage it follows.  Functions without an
independent pin say "parity unpinned" in their docstring.
"""

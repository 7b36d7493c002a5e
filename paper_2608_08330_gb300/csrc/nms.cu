// Rotated bird's-eye-view non-maximum suppression of the decoded boxes: the
// last step of the detections that end the complete-detection latency T^det
// (box decoding, score thresholding and rotated NMS, Sec. V-A-3).
//
// Greedy rule: in the decode's rank order (score descending, anchor index
// ascending), a box is kept iff its IoU with every box kept before it is at
// most the threshold.  Boxes are rectangles in the x-y plane: centre (x, y),
// length l along (cos yaw, sin yaw), width w along (-sin yaw, cos yaw).  The
// intersection is one rectangle clipped by the other's four half-planes
// (Sutherland-Hodgman), its area by the shoelace formula.
//
// One launch, two phases:
//   1. every block takes warps of pair tests: warp (i, word) tests box i
//      against boxes j = 32 word + lane (j > i) and a ballot gives the word of
//      the suppression bitmask (bit set = IoU > threshold), stored in global
//      memory.  An upper bound of the intersection (bounding-box overlaps)
//      settles most pairs before the clip;
//   2. the last block to finish (ticket counter) loads the bitmask into
//      shared memory and one warp resolves the greedy order 32 boxes at a
//      time: within a chunk, rounds of warp OR-reductions decide every row
//      whose possible suppressors are all decided (the only sequential part,
//      as long as the longest suppression chain), then each lane ORs the
//      kept rows of the chunk into its word of the removed set.  The kept boxes are staged in
//      rank order and copied into the pinned host result block; the done
//      flag follows a system-scope fence.
#include <cmath>

#include "common.cuh"
#include "kernels.h"
#include "rtcc.h"

namespace rtcc {

namespace {

constexpr int kNmsThreads = 256;
constexpr int kNmsWarps = kNmsThreads / 32;
constexpr int kNmsWords = kDecodeKeep / 32;     // mask words per row at most

// One box: centre, heading (cos, sin) and half extents.
struct RRect {
  float x, y, c, s, hl, hw;
};

__device__ __forceinline__ RRect rrect(const rtcc_box* b) {
  RRect r;
  r.x = b->x;
  r.y = b->y;
  sincosf(b->yaw, &r.s, &r.c);
  r.hl = 0.5f * b->l;
  r.hw = 0.5f * b->w;
  return r;
}

// Signed distance of (u, v) to side `side` of the box [-hl, hl] x [-hw, hw]
// (0: u <= hl, 1: v <= hw, 2: u >= -hl, 3: v >= -hw), positive inside.
__device__ __forceinline__ float side_dist(int side, float u, float v, float hl, float hw) {
  return side == 0 ? hl - u : side == 1 ? hw - v : side == 2 ? u + hl : v + hw;
}

// Area of the intersection of two rectangles, in B's frame (u along B's
// length, v along its width): A's corners clipped by B's four sides, one
// Sutherland-Hodgman pass per side.  The polygons live in this thread's
// column of shared memory (`col`, stride kNmsThreads: x and y of two
// ping-pong polygons of up to 8 vertices -- a convex polygon clipped by the
// 4 sides of a box has at most 8), so the loops stay short and indexed
// register arrays (local memory) are avoided; a vertex that rounding would
// add beyond 8 is dropped.
__device__ float intersection_area(const RRect& A, const RRect& B, float* col) {
  auto at = [&](int a, int k) -> float& { return col[(a * 8 + k) * kNmsThreads]; };
  const float dx = A.x - B.x, dy = A.y - B.y;
  const float uc = B.c * dx + B.s * dy, vc = -B.s * dx + B.c * dy;    // A's centre
  const float ct = A.c * B.c + A.s * B.s, st = A.s * B.c - A.c * B.s;  // A's heading
#pragma unroll
  for (int k = 0; k < 4; ++k) {                  // counter-clockwise corners of A
    const float u = (k == 0 || k == 3) ? A.hl : -A.hl;
    const float v = (k < 2) ? A.hw : -A.hw;
    at(0, k) = uc + ct * u - st * v;
    at(1, k) = vc + st * u + ct * v;
  }
  int n = 4, src = 0;
#pragma unroll 1
  for (int side = 0; side < 4; ++side) {
    const int dst = 2 - src;
    int m = 0;
    const float x0 = at(src, 0), y0 = at(src + 1, 0);
    const float d0 = side_dist(side, x0, y0, B.hl, B.hw);
    float xp = x0, yp = y0, dp = d0;
#pragma unroll 1
    for (int k = 0; k < n; ++k) {                // edge (k, k + 1)
      const bool last = k + 1 == n;
      const float xq = last ? x0 : at(src, k + 1), yq = last ? y0 : at(src + 1, k + 1);
      const float dq = last ? d0 : side_dist(side, xq, yq, B.hl, B.hw);
      if (dp >= 0.0f && m < 8) {
        at(dst, m) = xp;
        at(dst + 1, m) = yp;
        ++m;
      }
      if ((dp >= 0.0f) != (dq >= 0.0f) && m < 8) {
        const float t = dp / (dp - dq);
        at(dst, m) = xp + t * (xq - xp);
        at(dst + 1, m) = yp + t * (yq - yp);
        ++m;
      }
      xp = xq;
      yp = yq;
      dp = dq;
    }
    if (m == 0) return 0.0f;
    n = m;
    src = dst;
  }
  float s = 0.0f, xp = at(src, n - 1), yp = at(src + 1, n - 1);
#pragma unroll 1
  for (int k = 0; k < n; ++k) {                  // shoelace
    const float x = at(src, k), y = at(src + 1, k);
    s += xp * y - x * yp;
    xp = x;
    yp = y;
  }
  return fmaxf(0.5f * s, 0.0f);
}

// Area of the overlap of box B with the bounding box, in B's frame, of a
// box of half extents (hl, hw) centred at (uc, vc) and turned by (ct, st)
// relative to B: an upper bound of their intersection area (0: separated
// along one of B's axes).
__device__ __forceinline__ float aabb_bound(float uc, float vc, float ct, float st, float hl, float hw,
                                            const RRect& B) {
  const float eu = fabsf(ct) * hl + fabsf(st) * hw, ev = fabsf(st) * hl + fabsf(ct) * hw;
  const float ox = fminf(uc + eu, B.hl) - fmaxf(uc - eu, -B.hl);
  const float oy = fminf(vc + ev, B.hw) - fmaxf(vc - ev, -B.hw);
  return fmaxf(ox, 0.0f) * fmaxf(oy, 0.0f);
}

// IoU(i, j) > thr, compared as inter > thr * union (union > 0 for boxes of
// positive area).  The intersection is clipped only when an upper bound of it
// (the smaller of the two bounding-box overlaps, each box in the other's
// frame) leaves IoU > thr possible: IoU grows with the intersection, so
// bound / (a + b - bound) <= thr decides "no".  (A bound of 0 also settles
// every separated pair.)
__device__ __forceinline__ bool suppresses(const RRect& A, float area_a, const RRect& B, float area_b,
                                           float thr, float* col) {
  const float dx = A.x - B.x, dy = A.y - B.y;
  const float ct = A.c * B.c + A.s * B.s, st = A.s * B.c - A.c * B.s;     // A relative to B
  const float ub_a = aabb_bound(B.c * dx + B.s * dy, -B.s * dx + B.c * dy, ct, st, A.hl, A.hw, B);
  const float ub_b = aabb_bound(-(A.c * dx + A.s * dy), A.s * dx - A.c * dy, ct, -st, B.hl, B.hw, A);
  const float ub = fminf(ub_a, ub_b);
  if (ub <= thr * (area_a + area_b - ub)) return false;
  const float inter = intersection_area(A, B, col);
  return inter > thr * (area_a + area_b - inter);
}

__global__ void __launch_bounds__(kNmsThreads) k_nms(const rtcc_box* in, const int* n_in, uint32_t* mask,
                                                     unsigned* ticket, float thr, const int* err,
                                                     DetResultHeader* hdr, rtcc_box* out,
                                                     volatile int* done) {
  // phase 1: per-thread polygon slots; phase 2: the bitmask, then staged boxes
  __shared__ __align__(16) uint32_t sm[kDecodeKeep * kNmsWords];
  __shared__ uint32_t keepw[kNmsWords];
  __shared__ int pre[kNmsWords];
  __shared__ int s_last, s_nk;
  static_assert(sizeof(rtcc_box) * kDecodeKeep <= sizeof(uint32_t) * kDecodeKeep * kNmsWords,
                "the kept boxes are staged in the bitmask's shared memory");
  static_assert(kDecodeKeep <= 2 * kNmsThreads, "a thread stages at most two boxes");
  static_assert(32 * kNmsThreads <= kDecodeKeep * kNmsWords, "32 polygon slots per thread");
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  pdl_trigger();
  pdl_wait();                                   // the decoded boxes are the decode's output
  const int n = *n_in;
  const int W = (n + 31) >> 5;                  // row stride of the bitmask, in words

  // ---- 1. pair tests: warp (row i, word wd) for the words from row i's own
  // 32-box chunk on (the scan reads no others), enumerated chunk by chunk so
  // that every warp of the grid takes at most one when they suffice ----
  int tasks = 0;
  for (int c = 0; c < W; ++c) tasks += min(32, n - 32 * c) * (W - c);
  for (int t = blockIdx.x * kNmsWarps + warp; t < tasks; t += gridDim.x * kNmsWarps) {
    int c = 0, u = t;
    for (; c < W; ++c) {                          // the chunk of task t
      const int tc = min(32, n - 32 * c) * (W - c);
      if (u < tc) break;
      u -= tc;
    }
    const int i = 32 * c + u / (W - c), wd = c + u % (W - c);
    const int j = 32 * wd + lane;
    bool s = false;
    if (j > i && j < n) {
      const RRect A = rrect(in + i), B = rrect(in + j);
      s = suppresses(A, in[i].l * in[i].w, B, in[j].l * in[j].w, thr, reinterpret_cast<float*>(sm) + tid);
    }
    const unsigned m = __ballot_sync(0xFFFFFFFFu, s);
    if (lane == 0) mask[i * W + wd] = m;
  }
  __syncthreads();
  if (tid == 0) {
    __threadfence();                            // this block's words before its ticket
    s_last = atomicAdd(ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;

  // ---- 2. the last block: greedy resolution over the bitmask -------------
  __threadfence();
  if (tid == 0) *ticket = 0;                    // ready for the next frame
  // the boxes this thread stages (ranks tid, tid + 256), fetched while the
  // bitmask is resolved
  rtcc_box b0{}, b1{};
  if (tid < n) b0 = in[tid];
  if (tid + kNmsThreads < n) b1 = in[tid + kNmsThreads];
  {
    // rows are contiguous: 16-byte loads, all issued before use (the words
    // left of a row's own chunk were not written this frame and are never
    // read)
    const int nw = n * W;
    const uint4* m4 = reinterpret_cast<const uint4*>(mask);
    uint4* s4 = reinterpret_cast<uint4*>(sm);
#pragma unroll 4
    for (int q = tid; q < (nw >> 2); q += kNmsThreads) s4[q] = __ldcg(m4 + q);
    for (int t = (nw & ~3) + tid; t < nw; t += kNmsThreads) sm[t] = __ldcg(mask + t);
  }
  __syncthreads();
  if (warp == 0) {
    // Warp 0 alone, no block barriers.  Lane l holds word l of the removed
    // set (rows suppressed by kept rows of earlier chunks) and, once chunk l
    // is resolved, its keep word.  Chunk c (rows 32c + b): lane b holds row
    // b's own-chunk word (the later rows of the chunk it suppresses).  In
    // rounds, a row none of whose possible suppressors is still undecided
    // (OR of the undecided rows' words) is decided: kept iff no kept row
    // suppresses it (OR of the kept rows' words).  The lowest undecided row
    // is always decidable, so at most 32 rounds, usually a few (the longest
    // suppression chain).  Then lane l > c ORs the kept rows' word l into its
    // removed word.
    uint32_t rem_l = 0u, keep_l = 0u;
    for (int c = 0; c < W; ++c) {
      uint32_t r = __shfl_sync(0xFFFFFFFFu, rem_l, c);
      const int left = n - 32 * c;
      if (left < 32) r |= ~0u << left;           // no rows beyond n
      const uint32_t* rows = sm + (32 * c) * W;
      const uint32_t m = lane < left ? rows[lane * W + c] : 0u;
      uint32_t und = ~r, kept = 0u, sup = 0u;
      if (__ballot_sync(0xFFFFFFFFu, m != 0u) == 0u) {
        kept = und;                              // no row of the chunk suppresses another
        und = 0u;
      }
      for (int round = 0; round < 32 && und; ++round) {
        // rows still undecided may suppress later ones: those wait
        const uint32_t pot = __reduce_or_sync(0xFFFFFFFFu, ((und >> lane) & 1u) ? m : 0u);
        const bool ready = ((und >> lane) & 1u) && ((pot >> lane) & 1u) == 0u;
        const bool k = ready && ((sup >> lane) & 1u) == 0u;
        und &= ~__ballot_sync(0xFFFFFFFFu, ready);
        kept |= __ballot_sync(0xFFFFFFFFu, k);
        sup |= __reduce_or_sync(0xFFFFFFFFu, k ? m : 0u);
      }
      if (lane == c) keep_l = kept;
      if (lane > c && lane < W) {
        // 32 independent loads, masked rather than branched around (rows
        // at or beyond n are in bounds of the array and never kept)
        uint32_t v = 0u;
#pragma unroll
        for (int b = 0; b < 32; ++b) v |= rows[b * W + lane] & (0u - ((kept >> b) & 1u));
        rem_l |= v;
      }
    }
    // kept count per chunk -> exclusive prefix (the staging slot of a chunk's
    // first kept box)
    const int cnt = lane < W ? __popc(keep_l) : 0;
    int inc = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xFFFFFFFFu, inc, o);
      if (lane >= o) inc += y;
    }
    if (lane < W) {
      keepw[lane] = keep_l;
      pre[lane] = inc - cnt;
    }
    if (lane == 31) s_nk = inc;
  }
  __syncthreads();
  const int nk = s_nk;
  rtcc_box* st = reinterpret_cast<rtcc_box*>(sm);   // the bitmask is no longer read
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int i = tid + h * kNmsThreads;
    if (i < n) {
      const uint32_t kw = keepw[i >> 5];
      const uint32_t bit = 1u << (i & 31);
      if (kw & bit) st[pre[i >> 5] + __popc(kw & (bit - 1u))] = h ? b1 : b0;
    }
  }
  __syncthreads();
  if (tid == 0) {
    hdr->n_boxes = nk;
    hdr->err = *err;
  }
  const int nbytes = nk * (int)sizeof(rtcc_box);
  const uint4* src = reinterpret_cast<const uint4*>(sm);
  uint4* dst = reinterpret_cast<uint4*>(out);
  for (int i = tid; i < nbytes / 16; i += kNmsThreads) dst[i] = src[i];
  for (int i = (nbytes / 16) * 4 + tid; i < nbytes / 4; i += kNmsThreads)
    reinterpret_cast<uint32_t*>(out)[i] = sm[i];
  __threadfence_system();                       // this thread's writes, system-wide
  __syncthreads();
  if (tid == 0) *done = 1;
}

}  // namespace

size_t nms_mask_words(int max_boxes) { return (size_t)max_boxes * ((max_boxes + 31) / 32); }

cudaError_t launch_nms(const NmsArgs& a, cudaStream_t st) {
  if (a.max_boxes < 1 || a.max_boxes > kDecodeKeep || !(a.iou >= 0.0f && a.iou <= 1.0f) || !a.in ||
      !a.n_in || !a.mask || !a.ticket || !a.err || !a.out || !a.done)
    return cudaErrorInvalidValue;
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  // enough warps for the pair tests of a full list, at most one block per SM
  const int tasks = a.max_boxes * ((a.max_boxes + 31) / 32);
  int grid = (tasks + kNmsWarps - 1) / kNmsWarps;
  if (grid > sms) grid = sms;
  if (grid < 1) grid = 1;
  DetResultHeader* hdr = static_cast<DetResultHeader*>(a.out);
  rtcc_box* boxes = reinterpret_cast<rtcc_box*>(hdr + 1);
  return launch_pdl(k_nms, dim3(grid), dim3(kNmsThreads), 0, st, a.in, a.n_in, a.mask, a.ticket, a.iou,
                    a.err, hdr, boxes, a.done);
}

}  // namespace rtcc

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
//      memory.  A circumscribed-circle test rejects far pairs before the clip;
//   2. the last block to finish (ticket counter) loads the upper-triangle
//      bitmask into shared memory and resolves the greedy order 32 boxes at a
//      time: one thread walks the chunk's own word bit by bit (the only
//      sequential part), then each word of the removed set ORs in the rows of
//      the chunk's kept boxes with one warp reduction.  The kept boxes are
//      staged in rank order and copied into the pinned host result block; the
//      done flag follows a system-scope fence.
#include <cmath>

#include "common.cuh"
#include "kernels.h"
#include "rtcc.h"

namespace rtcc {

namespace {

constexpr int kNmsThreads = 256;
constexpr int kNmsWarps = kNmsThreads / 32;
constexpr int kNmsWords = kDecodeKeep / 32;     // mask words per row at most
constexpr int kPolyMax = 16;                     // vertex slots of a clipped polygon

// A box relative to a reference centre: centre offset, heading, half extents.
struct RRect {
  float x, y, c, s, hl, hw;
};

__device__ __forceinline__ RRect rrect(const rtcc_box* b, float ox, float oy) {
  RRect r;
  r.x = b->x - ox;
  r.y = b->y - oy;
  sincosf(b->yaw, &r.s, &r.c);
  r.hl = 0.5f * b->l;
  r.hw = 0.5f * b->w;
  return r;
}

// Corner k (counter-clockwise: front-left, rear-left, rear-right, front-right).
__device__ __forceinline__ void corner(const RRect& r, int k, float* x, float* y) {
  const float u = (k == 0 || k == 3) ? r.hl : -r.hl;
  const float v = (k < 2) ? r.hw : -r.hw;
  *x = r.x + r.c * u - r.s * v;
  *y = r.y + r.s * u + r.c * v;
}

// Area of the intersection of two rectangles: A's corners clipped by the
// half-plane on the left of each directed edge of B.  A clip can add vertices
// only where the boundary crosses the edge line; the slot count is capped so
// that no write leaves the arrays even for rounding-made sign patterns.
__device__ float intersection_area(const RRect& A, const RRect& B) {
  float px[kPolyMax], py[kPolyMax], qx[kPolyMax], qy[kPolyMax];
  int n = 4;
#pragma unroll
  for (int k = 0; k < 4; ++k) corner(A, k, &px[k], &py[k]);
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    float ax, ay, bx, by;
    corner(B, e, &ax, &ay);
    corner(B, (e + 1) & 3, &bx, &by);
    const float ex = bx - ax, ey = by - ay;
    int m = 0;
    for (int k = 0; k < n; ++k) {
      const int k1 = (k + 1 == n) ? 0 : k + 1;
      const float sp = ex * (py[k] - ay) - ey * (px[k] - ax);
      const float sq = ex * (py[k1] - ay) - ey * (px[k1] - ax);
      const bool in_p = sp >= 0.0f, in_q = sq >= 0.0f;
      if (in_p && m < kPolyMax) {
        qx[m] = px[k];
        qy[m] = py[k];
        ++m;
      }
      if (in_p != in_q && m < kPolyMax) {
        const float t = sp / (sp - sq);
        qx[m] = px[k] + t * (px[k1] - px[k]);
        qy[m] = py[k] + t * (py[k1] - py[k]);
        ++m;
      }
    }
    if (m == 0) return 0.0f;
    n = m;
    for (int k = 0; k < n; ++k) {
      px[k] = qx[k];
      py[k] = qy[k];
    }
  }
  float s = 0.0f;
  for (int k = 0; k < n; ++k) {
    const int k1 = (k + 1 == n) ? 0 : k + 1;
    s += px[k] * py[k1] - px[k1] * py[k];
  }
  return fmaxf(0.5f * s, 0.0f);
}

// IoU(i, j) > thr, compared as inter > thr * union (union > 0 for boxes of
// positive area); coordinates relative to box i's centre.
__device__ __forceinline__ bool suppresses(const rtcc_box* bi, const rtcc_box* bj, float thr) {
  const RRect A = rrect(bi, bi->x, bi->y);
  const RRect B = rrect(bj, bi->x, bi->y);
  const float ra = sqrtf(A.hl * A.hl + A.hw * A.hw), rb = sqrtf(B.hl * B.hl + B.hw * B.hw);
  const float d2 = B.x * B.x + B.y * B.y;
  const float rr = (ra + rb) * 1.0001f;
  if (d2 > rr * rr) return 0.0f > thr;                    // disjoint: IoU = 0
  const float inter = intersection_area(A, B);
  const float uni = bi->l * bi->w + bj->l * bj->w - inter;
  return inter > thr * uni;
}

__global__ void __launch_bounds__(kNmsThreads) k_nms(const rtcc_box* in, const int* n_in, uint32_t* mask,
                                                     unsigned* ticket, float thr, const int* err,
                                                     DetResultHeader* hdr, rtcc_box* out,
                                                     volatile int* done) {
  __shared__ __align__(16) uint32_t sm[kDecodeKeep * kNmsWords];   // bitmask; then staged boxes
  __shared__ uint32_t removed[kNmsWords], keepw[kNmsWords];
  __shared__ int pre[kNmsWords];
  __shared__ int s_last, s_nk;
  static_assert(sizeof(rtcc_box) * kDecodeKeep <= sizeof(uint32_t) * kDecodeKeep * kNmsWords,
                "the kept boxes are staged in the bitmask's shared memory");
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  pdl_trigger();
  pdl_wait();                                   // the decoded boxes are the decode's output
  const int n = *n_in;
  const int W = (n + 31) >> 5;                  // row stride of the bitmask, in words

  // ---- 1. pair tests, one warp per (row i, word wd) above the diagonal ----
  for (int t = blockIdx.x * kNmsWarps + warp; t < n * W; t += gridDim.x * kNmsWarps) {
    const int i = t / W, wd = t - i * W;
    if (32 * wd + 31 <= i) continue;            // no j > i in this word (warp-uniform)
    const int j = 32 * wd + lane;
    const bool s = j > i && j < n && suppresses(in + i, in + j, thr);
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
  for (int t = tid; t < n * W; t += kNmsThreads) {
    const int i = t / W, wd = t - i * W;
    sm[t] = (wd >= (i >> 5)) ? __ldcg(mask + t) : 0u;
  }
  if (tid < kNmsWords) removed[tid] = 0u;
  __syncthreads();
  for (int c = 0; c < W; ++c) {
    if (tid == 0) {
      // rows 32c .. 32c+31: bit b of their own word marks the later rows of
      // the chunk that row b suppresses
      uint32_t mm[32];
#pragma unroll
      for (int b = 0; b < 32; ++b) mm[b] = (32 * c + b < n) ? sm[(32 * c + b) * W + c] : 0u;
      uint32_t r = removed[c];
      const int rem = n - 32 * c;
      if (rem < 32) r |= ~0u << rem;            // no rows beyond n
      uint32_t keep = 0u;
#pragma unroll
      for (int b = 0; b < 32; ++b) {
        const bool k = ((r >> b) & 1u) == 0u;
        keep |= k ? (1u << b) : 0u;
        r |= k ? mm[b] : 0u;
      }
      keepw[c] = keep;
    }
    __syncthreads();
    const uint32_t keep = keepw[c];
    for (int wd = c + 1 + warp; wd < W; wd += kNmsWarps) {
      const uint32_t v = ((keep >> lane) & 1u) ? sm[(32 * c + lane) * W + wd] : 0u;
      const uint32_t o = __reduce_or_sync(0xFFFFFFFFu, v);
      if (lane == 0) removed[wd] |= o;
    }
    __syncthreads();
  }
  if (tid == 0) {
    int s = 0;
    for (int c = 0; c < W; ++c) {
      pre[c] = s;
      s += __popc(keepw[c]);
    }
    s_nk = s;
  }
  __syncthreads();
  const int nk = s_nk;
  rtcc_box* st = reinterpret_cast<rtcc_box*>(sm);   // the bitmask is no longer read
  for (int i = tid; i < n; i += kNmsThreads) {
    const uint32_t kw = keepw[i >> 5];
    const uint32_t bit = 1u << (i & 31);
    if (kw & bit) st[pre[i >> 5] + __popc(kw & (bit - 1u))] = in[i];
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

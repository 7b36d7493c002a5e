// Anchor decode, threshold and deterministic top-K of the head output (the
// detection post-processing that ends the complete-detection latency, Sec.
// V-A-3).  Rotated NMS is not part of this step.
//
// Order: class logit descending, then anchor index ascending; threshold on the
// logit (score = sigmoid(logit) is monotone), so the selection is an exact
// function of the head output.  The fusion kernel leaves one 32-bit key per
// anchor whose ascending order is descending logit order (0xFFFFFFFF below the
// threshold).  One block selects the K = min(max_boxes, #valid) smallest
// (key, index) pairs:
//   1. radix select on the key in three levels (12, 10, 10 bits) finds the
//      exact key T of the K-th pair and the count c of keys below T (the
//      fusion kernel builds the first level's histogram with global atomics;
//      the block builds the others in shared memory);
//   2. one pass collects the c keys below T; an ordered pass (each thread owns
//      a contiguous range of anchors, a block scan ranks its ties) adds the
//      K - c keys equal to T with the smallest indices;
//   3. the K pairs are sorted (bitonic, K <= 512) and decoded into boxes.
#include <cmath>

#include "common.cuh"
#include "kernels.h"
#include "rtcc.h"

namespace rtcc {

namespace {

constexpr uint32_t kInvalid = 0xFFFFFFFFu;
constexpr int kThreads = 1024;
constexpr int kMaxBins = 4096;

struct AnchorGeo {
  float x_min, y_min, sx, sy;       // cell size in metres
  int feat_w, anchors;
  float la, wa, ha, za, da;
};

// Exclusive block scan of one int per thread (1024 threads); *total = sum.
__device__ int block_scan_excl(int v, int* total) {
  __shared__ int ws[32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  int inc = v;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int o = __shfl_up_sync(0xFFFFFFFFu, inc, d);
    if (lane >= d) inc += o;
  }
  if (lane == 31) ws[wid] = inc;
  __syncthreads();
  if (wid == 0) {
    const int w = ws[lane];
    int winc = w;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int o = __shfl_up_sync(0xFFFFFFFFu, winc, d);
      if (lane >= d) winc += o;
    }
    ws[lane] = winc - w;
    if (lane == 31) *total = winc;
  }
  __syncthreads();
  const int r = ws[wid] + inc - v;
  __syncthreads();
  return r;
}

// The thread's contiguous chunk of keys, 16 bytes at a time (the key array is
// padded with invalid keys to kThreads * chunk entries).  f(key, index).
template <typename F>
__device__ __forceinline__ void for_chunk(const uint32_t* __restrict__ keys, int lo, int chunk4,
                                          F f) {
  const uint4* v = reinterpret_cast<const uint4*>(keys + lo);
  constexpr int B = 8;                                   // loads in flight per thread
  for (int base = 0; base < chunk4; base += B) {
    uint4 r[B];
#pragma unroll
    for (int j = 0; j < B; ++j)
      if (base + j < chunk4) r[j] = v[base + j];
#pragma unroll
    for (int j = 0; j < B; ++j) {
      if (base + j < chunk4) {
        const int i = lo + 4 * (base + j);
        f(r[j].x, i);
        f(r[j].y, i + 1);
        f(r[j].z, i + 2);
        f(r[j].w, i + 3);
      }
    }
  }
}

__global__ void __launch_bounds__(kThreads, 1)
k_decode_select(const uint32_t* __restrict__ keys, uint32_t* __restrict__ hist0,
                const float* __restrict__ head, int chunk4, int max_boxes, AnchorGeo g,
                const int* __restrict__ err, DetResultHeader* __restrict__ hdr,
                rtcc_box* __restrict__ boxes) {
  __shared__ int hist[kMaxBins];
  __shared__ unsigned long long sel[kDecodeKeep];
  __shared__ int s_total, s_bin, s_below, s_nsel;
  const int tid = threadIdx.x;
  const int lo = tid * chunk4 * 4;
  pdl_trigger();
  pdl_wait();

  // ---- 1. radix select: exact threshold key T and c = #keys < T ----------
  // level 0 (top 12 bits) was histogrammed by the fusion kernel; the others
  // (10 + 10 bits) are built here over the keys that match the prefix so far.
  uint32_t prefix = 0, pmask = 0;
  int below = 0, need = 0;
  const int shifts[3] = {20, 10, 0};
  const int widths[3] = {12, 10, 10};
  for (int lv = 0; lv < 3; ++lv) {
    const int nb = 1 << widths[lv];
    if (lv == 0) {
      for (int i = tid; i < nb; i += kThreads) {
        hist[i] = (int)hist0[i];
        hist0[i] = 0;                                  // ready for the next frame
      }
    } else {
      for (int i = tid; i < nb; i += kThreads) hist[i] = 0;
      __syncthreads();
      const int sh = shifts[lv];
      for_chunk(keys, lo, chunk4, [&](uint32_t k, int) {
        if (k != kInvalid && (k & pmask) == prefix) atomicAdd(&hist[(k >> sh) & (nb - 1)], 1);
      });
    }
    __syncthreads();
    // each thread owns a contiguous range of bins
    const int per = (nb + kThreads - 1) / kThreads;
    int mine = 0;
    for (int j = 0; j < per; ++j) {
      const int b = tid * per + j;
      if (b < nb) mine += hist[b];
    }
    int run = block_scan_excl(mine, &s_total);
    const int total = s_total;
    if (lv == 0) need = total < max_boxes ? total : max_boxes;   // K
    if (need == 0) break;
    // the bin where the cumulative count (offset by `below`) reaches need
    for (int j = 0; j < per; ++j) {
      const int b = tid * per + j;
      if (b < nb) {
        const int h = hist[b];
        if (below + run < need && below + run + h >= need) {
          s_bin = b;
          s_below = below + run;
        }
        run += h;
      }
    }
    __syncthreads();
    prefix |= static_cast<uint32_t>(s_bin) << shifts[lv];
    pmask |= static_cast<uint32_t>(nb - 1) << shifts[lv];
    below = s_below;
    __syncthreads();
  }
  if (tid == 0) {
    hdr->n_boxes = need;
    hdr->err = *err;
    s_nsel = 0;
  }
  if (need == 0) return;
  const uint32_t T = prefix;
  __syncthreads();

  // ---- 2. collect keys < T, then the (need - below) lowest-index ties ------
  int ties = 0;
  for_chunk(keys, lo, chunk4, [&](uint32_t k, int i) {
    if (k < T) {
      const int pos = atomicAdd(&s_nsel, 1);
      sel[pos] = (static_cast<unsigned long long>(k) << 32) | static_cast<unsigned>(i);
    } else if (k == T) {
      ++ties;
    }
  });
  int tie_base = block_scan_excl(ties, &s_total);
  const int take = need - below;
  if (ties > 0 && tie_base < take) {
    for_chunk(keys, lo, chunk4, [&](uint32_t k, int i) {
      if (k == T && tie_base < take) {
        sel[below + tie_base] = (static_cast<unsigned long long>(T) << 32) | static_cast<unsigned>(i);
        ++tie_base;
      }
    });
  }
  __syncthreads();

  // ---- 3. sort the K selected pairs and decode -----------------------------
  int P2 = 1;
  while (P2 < need) P2 <<= 1;
  for (int i = need + tid; i < P2; i += kThreads) sel[i] = ~0ull;
  __syncthreads();
  for (int k = 2; k <= P2; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = tid; i < P2; i += kThreads) {
        const int l = i ^ j;
        if (l > i) {
          const unsigned long long x = sel[i], y = sel[l];
          if ((x > y) == ((i & k) == 0)) {
            sel[i] = y;
            sel[l] = x;
          }
        }
      }
      __syncthreads();
    }
  }
  for (int r = tid; r < need; r += kThreads) {
    const int a = static_cast<int>(sel[r] & 0xFFFFFFFFull);
    const int cell = a / g.anchors, an = a - cell * g.anchors;
    const int ix = cell % g.feat_w, iy = cell / g.feat_w;
    const float* h = head + (size_t)cell * 16;
    const float cls = h[an];
    const float* rg = h + g.anchors + 7 * an;
    const float xa = g.x_min + ((float)ix + 0.5f) * g.sx;
    const float ya = g.y_min + ((float)iy + 0.5f) * g.sy;
    rtcc_box b;
    b.x = xa + rg[0] * g.da;
    b.y = ya + rg[1] * g.da;
    b.z = g.za + rg[2] * g.ha;
    b.l = g.la * expf(fminf(rg[3], 10.0f));
    b.w = g.wa * expf(fminf(rg[4], 10.0f));
    b.h = g.ha * expf(fminf(rg[5], 10.0f));
    b.yaw = (float)an * (3.14159265358979f / (float)g.anchors) + rg[6];
    b.score = 1.0f / (1.0f + expf(-cls));
    b.anchor = a;
    boxes[r] = b;
  }
}

}  // namespace

int decode_key_chunk4(int n_anchors) { return (n_anchors + 4 * kThreads - 1) / (4 * kThreads); }

cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t st) {
  const int n = a.feat_w * a.feat_h * a.anchors;
  if (a.max_boxes < 1 || a.max_boxes > kDecodeKeep) return cudaErrorInvalidValue;
  DetResultHeader* hdr = static_cast<DetResultHeader*>(a.out);
  rtcc_box* boxes = reinterpret_cast<rtcc_box*>(hdr + 1);
  AnchorGeo g;
  g.x_min = a.x_min;
  g.y_min = a.y_min;
  g.sx = (a.x_max - a.x_min) / (float)a.feat_w;
  g.sy = (a.y_max - a.y_min) / (float)a.feat_h;
  g.feat_w = a.feat_w;
  g.anchors = a.anchors;
  g.la = 3.9f;
  g.wa = 1.6f;
  g.ha = 1.56f;
  g.za = -1.0f;
  g.da = (float)std::sqrt(3.9 * 3.9 + 1.6 * 1.6);
  return launch_pdl(k_decode_select, dim3(1), dim3(kThreads), 0, st, a.keys, a.hist0, a.head,
                    decode_key_chunk4(n), a.max_boxes, g, a.err, hdr, boxes);
}

}  // namespace rtcc

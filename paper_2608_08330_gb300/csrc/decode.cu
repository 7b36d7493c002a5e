// Anchor decode, threshold and deterministic top-K of the head output (the
// detection post-processing that ends the complete-detection latency, Sec.
// V-A-3).  Rotated NMS is not part of this step.
//
// Order: class logit descending, then anchor index ascending; threshold on the
// logit (score = sigmoid(logit) is monotone), so the selection is an exact
// function of the head output.  The fusion kernel leaves one 32-bit key per
// anchor whose ascending order is descending logit order (0xFFFFFFFF below the
// threshold), and a histogram of the keys' top 12 bits.  One block selects the
// K = min(max_boxes, #valid) smallest (key, index) pairs:
//   1. a scan of the histogram finds the bin b0 that holds the K-th key and
//      the count c of keys in lower bins (c < K);
//   2. one coalesced pass over the keys puts the c keys of lower bins into the
//      selection and the keys of bin b0 into a shared-memory list;
//   3. both are sorted (bitonic, in lockstep) and the K - c smallest pairs of
//      bin b0 complete the selection, which is then already in order;
//   4. the K pairs are decoded into boxes.
// If bin b0 holds more keys than the list can take, a radix select refines
// the threshold over the next 10 + 10 key bits instead (two more passes), the
// keys below it are collected, and an ordered pass (each thread owns a
// contiguous range of anchors, a block scan ranks its ties) adds the
// lowest-index keys equal to it.
#include <cmath>

#include "common.cuh"
#include "kernels.h"
#include "rtcc.h"

namespace rtcc {

namespace {

constexpr uint32_t kInvalid = 0xFFFFFFFFu;
constexpr int kThreads = 1024;
constexpr int kMaxBins = 4096;
constexpr int kBndCap = 4096;                // keys of bin b0 held in shared memory

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

// Coalesced pass over the (padded) key array: thread t takes the 16-byte
// vectors t, t + kThreads, ...; f(key, index).
template <typename F>
__device__ __forceinline__ void for_strided(const uint32_t* __restrict__ keys, int n4, F f) {
  const uint4* v = reinterpret_cast<const uint4*>(keys);
  constexpr int B = 4;                                   // loads in flight per thread
  for (int base = threadIdx.x; base < n4; base += B * kThreads) {
    uint4 r[B];
#pragma unroll
    for (int j = 0; j < B; ++j)
      if (base + j * kThreads < n4) r[j] = v[base + j * kThreads];
#pragma unroll
    for (int j = 0; j < B; ++j) {
      const int q = base + j * kThreads;
      if (q < n4) {
        f(r[j].x, 4 * q);
        f(r[j].y, 4 * q + 1);
        f(r[j].z, 4 * q + 2);
        f(r[j].w, 4 * q + 3);
      }
    }
  }
}

__device__ __forceinline__ void cmp_swap(unsigned long long* a, int i, int l, int k) {
  const unsigned long long x = a[i], y = a[l];
  if ((x > y) == ((i & k) == 0)) {
    a[i] = y;
    a[l] = x;
  }
}

// Ascending bitonic sort of a[0..pa) and b[0..pb) (powers of two, padded with
// ~0) in shared memory, the two in lockstep.
__device__ void bitonic2(unsigned long long* a, int pa, unsigned long long* b, int pb) {
  const int P = pa > pb ? pa : pb;
  for (int k = 2; k <= P; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < P; i += kThreads) {
        const int l = i ^ j;
        if (l > i) {
          if (k <= pa) cmp_swap(a, i, l, k);
          if (k <= pb) cmp_swap(b, i, l, k);
        }
      }
      __syncthreads();
    }
  }
}

__device__ __forceinline__ int pow2_at_least(int n) {
  int p = 1;
  while (p < n) p <<= 1;
  return p;
}

__global__ void __launch_bounds__(kThreads, 1)
k_decode_select(const uint32_t* __restrict__ keys, uint32_t* __restrict__ hist0,
                const float* __restrict__ head, int chunk4, int max_boxes, AnchorGeo g,
                const int* __restrict__ err, DetResultHeader* __restrict__ hdr,
                rtcc_box* __restrict__ boxes) {
  extern __shared__ unsigned long long bnd[];        // [kBndCap] keys of bin b0
  __shared__ int hist[kMaxBins];
  __shared__ unsigned long long sel[kDecodeKeep];
  __shared__ int s_total, s_bin, s_below, s_nsel, s_nb;
  const int tid = threadIdx.x;
  const int lo = tid * chunk4 * 4;
  const int n4 = chunk4 * kThreads;                   // 16-byte vectors of padded keys
  pdl_trigger();
  pdl_wait();
  if (tid == 0) {
    s_nsel = 0;
    s_nb = 0;
  }

  // ---- 1. threshold bin from the top-12-bit histogram (level 0); when that
  // bin is too full for the list, a radix select over the next 10 + 10 bits
  // (levels 1, 2) finds the exact threshold key T and c = #keys < T
  uint32_t prefix = 0, pmask = 0;
  int below = 0, need = 0;
  bool list_path = false;
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
    if (lv == 0 && hist[prefix >> 20] <= kBndCap) {
      list_path = true;
      break;
    }
  }
  if (tid == 0) {
    hdr->n_boxes = need;
    hdr->err = *err;
  }
  if (need == 0) return;

  if (list_path) {
    // ---- 2. one pass: lower bins -> selection, bin b0 -> list ----------------
    const uint32_t b0 = prefix >> 20;
    const int nb0 = hist[b0];
    for_strided(keys, n4, [&](uint32_t k, int i) {
      if (k == kInvalid) return;
      const uint32_t bin = k >> 20;
      const unsigned long long e = (static_cast<unsigned long long>(k) << 32) | static_cast<unsigned>(i);
      if (bin < b0)
        sel[atomicAdd(&s_nsel, 1)] = e;
      else if (bin == b0)
        bnd[atomicAdd(&s_nb, 1)] = e;
    });
    __syncthreads();
    // ---- 3. sort both, complete the selection with bin b0's smallest --------
    const int pa = pow2_at_least(below), pb = pow2_at_least(nb0);
    for (int i = below + tid; i < pa; i += kThreads) sel[i] = ~0ull;
    for (int i = nb0 + tid; i < pb; i += kThreads) bnd[i] = ~0ull;
    __syncthreads();
    bitonic2(sel, pa, bnd, pb);
    for (int r = tid; r < need - below; r += kThreads) sel[below + r] = bnd[r];
    __syncthreads();
  } else {
    const uint32_t T = prefix;
    __syncthreads();

    // ---- 2'. collect keys < T, then the (need - below) lowest-index ties ----
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

    // sort the K selected pairs
    const int P2 = pow2_at_least(need);
    for (int i = need + tid; i < P2; i += kThreads) sel[i] = ~0ull;
    __syncthreads();
    bitonic2(sel, P2, sel, 1);
  }

  // ---- 4. decode the K pairs (in order) into boxes --------------------------
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
  const size_t dyn = kBndCap * sizeof(unsigned long long);
  cudaError_t e = cudaFuncSetAttribute(k_decode_select, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)dyn);
  if (e != cudaSuccess) return e;
  return launch_pdl(k_decode_select, dim3(1), dim3(kThreads), dyn, st, a.keys, a.hist0, a.head,
                    decode_key_chunk4(n), a.max_boxes, g, a.err, hdr, boxes);
}

}  // namespace rtcc

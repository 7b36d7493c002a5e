// Anchor decode, threshold and deterministic top-K of the head output (the
// detection post-processing that ends the complete-detection latency, Sec.
// V-A-3).  Rotated NMS is not part of this step.
//
// Order: class logit descending, then anchor index ascending.  The threshold
// and the order are decided on the logit itself (score = sigmoid(logit) is
// monotone), so the selected anchors are an exact function of the head
// output.  Keys are 64-bit: (order-preserving bits of -logit) << 32 | index,
// unique per anchor.
//   1. k_decode_chunk: each block sorts the keys of 4096 anchors in shared
//      memory (bitonic) and keeps its `keep` smallest.
//   2. k_decode_rank:  each kept key's global rank = its position in its chunk
//      + the number of smaller keys in every other chunk (binary search in the
//      sorted chunk lists, staged in shared memory).  Keys ranked below
//      max_boxes decode their box into output slot `rank`.
#include <cfloat>
#include <cmath>

#include "common.cuh"
#include "kernels.h"
#include "rtcc.h"

namespace rtcc {

namespace {

constexpr unsigned long long kNoKey = ~0ull;
constexpr int kChunkThreads = 1024;

__device__ __forceinline__ unsigned int ord_desc(float f) {
  // ascending unsigned order of the result == descending float order
  f = f + 0.0f;                                    // -0 -> +0
  const unsigned int u = __float_as_uint(f);
  const unsigned int asc = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ~asc;
}

__global__ void __launch_bounds__(kChunkThreads)
k_decode_chunk(const float* __restrict__ head, int n_anchors, int anchors, float thresh,
               int keep, unsigned long long* __restrict__ cand, int* __restrict__ cand_cnt) {
  __shared__ unsigned long long key[kDecodeChunk];
  __shared__ int nvalid;
  if (threadIdx.x == 0) nvalid = 0;
  __syncthreads();
  const int base = blockIdx.x * kDecodeChunk;
  int mine = 0;
  for (int i = threadIdx.x; i < kDecodeChunk; i += blockDim.x) {
    const int a = base + i;
    unsigned long long k = kNoKey;
    if (a < n_anchors) {
      const int cell = a / anchors, an = a - cell * anchors;
      const float cls = head[(size_t)cell * 16 + an];
      if (cls >= thresh) {
        k = (static_cast<unsigned long long>(ord_desc(cls)) << 32) | static_cast<unsigned>(a);
        ++mine;
      }
    }
    key[i] = k;
  }
  atomicAdd(&nvalid, mine);
  __syncthreads();
  for (int k = 2; k <= kDecodeChunk; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < kDecodeChunk; i += blockDim.x) {
        const int l = i ^ j;
        if (l > i) {
          const unsigned long long x = key[i], y = key[l];
          const bool asc = (i & k) == 0;
          if ((x > y) == asc) {
            key[i] = y;
            key[l] = x;
          }
        }
      }
      __syncthreads();
    }
  }
  for (int i = threadIdx.x; i < keep; i += blockDim.x)
    cand[(size_t)blockIdx.x * keep + i] = key[i];
  if (threadIdx.x == 0) cand_cnt[blockIdx.x] = nvalid < keep ? nvalid : keep;
}

struct AnchorGeo {
  float x_min, y_min, sx, sy;       // cell size in metres
  int feat_w, anchors;
  float la, wa, ha, za, da;
};

__global__ void k_decode_rank(const float* __restrict__ head,
                              const unsigned long long* __restrict__ cand,
                              const int* __restrict__ cand_cnt, int n_chunks, int keep,
                              int max_boxes, AnchorGeo g, const int* __restrict__ err,
                              DetResultHeader* __restrict__ hdr, rtcc_box* __restrict__ boxes) {
  extern __shared__ unsigned long long sk[];
  const int total = n_chunks * keep;
  for (int i = threadIdx.x; i < total; i += blockDim.x) sk[i] = cand[i];
  __syncthreads();
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    int n = 0;
    for (int c = 0; c < n_chunks; ++c) n += cand_cnt[c];
    hdr->n_boxes = n < max_boxes ? n : max_boxes;
    hdr->err = *err;
  }
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= total) return;
  const unsigned long long key = sk[t];
  if (key == kNoKey) return;
  const int mine = t / keep;
  int rank = t - mine * keep;
  for (int c = 0; c < n_chunks; ++c) {
    if (c == mine) continue;
    const unsigned long long* L = sk + (size_t)c * keep;
    int lo = 0, hi = keep;                          // count of L[i] < key
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (L[mid] < key) lo = mid + 1; else hi = mid;
    }
    rank += lo;
  }
  if (rank >= max_boxes) return;
  const int a = static_cast<int>(key & 0xFFFFFFFFull);
  const int cell = a / g.anchors, an = a - cell * g.anchors;
  const int ix = cell % g.feat_w, iy = cell / g.feat_w;
  const float* h = head + (size_t)cell * 16;
  const float cls = h[an];
  const float* r = h + g.anchors + 7 * an;
  const float xa = g.x_min + ((float)ix + 0.5f) * g.sx;
  const float ya = g.y_min + ((float)iy + 0.5f) * g.sy;
  rtcc_box b;
  b.x = xa + r[0] * g.da;
  b.y = ya + r[1] * g.da;
  b.z = g.za + r[2] * g.ha;
  b.l = g.la * expf(fminf(r[3], 10.0f));
  b.w = g.wa * expf(fminf(r[4], 10.0f));
  b.h = g.ha * expf(fminf(r[5], 10.0f));
  b.yaw = (float)an * (3.14159265358979f / (float)g.anchors) + r[6];
  b.score = 1.0f / (1.0f + expf(-cls));
  b.anchor = a;
  boxes[rank] = b;
}

int keep_for(int max_boxes) {
  int k = 1;
  while (k < max_boxes) k <<= 1;
  return k;
}

}  // namespace

int decode_chunks(int n_anchors) { return (n_anchors + kDecodeChunk - 1) / kDecodeChunk; }

cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t st) {
  const int n_anchors = a.feat_w * a.feat_h * a.anchors;
  const int nch = decode_chunks(n_anchors);
  const int keep = keep_for(a.max_boxes);
  if (keep > kDecodeKeep || keep > kDecodeChunk) return cudaErrorInvalidValue;
  DetResultHeader* hdr = static_cast<DetResultHeader*>(a.out);
  rtcc_box* boxes = reinterpret_cast<rtcc_box*>(hdr + 1);
  int* cnt = reinterpret_cast<int*>(a.cand + (size_t)nch * kDecodeKeep);
  k_decode_chunk<<<nch, kChunkThreads, 0, st>>>(a.head, n_anchors, a.anchors, a.cls_thresh,
                                                keep, a.cand, cnt);
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
  const int total = nch * keep;
  const size_t smem = sizeof(unsigned long long) * (size_t)total;
  if (smem > 48 * 1024) {
    if (smem > 200 * 1024) return cudaErrorInvalidValue;
    cudaFuncSetAttribute(k_decode_rank, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  }
  k_decode_rank<<<(total + 255) / 256, 256, smem, st>>>(a.head, a.cand, cnt, nch, keep,
                                                      a.max_boxes, g, a.err, hdr, boxes);
  return cudaGetLastError();
}

}  // namespace rtcc

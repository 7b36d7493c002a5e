// Anchor decode, threshold and deterministic top-K of the head output (the
// detection post-processing that ends the complete-detection latency, Sec.
// V-A-3).  Rotated NMS, when enabled, follows in its own kernel (nms.cu).
//
// Order: class logit descending, then anchor index ascending; threshold on the
// logit (score = sigmoid(logit) is monotone), so the selection is an exact
// function of the head output.  The fusion kernel leaves one 32-bit key per
// anchor whose ascending order is descending logit order (0xFFFFFFFF below the
// threshold), and a histogram of the keys' top 12 bits.  One block selects the
// K = min(max_boxes, #valid) smallest (key, index) pairs:
//   1. a scan of the histogram finds the bin b0 that holds the K-th pair and
//      the count of keys in lower bins;
//   2. one coalesced pass over the keys selects the keys of lower bins and
//      lists the keys of bin b0 in shared memory;
//   3. when both lists together fit one pair per thread (the usual case),
//      each pair's rank is the count of smaller pairs in its own list: the
//      lower bins' pairs take ranks 0 .. below-1, bin b0's pairs of rank
//      below K - below complete the K;
//   4. each ranked pair is decoded into the box of its rank (staged in shared
//      memory, then stored into the pinned host result block).
// Larger lists take two more steps instead of 3: a histogram of the listed
// keys' next 10 bits splits them into selected ones, the few of the bin b1
// that holds the K-th pair, and the rest; the selected pairs are ordered (warp
// bitonic runs of 32, then merge levels that place each pair by one binary
// search in its partner run; the pairs are distinct) and the lowest pairs of
// bin b1 complete the K.  When bin b0 or b1 is too full for the shared-memory
// lists (e.g. many equal logits), a radix select over the global keys (next
// 10 + 10 bits) finds the exact K-th key instead, the keys below it are
// collected, and an ordered pass (each thread owns a contiguous range of
// anchors, a block scan ranks its ties) adds the lowest-index keys equal to it.
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
constexpr int kTieCap = 64;                  // keys of the level-1 bin ranked directly
static_assert(sizeof(DetResultHeader) % 16 == 0, "the boxes follow the header 16-byte aligned");

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
__device__ __forceinline__ void for_chunk(const uint32_t* keys, int lo, int chunk4,
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

// Coalesced pass over the (padded) key array, one 16-byte vector (4 keys) at
// a time: thread t takes the vectors t, t + kThreads, ...; f(vector, index of
// its first key).
template <typename F>
__device__ __forceinline__ void for_strided4(const uint32_t* keys, int n4, F f) {
  const uint4* v = reinterpret_cast<const uint4*>(keys);
  constexpr int B = 8;                                   // loads in flight per thread
  for (int base = threadIdx.x; base < n4; base += B * kThreads) {
    uint4 r[B];
#pragma unroll
    for (int j = 0; j < B; ++j)
      if (base + j * kThreads < n4) r[j] = v[base + j * kThreads];
#pragma unroll
    for (int j = 0; j < B; ++j) {
      const int q = base + j * kThreads;
      if (q < n4) f(r[j], 4 * q);
    }
  }
}

// Append e to arr[] if pred, one shared-memory atomic per warp on the count
// (the appends of a pass all hit one counter).  Every active lane must call it.
__device__ __forceinline__ void warp_append(bool pred, unsigned long long e, int* count,
                                            unsigned long long* arr) {
  const unsigned act = __activemask();
  const unsigned m = __ballot_sync(act, pred);
  if (m == 0u) return;
  const int lane = threadIdx.x & 31;
  const int leader = __ffs(m) - 1;
  int base = 0;
  if (lane == leader) base = atomicAdd(count, __popc(m));
  base = __shfl_sync(act, base, leader);
  if (pred) arr[base + __popc(m & ((1u << lane) - 1u))] = e;
}

// Count of the pairs of a shared-memory list[0..n) (16-byte aligned) below v,
// shared by the S lanes q = 0..S-1 of a group (S a power of two): lane q
// reads the 16-byte chunks q, q + S, ... (two pairs each) and lane 0 the odd
// last pair.  The lanes of a group read consecutive chunks and the groups of
// a warp the same ones.  The caller sums the lanes.  (The count is bound by
// the shared-memory bandwidth: every compare's operand is delivered to its
// lane; explicit 16-byte loads halve the load instructions.)
__device__ __forceinline__ int count_below(const unsigned long long* list, int n, int q, int S,
                                           unsigned long long v) {
  const ulonglong2* l2 = reinterpret_cast<const ulonglong2*>(list);
  const int n2 = n >> 1;
  int cnt = 0;
#pragma unroll 4
  for (int j = q; j < n2; j += S) {
    const ulonglong2 x = l2[j];
    cnt += (x.x < v ? 1 : 0) + (x.y < v ? 1 : 0);
  }
  if ((n & 1) && q == 0) cnt += list[n - 1] < v ? 1 : 0;
  return cnt;
}

// Ascending bitonic sort of one value per lane across a warp.
__device__ __forceinline__ unsigned long long warp_sort32(unsigned long long v, int lane) {
#pragma unroll
  for (int k = 2; k <= 32; k <<= 1) {
#pragma unroll
    for (int j = k >> 1; j > 0; j >>= 1) {
      const unsigned long long p = __shfl_xor_sync(0xFFFFFFFFu, v, j);
      const bool up = (lane & k) == 0;                   // ascending sub-sequence
      const bool lower = (lane & j) == 0;                // lower lane of the pair
      v = (lower == up) ? (v < p ? v : p) : (v < p ? p : v);
    }
  }
  return v;
}

// Sort of n <= 512 distinct (key, index) pairs in two block-wide phases,
// run by the threads [t0, t0 + P) (P = n rounded up to a power of two >= 32):
// phase 1 sorts runs of 32 in registers (warp bitonic) into run[0..P);
// phase 2 ranks each pair by its position in its run plus binary searches in
// the other runs and hands the pairs of rank < limit to emit(rank, pair).
// The caller separates the phases with __syncthreads().
__device__ __forceinline__ int sort_width(int n) {
  int p = 32;
  while (p < n) p <<= 1;
  return p;
}
__device__ __forceinline__ void sort_phase1(const unsigned long long* in, int n, int t0, int P,
                                            unsigned long long* run) {
  const int t = threadIdx.x - t0;
  if (t >= 0 && t < P) run[t] = warp_sort32(t < n ? in[t] : ~0ull, threadIdx.x & 31);
}
// One level of the merge sort over warp-sorted runs, by the threads
// [t0, t0 + P): the runs of R pairs in src[0..P) merge pairwise into runs of
// 2R in dst.  A pair's place in the merged run is its index in its own run
// plus the count of the partner run's pairs below it (left run: strictly
// below; right run: below or equal), so every place is taken exactly once,
// padding (~0) included.
__device__ __forceinline__ void merge_level(const unsigned long long* src, unsigned long long* dst,
                                            int t0, int P, int R) {
  const int t = threadIdx.x - t0;
  if (t < 0 || t >= P || R >= P) return;
  const unsigned long long v = src[t];
  const int base = t & ~(2 * R - 1);
  const bool right = (t & R) != 0;
  const unsigned long long* other = src + base + (right ? 0 : R);
  int lo = 0, hi = R;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    const unsigned long long o = other[mid];
    if (right ? (o <= v) : (o < v)) lo = mid + 1;
    else hi = mid;
  }
  dst[base + (t & (R - 1)) + lo] = v;
}

// Box of the selected pair v (anchor = its low 32 bits), written to out.
__device__ __forceinline__ void decode_box(unsigned long long v, const float* head,
                                           const AnchorGeo& g, rtcc_box* out) {
  const int a = static_cast<int>(v & 0xFFFFFFFFull);
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
  *out = b;
}

__global__ void __launch_bounds__(kThreads, 1)
k_decode_select(const uint32_t* keys, uint32_t* hist0, const float* head, int chunk4, int max_boxes,
                AnchorGeo g, const int* err, DetResultHeader* __restrict__ hdr,
                rtcc_box* __restrict__ boxes, int* present, int K, volatile int* __restrict__ done,
                int* dev_n) {
  extern __shared__ __align__(16) unsigned long long bnd[];  // [kBndCap] keys of bin b0
  __shared__ int hist[kThreads];                     // level-1/2 histograms (10 bits)
  __shared__ __align__(16) unsigned long long sel[kDecodeKeep];  // selected, unordered
  __shared__ unsigned long long tie[kTieCap];
  __shared__ __align__(16) rtcc_box sbox[kDecodeKeep];  // boxes in rank order
  __shared__ int s_total, s_bin, s_below, s_nsel, s_nb, s_nl, s_nt;
  const int tid = threadIdx.x;
  const int n4 = chunk4 * kThreads;                   // 16-byte vectors of padded keys
  pdl_trigger();
  pdl_wait();
  if (tid == 0) {
    s_nsel = 0;
    s_nl = 0;
    s_nt = 0;
  }

  // ---- 1. level 0: the bin b0 of the top-12-bit histogram that holds the
  // K-th key, and the count below0 of keys in lower bins -------------------
  static_assert(kMaxBins == 4 * kThreads, "one 16-byte vector of bins per thread");
  int need;
  {
    // each thread: the contiguous bins 4*tid .. 4*tid+3
    uint4* hv = reinterpret_cast<uint4*>(hist0) + tid;
    const uint4 q = *hv;
    *hv = make_uint4(0u, 0u, 0u, 0u);                  // ready for the next frame
    const int h[4] = {(int)q.x, (int)q.y, (int)q.z, (int)q.w};
    int run = block_scan_excl(h[0] + h[1] + h[2] + h[3], &s_total);
    need = s_total < max_boxes ? s_total : max_boxes;  // K
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (run < need && run + h[j] >= need) {
        s_bin = 4 * tid + j;
        s_below = run;
        s_nb = h[j];
      }
      run += h[j];
    }
    __syncthreads();
  }
  if (tid == 0) {
    if (dev_n) {                                        // NMS follows: it writes the header
      *dev_n = need;
    } else {
      hdr->n_boxes = need;
      hdr->err = *err;
    }
  }
  if (need > 0) {
    const uint32_t b0 = static_cast<uint32_t>(s_bin);
    const int below0 = s_below;
    const int nb0 = s_nb;
    bool ranked = false;

    if (nb0 <= kBndCap) {
      // ---- 2. one coalesced pass: lower bins -> sel, bin b0 -> bnd ----------
      for_strided4(keys, n4, [&](const uint4& x, int i0) {
        // few keys are candidates (about K of tens of thousands): a warp
        // skips a round of 4 keys per lane after one vote on the smallest
        // key of each lane's vector (invalid keys: bin 4095 > b0)
        const uint32_t mn = min(min(x.x, x.y), min(x.z, x.w));
        if (__any_sync(__activemask(), (mn >> 20) <= b0)) {
          const uint32_t kk[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const uint32_t k = kk[e], bin = k >> 20;
            const bool cand = k != kInvalid && bin <= b0;
            const unsigned long long pr = (static_cast<unsigned long long>(k) << 32) | static_cast<unsigned>(i0 + e);
            warp_append(cand && bin < b0, pr, &s_nsel, sel);
            warp_append(cand && bin == b0, pr, &s_nl, bnd);
          }
        }
      });
      __syncthreads();                                   // every thread has read nb0
      if (below0 + nb0 <= kThreads) {
        // ---- 3. the candidates fit one per thread: rank each pair within its
        // list by counting the smaller pairs there (pairs are distinct, so the
        // ranks are a permutation).  The lower bins' pairs are all selected
        // and come first in rank order; a pair of bin b0 is selected when its
        // rank is below need - below0.  S lanes share a pair, each counting a
        // strided part of the list (broadcast shared-memory reads), and the
        // rank is the box slot: the box is decoded at once.
        const int nc = below0 + nb0;
        int S = 1;
        while (S < 32 && nc * 2 * S <= kThreads) S <<= 1;
        const int c = tid / S, q = tid & (S - 1);
        const bool lower = c < below0;
        unsigned long long v = 0;
        int cnt = 0;
        if (c < nc) {
          v = lower ? sel[c] : bnd[c - below0];
          cnt = lower ? count_below(sel, below0, q, S, v) : count_below(bnd, nb0, q, S, v);
        }
        for (int o = S >> 1; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xFFFFFFFFu, cnt, o);
        if (c < nc && q == 0) {
          const int slot = lower ? cnt : below0 + cnt;
          if (slot < need) decode_box(v, head, g, sbox + slot);
        }
        ranked = true;
      } else {
        // ---- 3'. level 1 over bnd (key bits 10..19 = pair bits 42..51) --------
        for (int i = tid; i < 1024; i += kThreads) hist[i] = 0;
        __syncthreads();
        // many listed keys share their next 10 bits: lanes with the same bin add
        // their count with one atomic (uniform trip count: warps stay converged)
        for (int i0 = 0; i0 < nb0; i0 += kThreads) {
          const int i = i0 + tid;
          const int bin1 = i < nb0 ? (int)((bnd[i] >> 42) & 1023) : -1;
          const unsigned peers = __match_any_sync(0xFFFFFFFFu, bin1);
          if (bin1 >= 0 && (tid & 31) == __ffs(peers) - 1) atomicAdd(&hist[bin1], __popc(peers));
        }
        __syncthreads();
        {
          int run = block_scan_excl(hist[tid], &s_total);  // 1024 bins, one per thread
          const int h = hist[tid];
          if (below0 + run < need && below0 + run + h >= need) {
            s_bin = tid;
            s_below = below0 + run;
          }
          __syncthreads();
        }
        const int b1 = s_bin, below1 = s_below, nb1 = hist[b1];
        if (nb1 <= kTieCap) {
          // bin-1 entries below b1 are selected; those in b1 compete for the rest
          for (int i = tid; i < nb0; i += kThreads) {
            const unsigned long long e = bnd[i];
            const int bin1 = (int)((e >> 42) & 1023);
            warp_append(bin1 < b1, e, &s_nsel, sel);
            warp_append(bin1 == b1, e, &s_nt, tie);
          }
          __syncthreads();
          // ---- 4'. order sel (below1 pairs) and tie (nb1 pairs, all above);
          // each ranked pair is decoded straight into its box slot
          // (bnd is free again and serves as the run buffer)
          const int P1 = sort_width(below1), P2 = sort_width(nb1);
          unsigned long long *a = bnd, *a2 = bnd + 2 * kDecodeKeep;              // sel runs
          unsigned long long *b = bnd + kDecodeKeep, *b2 = bnd + kDecodeKeep + kTieCap;  // tie runs
          sort_phase1(sel, below1, 0, P1, a);
          sort_phase1(tie, nb1, kDecodeKeep, P2, b);
          __syncthreads();
          for (int R = 32; R < (P1 > P2 ? P1 : P2); R *= 2) {
            merge_level(a, a2, 0, P1, R);
            merge_level(b, b2, kDecodeKeep, P2, R);
            __syncthreads();
            if (R < P1) { unsigned long long* x = a; a = a2; a2 = x; }
            if (R < P2) { unsigned long long* x = b; b = b2; b2 = x; }
          }
          if (tid < below1) decode_box(a[tid], head, g, sbox + tid);
          const int tt = tid - kDecodeKeep;
          if (tt >= 0 && tt < need - below1) decode_box(b[tt], head, g, sbox + below1 + tt);
          ranked = true;
        }
      }
    }

    if (!ranked) {
      __syncthreads();                                   // every thread has read hist
      // ---- 2'. radix select over the global keys: levels 1 and 2 (10 bits
      // each) below the bin-0 prefix give the exact K-th key T and the count
      // `below` of keys < T ---------------------------------------------------
      uint32_t prefix = b0 << 20, pmask = 0xFFFu << 20;
      int below = below0;
      const int lo = tid * chunk4 * 4;
      for (int lv = 1; lv <= 2; ++lv) {
        const int sh = lv == 1 ? 10 : 0;
        for (int i = tid; i < 1024; i += kThreads) hist[i] = 0;
        __syncthreads();
        for_chunk(keys, lo, chunk4, [&](uint32_t k, int) {
          if (k != kInvalid && (k & pmask) == prefix) atomicAdd(&hist[(k >> sh) & 1023], 1);
        });
        __syncthreads();
        int run = block_scan_excl(hist[tid], &s_total);
        const int h = hist[tid];
        if (below + run < need && below + run + h >= need) {
          s_bin = tid;
          s_below = below + run;
        }
        __syncthreads();
        prefix |= static_cast<uint32_t>(s_bin) << sh;
        pmask |= 1023u << sh;
        below = s_below;
        __syncthreads();
      }
      const uint32_t T = prefix;
      if (tid == 0) s_nsel = 0;
      __syncthreads();
      // collect keys < T, then the (need - below) lowest-index keys equal to T:
      // each thread owns a contiguous range of anchors and a block scan ranks
      // its ties
      int ties = 0;
      for_chunk(keys, lo, chunk4, [&](uint32_t k, int i) {
        if (k < T) {
          sel[atomicAdd(&s_nsel, 1)] = (static_cast<unsigned long long>(k) << 32) | static_cast<unsigned>(i);
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
      const int P = sort_width(need);
      unsigned long long *a = bnd, *a2 = bnd + 2 * kDecodeKeep;
      sort_phase1(sel, need, 0, P, a);
      __syncthreads();
      for (int R = 32; R < P; R *= 2) {
        merge_level(a, a2, 0, P, R);
        __syncthreads();
        unsigned long long* x = a;
        a = a2;
        a2 = x;
      }
      if (tid < need) decode_box(a[tid], head, g, sbox + tid);
    }
    // the boxes leave shared memory in 16-byte pieces (coalesced stores into
    // the pinned host block, or into device memory when NMS follows)
    __syncthreads();
    const int nbytes = need * (int)sizeof(rtcc_box);
    const uint4* src = reinterpret_cast<const uint4*>(sbox);
    uint4* dst = reinterpret_cast<uint4*>(boxes);
    for (int i = tid; i < nbytes / 16; i += kThreads) dst[i] = src[i];
    for (int i = (nbytes / 16) * 4 + tid; i < nbytes / 4; i += kThreads)
      reinterpret_cast<uint32_t*>(boxes)[i] = reinterpret_cast<const uint32_t*>(sbox)[i];
  }  // need > 0

  // the fusion kernel has read the presence flags: clear them for the next
  // frame, then publish the result block to the host (unless NMS follows: its
  // dependency wait makes this kernel's writes visible to it)
  if (tid < K) present[tid] = 0;
  if (!dev_n) {
    __threadfence_system();                        // this thread's box writes, system-wide
    __syncthreads();
    if (tid == 0) *done = 1;
  }
}


}  // namespace

int decode_key_chunk4(int n_anchors) { return (n_anchors + 4 * kThreads - 1) / (4 * kThreads); }

cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t st) {
  const int n = a.feat_w * a.feat_h * a.anchors;
  if (a.max_boxes < 1 || a.max_boxes > kDecodeKeep) return cudaErrorInvalidValue;
  DetResultHeader* hdr = static_cast<DetResultHeader*>(a.out);
  rtcc_box* boxes = a.dev_boxes ? a.dev_boxes : reinterpret_cast<rtcc_box*>(hdr + 1);
  if ((a.dev_boxes == nullptr) != (a.dev_n == nullptr)) return cudaErrorInvalidValue;
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
  if (!a.present || !a.done || a.K < 1 || a.K > RTCC_MAX_AGENTS) return cudaErrorInvalidValue;
  return launch_pdl(k_decode_select, dim3(1), dim3(kThreads), dyn, st, a.keys, a.hist0, a.head,
                    decode_key_chunk4(n), a.max_boxes, g, a.err, hdr, boxes, a.present, a.K,
                    a.done, a.dev_n);
}

}  // namespace rtcc

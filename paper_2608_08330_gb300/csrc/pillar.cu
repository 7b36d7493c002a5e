// Pillarisation, pillar feature net (PFN) and BEV scatter of one encoder
// branch E_k (the first stage of the per-agent encoder, Sec. III-B / Sec.
// V-A-1: a PointPillars encoder).
//
// The grouping is exactly the sequential rule "visit points in order; a new
// cell opens the next pillar id unless P_max pillars exist; a pillar keeps its
// first N_max points", computed without order-dependent atomics:
//   1. cells:   per point cell id (float32 index arithmetic), per-cell point
//               count and first point index (atomicAdd / atomicMin: both give
//               order-independent results).
//   2. scan:    a point is a "first point" iff first[cell] == i.  An exclusive
//               scan of first-point flags over point order gives each cell its
//               pillar id (= rank of its first occurrence); the same scan of
//               the cells' counts gives each pillar's offset in a point list.
//   3. fill:    every point of a kept pillar appends its index to the pillar's
//               list (slot order arbitrary).
//   4. PFN:     one warp per pillar selects the N_max smallest indices of its
//               list (warp bitonic sort/merge), i.e. the first N_max points in
//               point order, one point per lane.  The means sum in lane order;
//               then each lane owns C/32 output channels and folds the kept
//               points in one at a time (broadcast by shuffle): the linear map
//               of the 9-d decorated features, rewritten as 4 per-point terms
//               plus a per-pillar constant, ReLU, running max.  Every reduction
//               has a fixed order, so the result is run-to-run deterministic.
//   5. image:   the PFN writes each kept pillar's vector into its cell of the
//               pseudo-image and its id into cell2pillar (each cell has at most
//               one pillar: no atomics).  Elsewhere the image holds zeros and
//               cell2pillar -1: the first kernel of a pass clears the cells the
//               previous pass wrote (np_prev of them), and the fill kernel, the
//               last reader of the per-cell counters, restores them.
#include <climits>

#include "common.cuh"
#include "kernels.h"

namespace rtcc {

namespace {

constexpr unsigned kFull = 0xFFFFFFFFu;

// Pointers to data an earlier kernel of the chain writes are not __restrict__:
// a read through a const __restrict__ pointer may be scheduled above
// griddepcontrol.wait (the qualifier promises the data does not change while
// the kernel runs), and would then read the predecessor's output before it is
// complete.  Only the constant PFN weights keep the qualifier.

template <int CH>
__global__ void k_pillar_cells(const float4* pts, const int* n_hdr,
                               GridGeom g, int* cell_of, int* cnt_cell,
                               int* first_cell, int* stats,
                               const int* prev_cell, const int* np_prev,
                               int clear_all, uint4* image,
                               int* cell2pillar, int* present_flag,
                               const int* src_hdr, const float4* src_pts,
                               int* dst_hdr, float4* dst_pts) {
  __shared__ int s_n;
  pdl_trigger();
  pdl_wait();
  // zero-copy payload: one read of the header per block, every point read
  // once from the source and copied to the device slot the later kernels use
  if (threadIdx.x == 0) s_n = src_hdr ? *src_hdr : *n_hdr;
  __syncthreads();
  const int n = s_n;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i == 0 && dst_hdr) *dst_hdr = n;
  if (i == 0 && present_flag) *present_flag = 1;     // this agent's slot is filled this frame
  // clear what the previous pass wrote (CH 16-byte chunks per cell)
  {
    const long long stride = (long long)gridDim.x * blockDim.x;
    if (clear_all) {
      const long long tot = (long long)g.W * g.H * CH;
      for (long long q = i; q < tot; q += stride) {
        image[q] = make_uint4(0u, 0u, 0u, 0u);
        if (q % CH == 0) cell2pillar[q / CH] = -1;
      }
    } else {
      const long long tot = (long long)(*np_prev) * CH;
      for (long long q = i; q < tot; q += stride) {
        const int cell = prev_cell[q / CH];
        image[(size_t)cell * CH + q % CH] = make_uint4(0u, 0u, 0u, 0u);
        if (q % CH == 0) cell2pillar[cell] = -1;
      }
    }
  }
  if (i == 0) stats[0] = n;
  if (i < n) {
    const float4 p = src_pts ? src_pts[i] : pts[i];
    if (dst_pts) dst_pts[i] = p;
    // IEEE float32 subtraction and division with round-to-nearest.
    const float fx = __fdiv_rn(__fsub_rn(p.x, g.x_min), g.v);
    const float fy = __fdiv_rn(__fsub_rn(p.y, g.y_min), g.v);
    const bool ok = (p.z >= g.z_min) && (p.z < g.z_max) && (fx >= 0.f) && (fx < (float)g.W) &&
                    (fy >= 0.f) && (fy < (float)g.H);
    int cell = -1;
    if (ok) {
      const int ix = (int)floorf(fx);
      const int iy = (int)floorf(fy);
      cell = iy * g.W + ix;
      atomicAdd(&cnt_cell[cell], 1);
      atomicMin(&first_cell[cell], i);
    }
    cell_of[i] = cell;
  }
}

// Flag and count of point i for the pillar scan.
__device__ __forceinline__ int2 first_point_item(int i, int n, const int* cell_of,
                                                 const int* cnt_cell, const int* first_cell) {
  if (i >= n) return make_int2(0, 0);
  const int cell = cell_of[i];
  if (cell < 0 || first_cell[cell] != i) return make_int2(0, 0);
  return make_int2(1, cnt_cell[cell]);
}

__device__ __forceinline__ int2 add2(int2 a, int2 b) { return make_int2(a.x + b.x, a.y + b.y); }

__device__ __forceinline__ int2 shfl_up2(int2 v, int d) {
  return make_int2(__shfl_up_sync(kFull, v.x, d), __shfl_up_sync(kFull, v.y, d));
}
__device__ __forceinline__ int2 shfl_xor2(int2 v, int d) {
  return make_int2(__shfl_xor_sync(kFull, v.x, d), __shfl_xor_sync(kFull, v.y, d));
}

// Exclusive block scan of one int2 per thread (blockDim a multiple of 32, up to
// 1024); returns the exclusive prefix and writes the block total to *total.
__device__ int2 block_excl_scan(int2 v, int2* total) {
  __shared__ int2 warp_sums[32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  int2 inc = v;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int2 o = shfl_up2(inc, d);
    if (lane >= d) inc = add2(inc, o);
  }
  if (lane == 31) warp_sums[wid] = inc;
  __syncthreads();
  if (wid == 0) {
    int2 w = (lane < (int)(blockDim.x >> 5)) ? warp_sums[lane] : make_int2(0, 0);
    int2 winc = w;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int2 o = shfl_up2(winc, d);
      if (lane >= d) winc = add2(winc, o);
    }
    warp_sums[lane] = make_int2(winc.x - w.x, winc.y - w.y);   // exclusive
    if (lane == 31) *total = winc;
  }
  __syncthreads();
  const int2 wpre = warp_sums[wid];
  return make_int2(wpre.x + inc.x - v.x, wpre.y + inc.y - v.y);
}

constexpr int kScanThreads = 256;
constexpr int kItems = kScanTile / kScanThreads;   // 4 consecutive points per thread
static_assert(kItems == 4, "the item loads below move 4 points per thread");

// Same-address atomics serialise in L2, so the pass's counters are summed per
// block and added once per block (here and in the scan), not per point, warp
// or pillar.
__global__ void __launch_bounds__(kScanThreads)
k_pillar_blocksum(const int* n_hdr, const int* cell_of,
                  const int* cnt_cell, const int* first_cell,
                  int2* items, int2* blocksum, int* stats) {
  pdl_trigger();
  pdl_wait();
  const int n = *n_hdr;
  const int base = blockIdx.x * kScanTile + threadIdx.x * kItems;
  int2 s = make_int2(0, 0);
  int2 it[kItems];
  int inr = 0;                                 // points inside the grid
#pragma unroll
  for (int q = 0; q < kItems; ++q) {
    it[q] = first_point_item(base + q, n, cell_of, cnt_cell, first_cell);
    s = add2(s, it[q]);
    inr += (base + q < n && cell_of[base + q] >= 0) ? 1 : 0;
  }
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) inr += __shfl_xor_sync(kFull, inr, d);
  if (base < n) {
    int4* dst = reinterpret_cast<int4*>(items + base);
    dst[0] = make_int4(it[0].x, it[0].y, it[1].x, it[1].y);
    dst[1] = make_int4(it[2].x, it[2].y, it[3].x, it[3].y);
  }
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) s = add2(s, shfl_xor2(s, d));
  __shared__ int2 ws[32];
  __shared__ int wi[32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (lane == 0) {
    ws[wid] = s;
    wi[wid] = inr;
  }
  __syncthreads();
  if (wid == 0) {
    int2 t = lane < (int)(blockDim.x >> 5) ? ws[lane] : make_int2(0, 0);
    int ti = lane < (int)(blockDim.x >> 5) ? wi[lane] : 0;
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) {
      t = add2(t, shfl_xor2(t, d));
      ti += __shfl_xor_sync(kFull, ti, d);
    }
    if (lane == 0) {
      blocksum[blockIdx.x] = t;
      if (ti) atomicAdd(&stats[1], ti);
    }
  }
}

__global__ void __launch_bounds__(kScanThreads)
k_pillar_scan(const int* n_hdr, const int* cell_of,
              const int2* items, const int2* blocksum, int P, int N,
              int* c2p,
              int* pillar_cell, int* pcnt_raw, int* poff,
              int* cursor, int* stats) {
  __shared__ int2 pre;
  __shared__ int2 tot;
  pdl_trigger();
  pdl_wait();
  const int n = *n_hdr;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x < 32) {
    int2 s = make_int2(0, 0);
    for (int j = lane; j < (int)blockIdx.x; j += 32) s = add2(s, blocksum[j]);
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) s = add2(s, shfl_xor2(s, d));
    if (lane == 0) pre = s;
  }
  __syncthreads();
  const int base = blockIdx.x * kScanTile + threadIdx.x * kItems;
  int2 it[kItems] = {};
  if (base < n) {
    const int4* src = reinterpret_cast<const int4*>(items + base);
    const int4 a = src[0], b = src[1];
    it[0] = make_int2(a.x, a.y);
    it[1] = make_int2(a.z, a.w);
    it[2] = make_int2(b.x, b.y);
    it[3] = make_int2(b.z, b.w);
  }
  int2 own = make_int2(0, 0);
#pragma unroll
  for (int q = 0; q < kItems; ++q) own = add2(own, it[q]);
  int2 run = block_excl_scan(own, &tot);
  run = add2(run, pre);
  int kept = 0, raw = 0;                       // points of this thread's kept pillars
#pragma unroll
  for (int q = 0; q < kItems; ++q) {
    if (it[q].x) {
      const int i = base + q;
      const int cell = cell_of[i];
      const int pid = run.x;
      c2p[cell] = pid;
      if (pid < P) {
        pillar_cell[pid] = cell;
        pcnt_raw[pid] = it[q].y;
        poff[pid] = run.y;
        cursor[pid] = 0;
        kept += it[q].y < N ? it[q].y : N;
        raw += it[q].y;
      }
    }
    run = add2(run, it[q]);
  }
  // the PFN keeps min(raw, N) points of a pillar: stats 3 (kept), 6 (dropped
  // by the per-pillar cap), 7 (points of kept pillars), summed per block
  __shared__ int2 wk[32];
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) {
    kept += __shfl_xor_sync(kFull, kept, d);
    raw += __shfl_xor_sync(kFull, raw, d);
  }
  if (lane == 0) wk[threadIdx.x >> 5] = make_int2(kept, raw);
  __syncthreads();
  if (threadIdx.x == 0) {
    int2 t = make_int2(0, 0);
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t = add2(t, wk[w]);
    if (t.y) {
      atomicAdd(&stats[3], t.x);
      atomicAdd(&stats[6], t.y - t.x);
      atomicAdd(&stats[7], t.y);
    }
  }
  if (blockIdx.x == gridDim.x - 1 && threadIdx.x == 0) {
    const int total = pre.x + tot.x;
    stats[2] = total < P ? total : P;
  }
}

__global__ void k_pillar_fill(const int* n_hdr, const int* cell_of,
                              const int* c2p, int P, const int* poff,
                              int* cursor, int* list,
                              int* cnt_cell, int* first_cell) {
  pdl_trigger();
  pdl_wait();
  const int n = *n_hdr;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const int cell = cell_of[i];
  if (cell < 0) return;
  // the scan was the last reader of the per-cell counters: restore them for
  // the next pass (every point of the cell writes the same values)
  cnt_cell[cell] = 0;
  first_cell[cell] = kFirstInit;
  const int p = c2p[cell];
  if (p >= P) return;
  const int pos = poff[p] + atomicAdd(&cursor[p], 1);
  list[pos] = i;
}

// Ascending bitonic sort of one value per lane.
__device__ __forceinline__ int warp_sort_asc(int v, int lane) {
#pragma unroll
  for (int k = 2; k <= 32; k <<= 1) {
#pragma unroll
    for (int j = k >> 1; j > 0; j >>= 1) {
      const int o = __shfl_xor_sync(kFull, v, j);
      const bool up = (lane & k) == 0;
      const bool lower = (lane & j) == 0;
      v = (lower == up) ? min(v, o) : max(v, o);
    }
  }
  return v;
}

// Sort a bitonic sequence (one value per lane) ascending.
__device__ __forceinline__ int warp_merge_asc(int v, int lane) {
#pragma unroll
  for (int j = 16; j > 0; j >>= 1) {
    const int o = __shfl_xor_sync(kFull, v, j);
    v = ((lane & j) == 0) ? min(v, o) : max(v, o);
  }
  return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) v += __shfl_xor_sync(kFull, v, d);
  return v;
}

template <typename T, int C>
__global__ void __launch_bounds__(256)
k_pfn(const float4* pts, const int* stats_in,
      const int* pcnt_raw, const int* poff,
      const int* list, const int* pillar_cell,
      const float* __restrict__ w, const float* __restrict__ b, GridGeom g, int N,
      T* image, int* cell2pillar, int* np_prev,
      int* pcount, unsigned long long* span) {
  __shared__ float sw[C * 9];
  __shared__ float sb[C];
  pdl_trigger();
  for (int j = threadIdx.x; j < C * 9; j += blockDim.x) sw[j] = w[j];   // weights: constant
  pdl_wait();
  span_begin(span);
  for (int j = threadIdx.x; j < C; j += blockDim.x) sb[j] = b[j];
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int p = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int np = stats_in[2];
  if (blockIdx.x == 0 && threadIdx.x == 0) *np_prev = np;   // cleared by the next pass
  if (p < np) {
    const int raw = pcnt_raw[p];
    const int base = poff[p];
    // the min(raw, N) smallest point indices, ascending = the pillar's first points
    int idx = lane < raw ? list[base + lane] : INT_MAX;
    idx = warp_sort_asc(idx, lane);
    for (int c = 32; c < raw; c += 32) {
      int v = (c + lane < raw) ? list[base + c + lane] : INT_MAX;
      v = warp_sort_asc(v, lane);
      const int vr = __shfl_sync(kFull, v, 31 - lane);
      idx = warp_merge_asc(min(idx, vr), lane);
    }
    const int m = raw < N ? raw : N;
    const bool valid = lane < m;
    const float4 q = valid ? pts[idx] : make_float4(0.f, 0.f, 0.f, 0.f);
    const float fm = (float)m;
    const float mx = __fdiv_rn(warp_sum(q.x), fm);
    const float my = __fdiv_rn(warp_sum(q.y), fm);
    const float mz = __fdiv_rn(warp_sum(q.z), fm);
    const int cell = pillar_cell[p];
    const int cx = cell % g.W, cy = cell / g.W;
    const float xc = __fadd_rn(g.x_min, __fmul_rn((float)cx + 0.5f, g.v));
    const float yc = __fadd_rn(g.y_min, __fmul_rn((float)cy + 0.5f, g.v));
    // The 9 decorated features (x, y, z, i, x - mx, y - my, z - mz, x - xc,
    // y - yc) are affine in the point's (dx, dy, z, i) = (x - xc, y - yc, z,
    // i):  W f = (W0 + W4 + W7) dx + (W1 + W5 + W8) dy + (W2 + W6) z + W3 i
    //          + [W0 xc + W1 yc - W4 (mx - xc) - W5 (my - yc) - W6 mz],
    // the bracket the same for every point of the pillar.  Folding it into
    // the bias leaves 4 FMAs per point and channel instead of 9 (the loop was
    // bound by instruction issue), in fp32 throughout.  ReLU folds into the
    // running max, which starts at 0 (m >= 1).
    const float mdx = __fsub_rn(mx, xc), mdy = __fsub_rn(my, yc);
    const float pdx = __fsub_rn(q.x, xc), pdy = __fsub_rn(q.y, yc);   // this lane's point
    // channel-parallel: lane l owns channels [l*PER, (l+1)*PER); the pillar's
    // kept points (one per lane, in point order) are broadcast one at a time
    constexpr int PER = C / 32;
    float wc[PER][4], cst[PER], acc[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const float* wr = sw + (lane * PER + i) * 9;
      wc[i][0] = wr[0] + wr[4] + wr[7];
      wc[i][1] = wr[1] + wr[5] + wr[8];
      wc[i][2] = wr[2] + wr[6];
      wc[i][3] = wr[3];
      float c = sb[lane * PER + i];
      c = fmaf(wr[0], xc, c);
      c = fmaf(wr[1], yc, c);
      c = fmaf(-wr[4], mdx, c);
      c = fmaf(-wr[5], mdy, c);
      c = fmaf(-wr[6], mz, c);
      cst[i] = c;
      acc[i] = 0.f;
    }
    for (int j = 0; j < m; ++j) {
      const float dx = __shfl_sync(kFull, pdx, j);
      const float dy = __shfl_sync(kFull, pdy, j);
      const float zz = __shfl_sync(kFull, q.z, j);
      const float it = __shfl_sync(kFull, q.w, j);
#pragma unroll
      for (int i = 0; i < PER; ++i) {
        float sacc = fmaf(wc[i][0], dx, cst[i]);
        sacc = fmaf(wc[i][1], dy, sacc);
        sacc = fmaf(wc[i][2], zz, sacc);
        sacc = fmaf(wc[i][3], it, sacc);
        acc[i] = fmaxf(acc[i], sacc);
      }
    }
    // the pillar's vector goes straight into its cell of the pseudo-image
    T* dst = image + (size_t)cell * C + lane * PER;
    if (PER == 2) {
      *reinterpret_cast<uint32_t*>(dst) = Store<T>::pack2(acc[0], acc[PER - 1]);
    } else {
#pragma unroll
      for (int i = 0; i < PER; ++i) dst[i] = Store<T>::from_f(acc[i]);
    }
    if (lane == 0) {
      cell2pillar[cell] = p;
      pcount[p] = m;
    }
  }
  if (span) {
    __syncthreads();
    span_end(span);
  }
}

template <typename T, int C>
cudaError_t launch_all(const PillarBufs& b, const GridGeom& g, const float* pfn_w,
                       const float* pfn_b, cudaStream_t st) {
  const int nblk = scan_blocks(b.cap);
  cudaError_t e;
  constexpr int CH = C * 2 / 16;                  // 16-byte chunks per cell
  e = launch_pdl(k_pillar_cells<CH>, dim3((b.cap + 255) / 256), dim3(256), 0, st, b.pts, b.n_hdr,
                 g, b.cell_of, b.cnt_cell, b.first_cell, b.stats,
                 static_cast<const int*>(b.pillar_cell), static_cast<const int*>(b.np_prev),
                 b.clear_all, static_cast<uint4*>(b.image), b.cell2pillar, b.present_flag,
                 b.src_hdr, b.src_pts, b.dst_hdr, b.dst_pts);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k_pillar_blocksum, dim3(nblk), dim3(kScanThreads), 0, st, b.n_hdr, b.cell_of,
                 b.cnt_cell, b.first_cell, b.items, b.blocksum, b.stats);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k_pillar_scan, dim3(nblk), dim3(kScanThreads), 0, st, b.n_hdr, b.cell_of,
                 b.items, b.blocksum, b.P, b.N, b.c2p, b.pillar_cell, b.pcnt_raw, b.poff, b.cursor,
                 b.stats);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k_pillar_fill, dim3((b.cap + 255) / 256), dim3(256), 0, st, b.n_hdr, b.cell_of,
                 b.c2p, b.P, b.poff, b.cursor, b.list, b.cnt_cell, b.first_cell);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k_pfn<T, C>, dim3((b.P + 7) / 8), dim3(256), 0, st, b.pts, b.stats, b.pcnt_raw,
                 b.poff, b.list, b.pillar_cell, pfn_w, pfn_b, g, b.N, static_cast<T*>(b.image),
                 b.cell2pillar, b.np_prev, b.pcount, b.pfn_span);
  return e;                                       // each launch reported its own status
}

}  // namespace

cudaError_t launch_pillarise(const PillarBufs& b, const GridGeom& g, const float* pfn_w,
                             const float* pfn_b, bool bf16, int* /*err*/, cudaStream_t st) {
  if (b.C == 64) {
    return bf16 ? launch_all<__nv_bfloat16, 64>(b, g, pfn_w, pfn_b, st)
                : launch_all<__half, 64>(b, g, pfn_w, pfn_b, st);
  }
  if (b.C == 32) {
    return bf16 ? launch_all<__nv_bfloat16, 32>(b, g, pfn_w, pfn_b, st)
                : launch_all<__half, 32>(b, g, pfn_w, pfn_b, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace rtcc

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
//               point order, then computes the 9-d features, the linear layer,
//               ReLU and the max over points; every reduction has a fixed
//               order, so the result is run-to-run deterministic.
//   5. scatter: one pass over all cells writes the pillar vector or zeros
//               (each cell has at most one pillar: no atomics) and restores the
//               per-cell scratch for the next pass.
#include <climits>

#include "common.cuh"
#include "kernels.h"

namespace rtcc {

namespace {

constexpr unsigned kFull = 0xFFFFFFFFu;

__global__ void k_pillar_cells(const float4* __restrict__ pts, const int* __restrict__ n_hdr,
                               GridGeom g, int* __restrict__ cell_of, int* __restrict__ cnt_cell,
                               int* __restrict__ first_cell, int* __restrict__ stats) {
  const int n = *n_hdr;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i == 0) stats[0] = n;
  bool ok = false;
  if (i < n) {
    const float4 p = pts[i];
    // IEEE float32 subtraction and division with round-to-nearest.
    const float fx = __fdiv_rn(__fsub_rn(p.x, g.x_min), g.v);
    const float fy = __fdiv_rn(__fsub_rn(p.y, g.y_min), g.v);
    ok = (p.z >= g.z_min) && (p.z < g.z_max) && (fx >= 0.f) && (fx < (float)g.W) &&
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
  const unsigned in_range = __ballot_sync(kFull, ok);
  if ((threadIdx.x & 31) == 0 && in_range) atomicAdd(&stats[1], __popc(in_range));
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

// Exclusive block scan of one int2 per thread (1024 threads); returns the
// exclusive prefix and writes the block total to *total.
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

constexpr int kScanThreads = 1024;
constexpr int kItems = kScanTile / kScanThreads;   // 4 consecutive points per thread

__global__ void __launch_bounds__(kScanThreads)
k_pillar_blocksum(const int* __restrict__ n_hdr, const int* __restrict__ cell_of,
                  const int* __restrict__ cnt_cell, const int* __restrict__ first_cell,
                  int2* __restrict__ blocksum) {
  const int n = *n_hdr;
  const int base = blockIdx.x * kScanTile + threadIdx.x * kItems;
  int2 s = make_int2(0, 0);
#pragma unroll
  for (int q = 0; q < kItems; ++q) s = add2(s, first_point_item(base + q, n, cell_of, cnt_cell, first_cell));
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) s = add2(s, shfl_xor2(s, d));
  __shared__ int2 ws[32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (lane == 0) ws[wid] = s;
  __syncthreads();
  if (wid == 0) {
    int2 t = ws[lane];
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) t = add2(t, shfl_xor2(t, d));
    if (lane == 0) blocksum[blockIdx.x] = t;
  }
}

__global__ void __launch_bounds__(kScanThreads)
k_pillar_scan(const int* __restrict__ n_hdr, const int* __restrict__ cell_of,
              const int* __restrict__ cnt_cell, const int* __restrict__ first_cell,
              const int2* __restrict__ blocksum, int P, int* __restrict__ c2p,
              int* __restrict__ pillar_cell, int* __restrict__ pcnt_raw, int* __restrict__ poff,
              int* __restrict__ cursor, int* __restrict__ stats) {
  __shared__ int2 pre;
  __shared__ int2 tot;
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
  int2 it[kItems];
  int2 own = make_int2(0, 0);
#pragma unroll
  for (int q = 0; q < kItems; ++q) {
    it[q] = first_point_item(base + q, n, cell_of, cnt_cell, first_cell);
    own = add2(own, it[q]);
  }
  int2 run = block_excl_scan(own, &tot);
  run = add2(run, pre);
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
      }
    }
    run = add2(run, it[q]);
  }
  if (blockIdx.x == gridDim.x - 1 && threadIdx.x == 0) {
    const int total = pre.x + tot.x;
    stats[2] = total < P ? total : P;
  }
}

__global__ void k_pillar_fill(const int* __restrict__ n_hdr, const int* __restrict__ cell_of,
                              const int* __restrict__ c2p, int P, const int* __restrict__ poff,
                              int* __restrict__ cursor, int* __restrict__ list) {
  const int n = *n_hdr;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const int cell = cell_of[i];
  if (cell < 0) return;
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
k_pfn(const float4* __restrict__ pts, const int* __restrict__ stats_in,
      const int* __restrict__ pcnt_raw, const int* __restrict__ poff,
      const int* __restrict__ list, const int* __restrict__ pillar_cell,
      const float* __restrict__ w, const float* __restrict__ b, GridGeom g, int N,
      T* __restrict__ feat, int* __restrict__ pcount, int* __restrict__ stats) {
  __shared__ float sw[C * 9];
  __shared__ float sb[C];
  for (int j = threadIdx.x; j < C * 9; j += blockDim.x) sw[j] = w[j];
  for (int j = threadIdx.x; j < C; j += blockDim.x) sb[j] = b[j];
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int p = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int np = stats_in[2];
  if (p >= np) return;
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
  float f[9] = {q.x, q.y, q.z, q.w, q.x - mx, q.y - my, q.z - mz, q.x - xc, q.y - yc};
  float acc[C];
#pragma unroll
  for (int j = 0; j < C; ++j) {
    float s = sb[j];
#pragma unroll
    for (int d = 0; d < 9; ++d) s = fmaf(sw[j * 9 + d], f[d], s);
    acc[j] = valid ? relu_f(s) : 0.f;   // invalid lanes add 0: the max is >= 0 anyway
  }
  // reduce-scatter max over lanes: lane l ends with channels [l*C/32, (l+1)*C/32)
  int n = C;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const int h = n >> 1;
    const bool upper = (lane & off) != 0;
#pragma unroll
    for (int i = 0; i < C / 2; ++i) {
      if (i < h) {
        const float send = upper ? acc[i] : acc[i + h];
        const float keep = upper ? acc[i + h] : acc[i];
        acc[i] = fmaxf(keep, __shfl_xor_sync(kFull, send, off));
      }
    }
    n = h;
  }
  constexpr int PER = C / 32;
  T* dst = feat + (size_t)p * C + lane * PER;
#pragma unroll
  for (int i = 0; i < PER; ++i) dst[i] = Store<T>::from_f(acc[i]);
  if (lane == 0) {
    pcount[p] = m;
    atomicAdd(&stats[3], m);
    atomicAdd(&stats[6], raw - m);
    atomicAdd(&stats[7], raw);
  }
}

// One thread per (cell, 16-byte chunk): write the pillar's vector or zeros,
// publish cell2pillar, and restore the per-cell scratch.
template <int C>
__global__ void k_scatter(const int* __restrict__ stats_in, const int* __restrict__ c2p, int P,
                          const uint4* __restrict__ feat, int cells, int* __restrict__ cnt_cell,
                          int* __restrict__ first_cell, int* __restrict__ cell2pillar,
                          uint4* __restrict__ image) {
  constexpr int CH = C * 2 / 16;   // 16-byte chunks per cell (divides 32)
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  const int cell = t / CH, ch = t % CH;
  if (cell >= cells) return;     // all CH threads of a cell leave together
  const int cnt = cnt_cell[cell];
  int p = cnt > 0 ? c2p[cell] : -1;
  if (p >= P) p = -1;
  uint4 v = make_uint4(0, 0, 0, 0);
  if (p >= 0) v = feat[(size_t)p * CH + ch];
  image[(size_t)cell * CH + ch] = v;
  const int lane = threadIdx.x & 31;
  const unsigned grp = ((CH == 32) ? kFull : ((1u << CH) - 1u)) << (lane & ~(CH - 1));
  __syncwarp(grp);
  if (ch == 0) {
    cell2pillar[cell] = p;
    cnt_cell[cell] = 0;
    first_cell[cell] = kFirstInit;
  }
}

template <typename T, int C>
cudaError_t launch_all(const PillarBufs& b, const GridGeom& g, const float* pfn_w,
                       const float* pfn_b, cudaStream_t st) {
  const int cells = g.W * g.H;
  const int nblk = scan_blocks(b.cap);
  k_pillar_cells<<<(b.cap + 255) / 256, 256, 0, st>>>(b.pts, b.n_hdr, g, b.cell_of, b.cnt_cell,
                                                     b.first_cell, b.stats);
  k_pillar_blocksum<<<nblk, kScanThreads, 0, st>>>(b.n_hdr, b.cell_of, b.cnt_cell, b.first_cell,
                                                   b.blocksum);
  k_pillar_scan<<<nblk, kScanThreads, 0, st>>>(b.n_hdr, b.cell_of, b.cnt_cell, b.first_cell,
                                               b.blocksum, b.P, b.c2p, b.pillar_cell, b.pcnt_raw,
                                               b.poff, b.cursor, b.stats);
  k_pillar_fill<<<(b.cap + 255) / 256, 256, 0, st>>>(b.n_hdr, b.cell_of, b.c2p, b.P, b.poff,
                                                     b.cursor, b.list);
  k_pfn<T, C><<<(b.P + 7) / 8, 256, 0, st>>>(b.pts, b.stats, b.pcnt_raw, b.poff, b.list,
                                             b.pillar_cell, pfn_w, pfn_b, g, b.N,
                                             static_cast<T*>(b.feat), b.pcount, b.stats);
  constexpr int CH = C * 2 / 16;
  const long long thr = (long long)cells * CH;
  k_scatter<C><<<(unsigned)((thr + 255) / 256), 256, 0, st>>>(
      b.stats, b.c2p, b.P, static_cast<const uint4*>(b.feat), cells, b.cnt_cell, b.first_cell,
      b.cell2pillar, static_cast<uint4*>(b.image));
  return cudaGetLastError();
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

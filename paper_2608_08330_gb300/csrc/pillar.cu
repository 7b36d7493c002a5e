// Pillarisation, pillar feature net (PFN) and BEV scatter of one encoder
// branch E_k (the first stage of the per-agent encoder, Sec. III-B / Sec.
// V-A-1: a PointPillars encoder).
//
// The grouping is exactly the sequential rule "visit points in order; a new
// cell opens the next pillar id unless P_max pillars exist; a pillar keeps its
// first N_max points", computed in three kernels without order-dependent
// results:
//   1. cells:   per point its cell (float32 index arithmetic); per cell the
//               point count and the first point index (atomicAdd / atomicMin).
//               The value atomicAdd returns is the point's slot in its cell,
//               0 .. count-1: unique, in arbitrary order.
//   2. scan:    a point is a "first point" iff first[cell] == i.  A single-pass
//               exclusive scan of (first-point flag, count of its cell) over
//               point order gives each touched cell its pillar id (the rank of
//               its first occurrence) and the offset of its point list.  Each
//               tile of 1024 points publishes its aggregate and adds those of
//               all earlier tiles (no grid-wide barrier); once a tile has
//               written its cells' (id, offset) records it raises a flag, and
//               every point of a kept pillar then reads its cell's record
//               (after the flags of the tiles holding its cell's first point)
//               and stores itself at offset + slot: the point itself when its
//               pillar keeps all its points, its index otherwise.
//   3. PFN:     one warp per kept pillar.  A pillar of at most N_max points has
//               them all in its list (one per lane, slot order); a larger one
//               selects the N_max smallest indices of its list (warp bitonic
//               sort / merge), i.e. its first N_max points in point order.  The
//               means are fixed-point sums (exact integer adds, so their value
//               does not depend on the lanes' order); each lane owns
//               C/32 output channels and folds the kept points in one at a time
//               (broadcast by shuffle): the linear map of the 9-d decorated
//               features, rewritten as 4 per-point terms plus a per-pillar
//               constant, ReLU, running max (order-free).  The result is
//               therefore run-to-run deterministic.
//   Image:     the PFN writes each kept pillar's vector into its cell of the
//               pseudo-image and its id into cell2pillar (each cell has at most
//               one pillar: no atomics).  Elsewhere the image holds zeros and
//               cell2pillar -1: the first kernel of a pass clears the cells the
//               previous pass wrote (np_prev of them), and the PFN, which runs
//               after the scan (the last reader of the per-cell counters),
//               restores the counters of every cell the pass touched.
#include <climits>
#include <cmath>
#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace rtcc {

namespace {

constexpr unsigned kFull = 0xFFFFFFFFu;
constexpr int kItems = 4;                          // consecutive points per scan thread
constexpr int kPfnWarps = 8;                       // PFN block: 256 threads, a pillar per warp

// Pointers to data an earlier kernel of the chain writes are not __restrict__:
// a read through a const __restrict__ pointer may be scheduled above
// griddepcontrol.wait (the qualifier promises the data does not change while
// the kernel runs), and would then read the predecessor's output before it is
// complete.  Only the constant PFN weights keep the qualifier.

__device__ __forceinline__ void st_release_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.release.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void fence_acq_rel_gpu() {
  asm volatile("fence.acq_rel.gpu;" ::: "memory");
}

// A tile's aggregate in one 64-bit word: bit 63 = published, bits 32..62 = the
// tile's first points, bits 0..31 = the points of their cells.
__device__ __forceinline__ unsigned long long pack_agg(int2 a) {
  return (1ull << 63) | ((unsigned long long)(unsigned)a.x << 32) | (unsigned)a.y;
}
__device__ __forceinline__ int2 unpack_agg(unsigned long long w) {
  return make_int2((int)((w >> 32) & 0x7FFFFFFFu), (int)(w & 0xFFFFFFFFu));
}

template <int CH>
__global__ void __launch_bounds__(256) k_pillar_cells(const PillarBufs b, const GridGeom g,
                                                      int ntiles) {
  __shared__ int s_n;
  pdl_trigger();
  pdl_wait();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  // Independent loads first: the count (one read of the header per block),
  // the previous pass's pillar count and, from the device slot (which holds
  // cap points), the point, so that it need not wait for the count.  With a
  // zero-copy payload the header and the points come from the source (pinned
  // host memory; only the n valid points are read) and are copied to the
  // device slot the later kernels read.
  if (threadIdx.x == 0) s_n = b.src_hdr ? *b.src_hdr : *b.n_hdr;
  float4 p = (!b.src_pts && i < b.cap) ? b.pts[i] : make_float4(0.f, 0.f, 0.f, 0.f);
  const int npv = b.clear_all ? 0 : *b.np_prev;
  __syncthreads();
  const int n = s_n;
  if (b.src_pts && i < n) p = b.src_pts[i];
  // per-pass words: the stats (word 0 = n) and the caller's counters that
  // follow them; the scan's tile words
  if (i < b.n_zero) b.zero_words[i] = i == 0 ? n : 0;
  if (i < ntiles) b.tile_agg[(size_t)i * kAggStride] = 0ull;
  if (i == 0 && b.dst_hdr) *b.dst_hdr = n;
  if (i == 0 && b.present_flag) *b.present_flag = 1;   // this agent's slot is filled this frame
  // the previous pass's pillar cell this thread clears first (loaded ahead of
  // the atomics below, so that the two round trips overlap)
  const long long stride = (long long)gridDim.x * blockDim.x;
  const long long tot_prev = (long long)npv * CH;
  const int c_prev = (!b.clear_all && i < tot_prev) ? b.pillar_cell[i / CH] : -1;
  int cell = -1, slot = 0;
  if (i < n) {
    if (b.dst_pts) b.dst_pts[i] = p;
    // IEEE float32 subtraction and division with round-to-nearest.
    const float fx = __fdiv_rn(__fsub_rn(p.x, g.x_min), g.v);
    const float fy = __fdiv_rn(__fsub_rn(p.y, g.y_min), g.v);
    const bool ok = (p.z >= g.z_min) && (p.z < g.z_max) && (fx >= 0.f) && (fx < (float)g.W) &&
                    (fy >= 0.f) && (fy < (float)g.H);
    if (ok) {
      const int ix = (int)floorf(fx);
      const int iy = (int)floorf(fy);
      cell = iy * g.W + ix;
      slot = atomicAdd(&b.cnt_cell[cell], 1);
      atomicMin(&b.first_cell[cell], i);
    }
  }
  // clear what the previous pass wrote (CH 16-byte chunks per cell)
  {
    uint4* image = static_cast<uint4*>(b.image);
    const unsigned cells = (unsigned)(g.W * g.H);
    if (b.clear_all) {
      const long long tot = (long long)g.W * g.H * CH;
      for (long long q = i; q < tot; q += stride) {
        image[q] = make_uint4(0u, 0u, 0u, 0u);
        if (q % CH == 0) b.cell2pillar[q / CH] = -1;
      }
    } else {
      for (long long q = i; q < tot_prev; q += stride) {
        const int c = q == i ? c_prev : b.pillar_cell[q / CH];
        if ((unsigned)c >= cells) continue;      // only after a wait ran out
        image[(size_t)c * CH + q % CH] = make_uint4(0u, 0u, 0u, 0u);
        if (q % CH == 0) b.cell2pillar[c] = -1;
      }
    }
  }
  if (i < n) {
    b.cell_of[i] = cell;
    b.slot_of[i] = slot;
  }
}

__device__ __forceinline__ int2 add2(int2 a, int2 b) { return make_int2(a.x + b.x, a.y + b.y); }

__device__ __forceinline__ int2 shfl_up2(int2 v, int d) {
  return make_int2(__shfl_up_sync(kFull, v.x, d), __shfl_up_sync(kFull, v.y, d));
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

// Single-pass scan of (first-point flag, count of its cell) over point order,
// fused with the fill of the pillars' points.  A tile first writes, for each
// cell whose first point it holds, the cell's rank and count offset within
// the tile (cell_loc), then publishes its aggregate with release semantics.
// It then reads every earlier tile's aggregate (acquire), which gives it the
// exclusive prefix of each earlier tile; a point of a cell opened in tile f
// reads cell_loc and adds tile f's prefix to get its pillar id and list
// offset.  Every block stays resident (cooperative launch) and takes the
// tiles blockIdx, blockIdx + grid, ... in order; a tile waits only for
// earlier tiles' aggregates, published before any wait, so the waits always
// end.  Same-address atomics serialise in L2, so the pass's counters are
// summed per tile and added once per tile.
__global__ void __launch_bounds__(1024, 1)
k_pillar_scan(const PillarBufs b, int ntiles, int W) {
  const int kTile = kItems * blockDim.x;
  extern __shared__ int2 s_tpre[];               // [ntiles] exclusive prefix of each tile
  __shared__ int2 s_tot;
  __shared__ int s_red[32][3];
  pdl_trigger();
  pdl_wait();
  const int n = *b.n_hdr;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  bool ok = true;                                 // no record out of range
  bool wok = true;                                // warp 0: every wait ended in time
  for (int t = blockIdx.x; t < ntiles; t += gridDim.x) {
    const int base = t * kTile + threadIdx.x * kItems;
    // the scratch holds whole tiles: the vector loads stay inside it
    const int4 c4 = *reinterpret_cast<const int4*>(b.cell_of + base);
    const int4 s4 = *reinterpret_cast<const int4*>(b.slot_of + base);
    int cell[kItems] = {c4.x, c4.y, c4.z, c4.w};
    const int slot[kItems] = {s4.x, s4.y, s4.z, s4.w};
    int cc[kItems];
    bool first[kItems];
#pragma unroll
    for (int q = 0; q < kItems; ++q) {
      if (base + q >= n) cell[q] = -1;
      const int fc = cell[q] >= 0 ? b.first_cell[cell[q]] : -1;
      cc[q] = cell[q] >= 0 ? b.cnt_cell[cell[q]] : 0;
      first[q] = cell[q] >= 0 && fc == base + q;
    }
    int2 own = make_int2(0, 0);
#pragma unroll
    for (int q = 0; q < kItems; ++q) own = add2(own, first[q] ? make_int2(1, cc[q]) : make_int2(0, 0));
    int2 run = block_excl_scan(own, &s_tot);      // within the tile
    const int2 tot = s_tot;
    // the tile-local records of the cells this tile opens
    {
      int2 r = run;
#pragma unroll
      for (int q = 0; q < kItems; ++q) {
        if (first[q]) {
          b.cell_loc[cell[q]] = make_int2((t << 12) | r.x, r.y);
          r = add2(r, make_int2(1, cc[q]));
        }
      }
    }
    __syncthreads();                              // the records precede the release below
    if (threadIdx.x == 0) st_release_u64(&b.tile_agg[(size_t)t * kAggStride], pack_agg(tot));
    // every earlier tile's exclusive prefix (and so this tile's)
    if (wid == 0) {
      int2 carry = make_int2(0, 0);
      for (int j0 = 0; j0 < t; j0 += 128) {
        unsigned long long wv[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          const int j = j0 + r * 32 + lane;
          wv[r] = j < t ? ld_relaxed_u64(&b.tile_agg[(size_t)j * kAggStride]) : (1ull << 63);
        }
        // poll the unpublished words together: one round trip per round
        const long long t0 = clock64();
        while (wok) {                             // wok is uniform across warp 0
          bool all = true;
#pragma unroll
          for (int r = 0; r < 4; ++r) all = all && (wv[r] >> 63);
          if (__all_sync(kFull, all)) break;
          if (__any_sync(kFull, clock64() - t0 > kWaitBudgetCycles)) wok = false;
#pragma unroll
          for (int r = 0; r < 4; ++r)
            if (!(wv[r] >> 63))
              wv[r] = ld_relaxed_u64(&b.tile_agg[(size_t)(j0 + r * 32 + lane) * kAggStride]);
        }
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          const int j = j0 + r * 32 + lane;
          const int2 a = j < t ? unpack_agg(wv[r]) : make_int2(0, 0);
          int2 inc = a;
#pragma unroll
          for (int d = 1; d < 32; d <<= 1) {
            const int2 o = shfl_up2(inc, d);
            if (lane >= d) inc = add2(inc, o);
          }
          if (j < t) s_tpre[j] = add2(carry, make_int2(inc.x - a.x, inc.y - a.y));
          carry = add2(carry, make_int2(__shfl_sync(kFull, inc.x, 31), __shfl_sync(kFull, inc.y, 31)));
        }
      }
      if (lane == 0) s_tpre[t] = carry;
      fence_acq_rel_gpu();                        // acquire: the earlier tiles' cell records
    }
    __syncthreads();
    const int2 pre = s_tpre[t];
    run = add2(run, pre);
    // pillar records, the fill, the pass's counters.  Every load comes before
    // the first store: a store may alias a later load, which could then not
    // be issued ahead of it.
    int2 loc[kItems];
    float4 pt[kItems];
#pragma unroll
    for (int q = 0; q < kItems; ++q) {
      const bool other = cell[q] >= 0 && !first[q];
      loc[q] = other ? b.cell_loc[cell[q]] : make_int2(0, 0);
      pt[q] = (cell[q] >= 0 && cc[q] <= b.N) ? b.pts[base + q] : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    int inr = 0, kept = 0, rawk = 0;
#pragma unroll
    for (int q = 0; q < kItems; ++q) {
      if (cell[q] < 0) continue;
      ++inr;
      const int i = base + q;
      const bool whole = cc[q] <= b.N;
      int pid, off;
      if (first[q]) {
        pid = run.x;
        off = run.y;
        run = add2(run, make_int2(1, cc[q]));
        b.touched[pid] = cell[q];
        if (pid < b.P) {
          b.pillar_rec[pid] = make_int4(cell[q], cc[q], off, (cell[q] % W) | ((cell[q] / W) << 16));
          b.pillar_cell[pid] = cell[q];
          kept += cc[q] < b.N ? cc[q] : b.N;
          rawk += cc[q];
        }
      } else {
        const int2 r = loc[q];
        const int f = r.x >> 12;
        if (f > t) {                              // only after a wait ran out
          ok = false;
          continue;
        }
        const int2 fp = s_tpre[f];
        pid = fp.x + (r.x & 4095);
        off = fp.y + r.y;
      }
      if (pid < b.P) {
        if (whole) {
          b.bucket[(size_t)pid * b.N + slot[q]] = pt[q];
        } else if ((unsigned)(off + slot[q]) < (unsigned)b.cap) {
          b.list[off + slot[q]] = i;
        } else {
          ok = false;                             // only after a wait ran out
        }
      }
    }
    // counters 1 (points in the grid), 3 (kept points), 6 (dropped by the
    // per-pillar cap), 7 (points of kept pillars)
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) {
      inr += __shfl_xor_sync(kFull, inr, d);
      kept += __shfl_xor_sync(kFull, kept, d);
      rawk += __shfl_xor_sync(kFull, rawk, d);
    }
    if (lane == 0) {
      s_red[wid][0] = inr;
      s_red[wid][1] = kept;
      s_red[wid][2] = rawk;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int a0 = 0, a1 = 0, a2 = 0;
      for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
        a0 += s_red[w][0];
        a1 += s_red[w][1];
        a2 += s_red[w][2];
      }
      if (a0) atomicAdd(&b.stats[1], a0);
      if (a2) {
        atomicAdd(&b.stats[3], a1);
        atomicAdd(&b.stats[6], a2 - a1);
        atomicAdd(&b.stats[7], a2);
      }
      if (t == ntiles - 1) {
        const int total = pre.x + tot.x;         // pillars of the pass, kept or not
        b.stats[2] = total < b.P ? total : b.P;
        *b.ntouched = total;
      }
    }
    __syncthreads();                              // shared words are reused by the next tile
  }
  if (!(ok && wok) && b.err) atomicOr(b.err, ERR_WAIT_PILLAR);
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


// The PFN of one pillar by the lanes in `mask` (a whole warp, or one half):
// NL lanes, lane l of them owns channels [l*PER, (l+1)*PER) (PER = C / NL).
// q0 / q1: this lane's points (slots l and l + NL of the pillar; zeros past
// m).  The pillar's kept points are written to `sp` and read back one at a
// time (a shared-memory broadcast).
//
// The 9 decorated features (x, y, z, i, x - mx, y - my, z - mz, x - xc,
// y - yc) are affine in the point's (dx, dy, z, i) = (x - xc, y - yc, z, i):
//   W f = (W0 + W4 + W7) dx + (W1 + W5 + W8) dy + (W2 + W6) z + W3 i
//       + [W0 xc + W1 yc - W4 (mx - xc) - W5 (my - yc) - W6 mz],
// the bracket the same for every point of the pillar.  Folding it into the
// bias leaves 4 FMAs per point and channel instead of 9, in fp32 throughout;
// ReLU folds into the running max, which starts at 0 (m >= 1).
template <typename T, int C, int NL>
__device__ __forceinline__ void pfn_pillar(const PillarBufs& b, const GridGeom& g,
                                           const float4* s_wf, const float4* s_wk,
                                           const float2* s_wb, float4* sp, unsigned mask,
                                           int l, int p, int4 rec, float4 q0, float4 q1, int m) {
  constexpr int PER = C / NL;
  constexpr int HP = C / 16;                      // see wpos
  const int cell = rec.x;
  const int cx = rec.w & 0xFFFF, cy = rec.w >> 16;
  const float xc = __fadd_rn(g.x_min, __fmul_rn((float)cx + 0.5f, g.v));
  const float yc = __fadd_rn(g.y_min, __fmul_rn((float)cy + 0.5f, g.v));
  const float dx0 = __fsub_rn(q0.x, xc), dy0 = __fsub_rn(q0.y, yc);
  const float dx1 = __fsub_rn(q1.x, xc), dy1 = __fsub_rn(q1.y, yc);
  // The means, as offsets from the pillar centre (x, y) and from z_min (z):
  // sums in fixed point (|x - xc|, |y - yc| < v; 0 <= z - z_min <= the z
  // range; the scales keep 32 terms below 2^30), exact integer adds whose
  // value does not depend on the lanes' order, rounded once to float32 and
  // scaled by 1 / m.
  const bool a0 = l < m, a1 = l + NL < m;
  int sx = (a0 ? __float2int_rn(__fmul_rn(dx0, g.qxy)) : 0) +
           (a1 ? __float2int_rn(__fmul_rn(dx1, g.qxy)) : 0);
  int sy = (a0 ? __float2int_rn(__fmul_rn(dy0, g.qxy)) : 0) +
           (a1 ? __float2int_rn(__fmul_rn(dy1, g.qxy)) : 0);
  int sz = (a0 ? __float2int_rn(__fmul_rn(__fsub_rn(q0.z, g.z_min), g.qz)) : 0) +
           (a1 ? __float2int_rn(__fmul_rn(__fsub_rn(q1.z, g.z_min), g.qz)) : 0);
#pragma unroll
  for (int d = NL / 2; d > 0; d >>= 1) {
    sx += __shfl_xor_sync(mask, sx, d);
    sy += __shfl_xor_sync(mask, sy, d);
    sz += __shfl_xor_sync(mask, sz, d);
  }
  const float inv_m = __frcp_rn((float)m);
  const float mdx = __fmul_rn(__fmul_rn(__int2float_rn(sx), g.qxy_inv), inv_m);
  const float mdy = __fmul_rn(__fmul_rn(__int2float_rn(sy), g.qxy_inv), inv_m);
  const float mz = __fadd_rn(g.z_min, __fmul_rn(__fmul_rn(__int2float_rn(sz), g.qz_inv), inv_m));
  sp[l] = make_float4(dx0, dy0, q0.z, q0.w);
  if (NL < 32) sp[l + NL] = make_float4(dx1, dy1, q1.z, q1.w);
  __syncwarp(mask);
  float4 wf[PER];
  float cst[PER], acc[PER];
#pragma unroll
  for (int i = 0; i < PER; ++i) {
    const int ch = l * PER + i;
    const int wp = (ch % HP) * 16 + ch / HP;      // wpos(ch)
    wf[i] = s_wf[wp];
    const float4 k = s_wk[wp];
    const float2 kb = s_wb[wp];
    float c = kb.y;
    c = fmaf(k.x, xc, c);
    c = fmaf(k.y, yc, c);
    c = fmaf(-k.z, mdx, c);
    c = fmaf(-k.w, mdy, c);
    c = fmaf(-kb.x, mz, c);
    cst[i] = c;
    acc[i] = 0.f;
  }
  for (int j = 0; j < m; ++j) {
    const float4 d = sp[j];
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      float s = fmaf(wf[i].x, d.x, cst[i]);
      s = fmaf(wf[i].y, d.y, s);
      s = fmaf(wf[i].z, d.z, s);
      s = fmaf(wf[i].w, d.w, s);
      acc[i] = fmaxf(acc[i], s);
    }
  }
  __syncwarp(mask);                               // sp may be reused after this
  // the pillar's vector goes straight into its cell of the pseudo-image (a
  // canonical +0 where every term was non-positive)
  T* dst = static_cast<T*>(b.image) + (size_t)cell * C + l * PER;
  if constexpr (PER == 1) {
    dst[0] = Store<T>::from_f(relu_f(acc[0]));
  } else {
    uint32_t pk[PER / 2];
#pragma unroll
    for (int i = 0; i < PER / 2; ++i)
      pk[i] = Store<T>::pack2(relu_f(acc[2 * i]), relu_f(acc[2 * i + 1]));
    if constexpr (PER == 2) {
      *reinterpret_cast<uint32_t*>(dst) = pk[0];
    } else if constexpr (PER == 4) {
      *reinterpret_cast<uint2*>(dst) = make_uint2(pk[0], pk[1]);
    } else {
#pragma unroll
      for (int i = 0; i < PER / 2; ++i) reinterpret_cast<uint32_t*>(dst)[i] = pk[i];
    }
  }
  if (l == 0) {
    b.cell2pillar[cell] = p;
    b.pcount[p] = m;
  }
}

// One warp per two pillars.  When neither has more than N_max points (all
// its points kept, no selection), each half-warp takes one; otherwise the
// whole warp takes them one after the other, selecting the N_max smallest
// point indices (warp bitonic sort / merge) where a pillar has more.
template <typename T, int C>
__global__ void __launch_bounds__(256, 5)
k_pfn(const PillarBufs b, const float* __restrict__ w, const float* __restrict__ bias,
      const GridGeom g) {
  // Per channel ch the folded weights sit at wpos(ch) = (ch % HP) * 16 + ch /
  // HP (HP = C / 16): the 16 lanes of a half-warp, which own channels l * HP
  // + i, read 16 consecutive entries for each i (no bank conflicts).  The
  // points of the two half-warps' pillars sit 33 entries apart (different
  // banks when both halves read one).
  __shared__ float4 s_wf[C];
  __shared__ float4 s_wk[C];
  __shared__ float2 s_wb[C];
  __shared__ float4 s_pts[kPfnWarps][2][33];
  pdl_trigger();
  for (int c = threadIdx.x; c < C; c += blockDim.x) {      // weights: constant
    const float* wr = w + c * 9;
    const int wp = (c % (C / 16)) * 16 + c / (C / 16);
    s_wf[wp] = make_float4(wr[0] + wr[4] + wr[7], wr[1] + wr[5] + wr[8], wr[2] + wr[6], wr[3]);
    s_wk[wp] = make_float4(wr[0], wr[1], wr[4], wr[5]);
    s_wb[wp] = make_float2(wr[6], bias[c]);
  }
  pdl_wait();
  span_begin(b.pfn_span);
  __syncthreads();
  const int gid = blockIdx.x * blockDim.x + threadIdx.x;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int h = lane >> 4, hl = lane & 15;
  const int p = (gid >> 5) * 2 + h;               // this half's pillar
  const int np = b.stats[2];
  const int nt = *b.ntouched;
  const int N = b.N;
  const int cells = g.W * g.H;
  const int4 rec = p < b.P ? b.pillar_rec[p] : make_int4(0, 0, 0, 0);
  // the first points of the pillar's bucket, read with its record (most
  // pillars hold at most kSpec points)
  constexpr int kSpec = 8;
  float4 q0 = (p < b.P && hl < kSpec && hl < N) ? b.bucket[(size_t)p * N + hl]
                                                 : make_float4(0.f, 0.f, 0.f, 0.f);
  // the first cell whose counters this thread restores (see below)
  const int t0 = gid < b.cap ? b.touched[gid] : -1;
  const bool sane = (unsigned)rec.x < (unsigned)cells && rec.y >= 1 && rec.z >= 0 &&
                    rec.z <= b.cap - rec.y;
  const bool act = p < np && sane;
  if (p < np && !sane && hl == 0 && b.err) atomicOr(b.err, ERR_BOUNDS);
  const float4 z4 = make_float4(0.f, 0.f, 0.f, 0.f);
  if (__all_sync(kFull, !act || rec.y <= N)) {
    if (act) {
      const int m = rec.y;                        // every point kept
      if (hl >= m) q0 = z4;
      else if (hl >= kSpec) q0 = b.bucket[(size_t)p * N + hl];
      const float4 q1 = hl + 16 < m ? b.bucket[(size_t)p * N + hl + 16] : z4;
      pfn_pillar<T, C, 16>(b, g, s_wf, s_wk, s_wb, s_pts[wid][h], 0xFFFFu << (16 * h), hl, p,
                           rec, q0, q1, m);
    }
  } else {
    for (int k = 0; k < 2; ++k) {
      const int pk = (gid >> 5) * 2 + k;
      const int4 rk = make_int4(__shfl_sync(kFull, rec.x, 16 * k), __shfl_sync(kFull, rec.y, 16 * k),
                                __shfl_sync(kFull, rec.z, 16 * k), __shfl_sync(kFull, rec.w, 16 * k));
      if (!__shfl_sync(kFull, act, 16 * k)) continue;
      const int raw = rk.y, base = rk.z;
      const int m = raw < N ? raw : N;
      float4 q;
      if (raw <= N) {
        q = lane < raw ? b.bucket[(size_t)pk * N + lane] : z4;
      } else {
        // the N smallest point indices of the list = the pillar's first points
        int idx = lane < raw ? b.list[base + lane] : INT_MAX;
        idx = warp_sort_asc(idx, lane);
        for (int c = 32; c < raw; c += 32) {
          int v = (c + lane < raw) ? b.list[base + c + lane] : INT_MAX;
          v = warp_sort_asc(v, lane);
          const int vr = __shfl_sync(kFull, v, 31 - lane);
          idx = warp_merge_asc(min(idx, vr), lane);
        }
        q = (lane < m && (unsigned)idx < (unsigned)b.cap) ? b.pts[idx] : z4;
      }
      pfn_pillar<T, C, 32>(b, g, s_wf, s_wk, s_wb, s_pts[wid][0], kFull, lane, pk, rk, q, z4, m);
    }
  }
  // the scan was the last reader of the per-cell counters: restore those of
  // every cell this pass touched for the next pass
  for (int j = gid; j < nt; j += gridDim.x * blockDim.x) {
    const int c = j == gid ? t0 : b.touched[j];
    if ((unsigned)c >= (unsigned)cells) continue;   // only after a scan wait ran out
    b.cnt_cell[c] = 0;
    b.first_cell[c] = kFirstInit;
  }
  if (gid == 0) *b.np_prev = np;                 // cleared by the next pass
  if (b.pfn_span) {
    __syncthreads();
    span_end(b.pfn_span);
  }
}

int sm_count() {
  static std::once_flag once;
  static int sms = 0;
  std::call_once(once, [] {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      sms = 0;
  });
  return sms;
}

// Launch the scan with `threads` threads per block (a multiple of 32, 256 to
// 1024): a cooperative launch (every block resident at once), at most as many
// blocks as fit.
cudaError_t launch_scan(const PillarBufs& b, int W, int threads, cudaStream_t st) {
  static std::mutex mu;
  static size_t attr_set = 48 * 1024;             // the default dynamic limit
  const int tile = kItems * threads;
  const int ntiles = b.cap > 0 ? (b.cap + tile - 1) / tile : 1;
  const size_t smem = (size_t)ntiles * sizeof(int2);
  {
    std::lock_guard<std::mutex> lk(mu);
    if (smem > attr_set) {
      cudaError_t e = cudaFuncSetAttribute(k_pillar_scan,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e != cudaSuccess) return e;
      attr_set = smem;
    }
  }
  int per = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, k_pillar_scan, threads, smem);
  if (e != cudaSuccess) return e;
  const int cap_blocks = per * sm_count();
  if (cap_blocks < 1 || ntiles >= (1 << 19)) return cudaErrorInvalidValue;
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3(ntiles < cap_blocks ? ntiles : cap_blocks);
  lc.blockDim = dim3(threads);
  lc.dynamicSmemBytes = smem;
  lc.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;     // a tile waits on earlier tiles' blocks
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  lc.attrs = attr;
  lc.numAttrs = 2;
  return cudaLaunchKernelEx(&lc, k_pillar_scan, b, ntiles, W);
}

template <typename T, int C>
cudaError_t launch_all(const PillarBufs& b, const GridGeom& g0, const float* pfn_w,
                       const float* pfn_b, cudaStream_t st) {
  GridGeom g = g0;
  g.qxy = std::ldexp(1.f, std::ilogb(33554432.0 / g.v));                 // 2^25 / v
  g.qz = std::ldexp(1.f, std::ilogb(33554432.0 / ((double)g.z_max - g.z_min)));
  g.qxy_inv = 1.f / g.qxy;                                                // exact: powers of two
  g.qz_inv = 1.f / g.qz;
  const int sms = sm_count();
  if (sms < 1 || b.stats != b.zero_words || b.n_zero < 8) return cudaErrorInvalidValue;
  constexpr int CH = C * 2 / 16;                  // 16-byte chunks per cell
  const int ntiles_max = scan_tiles(b.cap);       // the tile words the first kernel clears
  const int cells_threads = b.cap > ntiles_max ? b.cap : ntiles_max;
  cudaError_t e = launch_pdl(k_pillar_cells<CH>, dim3((cells_threads + 255) / 256), dim3(256), 0,
                             st, b, g, ntiles_max);
  if (e != cudaSuccess) return e;
  // the scan: the smallest block (a multiple of 32 threads, at least 256)
  // whose tiles fit one block per SM (two scan blocks on one SM delay each
  // other's publication), at most 1024 threads
  const long long pts = b.cap > 0 ? b.cap : 1;
  long long warps = (pts + 4LL * 32 * sms - 1) / (4LL * 32 * sms);
  warps = warps < 8 ? 8 : (warps > 32 ? 32 : warps);
  e = launch_scan(b, g.W, (int)warps * 32, st);
  if (e != cudaSuccess) return e;
  return launch_pdl(k_pfn<T, C>, dim3((b.P + 15) / 16), dim3(256), 0, st, b, pfn_w, pfn_b, g);
}

}  // namespace

cudaError_t launch_pillarise(const PillarBufs& b, const GridGeom& g, const float* pfn_w,
                             const float* pfn_b, bool bf16, cudaStream_t st) {
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

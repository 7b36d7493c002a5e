// Max fusion of the agents' BEV feature slots followed by the 1x1 detection
// head, on the 5th-generation tensor cores (the shared post-join subgraph,
// Sec. III-B / Sec. IV-D, with the element-wise max fusion).
//
//   F[cell][c]   = max over present agents k of X_k[cell][c]
//   out[cell][o] = b[o] + sum_c W[o][c] F[cell][c],   o < 16
//
// The head is a GEMM with M = cells, N = 16, K = C.  One work item is a tile
// of 128 consecutive cells.  For each 64- (or 32-) channel chunk of the tile,
// TMA loads the chunk of every present agent's slot into one pipeline stage
// (one 3-D box over all K consecutive slots when every agent is present, one
// box per present agent otherwise), all with the same 128-byte (64-byte)
// swizzle; because the max is taken
// position by position, the max of the swizzled agent tiles is the swizzled
// fused tile, i.e. directly the A operand of tcgen05.mma.  B is the head
// weight matrix [16][C] (K-major, loaded once per CTA).  The accumulator is 16
// fp32 columns of tensor memory; the epilogue adds the bias and writes the
// head output and, per anchor, the decode key (the class logit mapped to an
// unsigned integer whose ascending order is descending logit order, or
// 0xFFFFFFFF below the threshold) with a histogram of its top 12 bits.
//
// Roles (320 threads): warp 0 = TMA producer, warp 1 = tensor-memory owner and
// MMA issuer, warps 2..9 = max workers, of which warps 2..5 (one tensor-memory
// lane quarter each) also run the epilogue.  The workers write the
// max into one of two fused-chunk buffers and release the agent stage at
// once, so the producer refills it while the MMA still reads the fused chunk.  The slots hold ReLU
// outputs, so the 16-bit max is exact and matches the agent-index-order max;
// the MMA's summation order is fixed by the hardware, so the output is
// bit-reproducible.  Every wait is bounded (an error bit, no hang).
#include "common.cuh"
#include "kernels.h"

namespace rtcc {

namespace {

constexpr int kThreads = 320;
constexpr int kWorkers = kThreads - 64;        // warps 2..9 take the max; warps 2..5 the epilogue
constexpr int kTile = 128;                     // cells per work item (MMA M)
constexpr int kMaxStages = 8;
constexpr int kMaxC = 512;
// The agent-chunk stages and the two fused chunks (the MMA's A operand, 128
// rows of bkc channels each) share one area, so 32-channel chunks leave room
// for more stages.
constexpr int kArea = 208 * 1024;
__host__ __device__ constexpr int fused_bytes(int bkc) { return kTile * bkc * 2; }
__host__ __device__ constexpr int stage_area(int bkc) { return kArea - 2 * fused_bytes(bkc); }
constexpr int kWBytes = kFuseHeadOut * kMaxC * 2;
constexpr int kSmem = kArea + kWBytes + 1024 + 256;
static_assert(kSmem <= 227 * 1024, "shared memory budget");

template <typename T>
__device__ __forceinline__ uint32_t max2(uint32_t a, uint32_t b);
template <>
__device__ __forceinline__ uint32_t max2<__half>(uint32_t a, uint32_t b) {
  __half2 r = __hmax2(*reinterpret_cast<__half2*>(&a), *reinterpret_cast<__half2*>(&b));
  return *reinterpret_cast<uint32_t*>(&r);
}
template <>
__device__ __forceinline__ uint32_t max2<__nv_bfloat16>(uint32_t a, uint32_t b) {
  __nv_bfloat162 r =
      __hmax2(*reinterpret_cast<__nv_bfloat162*>(&a), *reinterpret_cast<__nv_bfloat162*>(&b));
  return *reinterpret_cast<uint32_t*>(&r);
}
template <typename T>
__device__ __forceinline__ uint4 max8(uint4 a, uint4 b) {
  return make_uint4(max2<T>(a.x, b.x), max2<T>(a.y, b.y), max2<T>(a.z, b.z), max2<T>(a.w, b.w));
}

// ascending unsigned order of the result == descending float order; -0 -> +0
__device__ __forceinline__ uint32_t ord_desc(float f) {
  f = f + 0.0f;
  const uint32_t u = __float_as_uint(f);
  const uint32_t asc = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ~asc;
}

// Count `key` (if `keep`) in the top-12-bit histogram: the lanes of a warp
// that share a bin add their count with one atomic (valid logits crowd into
// a few dozen bins, so per-key atomics would serialise on them).  Every lane
// of the warp must call it.
__device__ __forceinline__ void hist_add(uint32_t* hist0, bool keep, uint32_t key, int lane) {
  const uint32_t bin = keep ? (key >> 20) : 0xFFFFFFFFu;
  const unsigned peers = __match_any_sync(0xFFFFFFFFu, bin);
  if (keep && lane == __ffs(peers) - 1) atomicAdd(&hist0[bin], (uint32_t)__popc(peers));
}

// Element-wise max of the KP present agents' copies of one staged chunk (nvec
// 16-byte vectors each, agent i at st + i * nvec) into fb, by the worker
// threads; 0 agents give zeros.  KP fixed at compile time lets the loads of
// two vectors be in flight together.
template <typename T, int KP>
__device__ __forceinline__ void max_chunk(const uint4* __restrict__ st, uint4* __restrict__ fb,
                                          int nvec, int wt) {
#pragma unroll 2
  for (int v = wt; v < nvec; v += kWorkers) {
    uint4 m = make_uint4(0u, 0u, 0u, 0u);
    if (KP > 0) m = st[v];
#pragma unroll
    for (int i = 1; i < KP; ++i) m = max8<T>(m, st[i * nvec + v]);
    fb[v] = m;
  }
}
template <typename T>
__device__ __forceinline__ void max_chunk_any(const uint4* st, uint4* fb, int nvec, int wt, int kp) {
  switch (kp) {
    case 0: max_chunk<T, 0>(st, fb, nvec, wt); break;
    case 1: max_chunk<T, 1>(st, fb, nvec, wt); break;
    case 2: max_chunk<T, 2>(st, fb, nvec, wt); break;
    case 3: max_chunk<T, 3>(st, fb, nvec, wt); break;
    case 4: max_chunk<T, 4>(st, fb, nvec, wt); break;
    default:
      for (int v = wt; v < nvec; v += kWorkers) {
        uint4 m = st[v];
        for (int i = 1; i < kp; ++i) m = max8<T>(m, st[i * nvec + v]);
        fb[v] = m;
      }
  }
}

template <typename T>
__global__ void __launch_bounds__(kThreads, 1) k_fuse_max_head(const __grid_constant__ FuseTcParams P) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int fbytes = fused_bytes(P.bkc);
  uint8_t* fbuf = smem + stage_area(P.bkc);    // [2] fused chunks (the MMA's A operand)
  uint8_t* wsm = smem + kArea;                 // head weights [C / bkc][16][bkc]
  uint64_t* full = reinterpret_cast<uint64_t*>(wsm + kWBytes);   // [kMaxStages] agent chunks landed
  uint64_t* empty = full + kMaxStages;         // [kMaxStages] workers have read the stage
  uint64_t* fready = empty + kMaxStages;       // [2] fused chunk written
  uint64_t* fempty = fready + 2;               // [2] MMA has read the fused chunk
  uint64_t* accfull = fempty + 2;              // [2]
  uint64_t* accempty = accfull + 2;            // [2] (4 arrivals)
  uint64_t* wbar = accempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(wbar + 1);
  __shared__ int s_list[RTCC_MAX_AGENTS];
  __shared__ int s_kp;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int C = P.C, bkc = P.bkc;
  const int nch = C / bkc;
  const int slot_bytes = kTile * bkc * 2;
  const int stage_bytes = P.K * slot_bytes;    // room for every configured agent
  const int nst = P.stages;
  const int tiles = (P.cells + kTile - 1) / kTile;

  // One agent and no debug copy: the max is the staged chunk itself, so the
  // MMA reads the stage directly and its commit releases the stage.
  const bool direct = P.K == 1 && P.fused == nullptr;
  if (warp == 0 && lane == 0) {
    for (int s = 0; s < nst; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], direct ? 1 : kWorkers);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&fready[b], kWorkers);
      mbar_init(&fempty[b], 1);
      mbar_init(&accfull[b], 1);
      mbar_init(&accempty[b], 4);
    }
    mbar_init(wbar, 1);
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 32);                 // two 16-column accumulators
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();
  // the head weights are constant: their load overlaps the previous kernel
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&P.wmap);
    mbar_arrive_expect_tx(wbar, (uint32_t)(kFuseHeadOut * C * 2));
    for (int j = 0; j < nch; ++j)
      tma_load_2d(wsm + j * kFuseHeadOut * bkc * 2, &P.wmap, wbar, j * bkc, 0);
  }
  pdl_wait();                                  // the slots are the branches' output
  span_begin(P.span);
  if (threadIdx.x == 0) {
    int n = 0;
    for (int k = 0; k < P.K; ++k)
      if (P.present[k]) s_list[n++] = k;
    s_kp = n;
  }
  __syncthreads();
  const int Kp = s_kp;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer: agent chunks -> stages ----------------
      if (Kp == P.K)
        tma_prefetch_desc(&P.feat_all);
      else
        for (int k = 0; k < Kp; ++k) tma_prefetch_desc(&P.feat[s_list[k]]);
      uint32_t it = 0;
      bool alive = true;
      for (int t = blockIdx.x; t < tiles && alive; t += gridDim.x) {
        for (int j = 0; j < nch; ++j, ++it) {
          const int s = it % nst;
          if (!mbar_wait(&empty[s], ((it / nst) & 1) ^ 1)) {
            atomicOr(P.err, ERR_WAIT_FUSE);
            alive = false;
            break;
          }
          mbar_arrive_expect_tx(&full[s], (uint32_t)(Kp * slot_bytes));
          if (Kp == P.K) {
            // every slot present: one box of all K agents' chunks (a thread's
            // boxes complete one after another, whatever their size)
            tma_load_3d(smem + s * stage_bytes, &P.feat_all, &full[s], j * bkc, t * kTile, 0);
          } else {
            for (int i = 0; i < Kp; ++i)
              tma_load_2d(smem + s * stage_bytes + i * slot_bytes, &P.feat[s_list[i]], &full[s],
                          j * bkc, t * kTile);
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer: fused chunk x head weights ----------------
      bool alive = mbar_wait(wbar, 0);
      if (!alive) atomicOr(P.err, ERR_WAIT_FUSE);
      const uint32_t idesc = idesc_f16(kTile, kFuseHeadOut, std::is_same<T, __nv_bfloat16>::value);
      const uint32_t swz = bkc == 64 ? 2u : 4u;   // 128B : 64B swizzle
      const uint32_t sbo = 8u * bkc * 2u;          // bytes between 8-row atoms
      const uint32_t f0 = smem_u32(fbuf), w0 = smem_u32(wsm);
      uint32_t it = 0, tc = 0;
      for (int t = blockIdx.x; t < tiles && alive; t += gridDim.x, ++tc) {
        const int acc = tc & 1;
        if (!mbar_wait(&accempty[acc], ((tc >> 1) & 1) ^ 1)) {
          atomicOr(P.err, ERR_WAIT_FUSE);
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem + acc * kFuseHeadOut;
        for (int j = 0; j < nch; ++j, ++it) {
          const int b = it & 1, s = it % nst;
          if (direct ? !mbar_wait(&full[s], (it / nst) & 1) : !mbar_wait(&fready[b], (it >> 1) & 1)) {
            atomicOr(P.err, ERR_WAIT_FUSE);
            alive = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = direct ? smem_desc(smem_u32(smem) + s * stage_bytes, sbo, swz)
                                     : smem_desc(f0 + b * fbytes, sbo, swz);
          const uint64_t bd = smem_desc(w0 + j * kFuseHeadOut * bkc * 2, sbo, swz);
          for (int kk = 0; kk < bkc / 16; ++kk)      // K advance: 32 bytes = +2
            umma_f16(d_tmem, ad + 2 * kk, bd + 2 * kk, idesc, (j > 0 || kk > 0) ? 1u : 0u);
          umma_commit(direct ? &empty[s] : &fempty[b]);
        }
        umma_commit(&accfull[acc]);
      }
    }
  } else {
    // ---------------- max workers + epilogue ----------------
    const int wt = threadIdx.x - 64;           // 0..kWorkers-1
    const bool epi = warp < 6;                 // warps 2..5: one TMEM lane quarter each
    const int qd = warp & 3;                   // tensor-memory lane quarter of this warp
    const int row = qd * 32 + lane;            // cell within the tile
    float hb[kFuseHeadOut];
#pragma unroll
    for (int o = 0; o < kFuseHeadOut; ++o) hb[o] = P.head_b[o];
    const int vpr = bkc * 2 / 16;              // 16-byte vectors per staged row
    const int nvec = kTile * vpr;              // vectors per agent chunk
    T* fused = static_cast<T*>(P.fused);
    uint32_t it = 0, tc = 0;
    bool alive = true;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++tc) {
      for (int j = 0; j < nch && !direct; ++j, ++it) {
        const int s = it % nst, b = it & 1;
        if (alive && !mbar_wait(&full[s], (it / nst) & 1)) {
          atomicOr(P.err, ERR_WAIT_FUSE);
          alive = false;
        }
        // the fused buffer must have been read by the MMA of two chunks ago
        if (alive && !mbar_wait(&fempty[b], ((it >> 1) & 1) ^ 1)) {
          atomicOr(P.err, ERR_WAIT_FUSE);
          alive = false;
        }
        const uint4* st = reinterpret_cast<const uint4*>(smem + s * stage_bytes);
        uint4* fb = reinterpret_cast<uint4*>(fbuf + b * fbytes);
        max_chunk_any<T>(st, fb, nvec, wt, Kp);
        if (fused) {
          // debug copy of the fused features, unswizzled to [cell][C]
          for (int v = wt; v < nvec; v += kWorkers) {
            const int r = v / vpr, ch = v - r * vpr;
            const int x = (bkc == 64) ? (r & 7) : ((r >> 1) & 3);
            const int cell = t * kTile + r;
            if (cell < P.cells)
              *reinterpret_cast<uint4*>(fused + (size_t)cell * C + j * bkc + ((ch ^ x) << 3)) = fb[v];
          }
        }
        // the stage is read: hand it back to the producer at once; the fused
        // chunk (generic-proxy writes) goes to the MMA
        mbar_arrive(&empty[s]);
        fence_async_smem();
        mbar_arrive(&fready[b]);
      }
      // epilogue of tile t (warps 2..5)
      if (!epi) continue;
      const int acc = tc & 1;
      if (alive && !mbar_wait(&accfull[acc], (tc >> 1) & 1)) {
        if (lane == 0) atomicOr(P.err, ERR_WAIT_FUSE);
        alive = false;
      }
      tc_fence_after();
      float v[16];
      tmem_ld16(tmem + acc * kFuseHeadOut + (static_cast<uint32_t>(qd * 32) << 16), v);
      tc_fence_before();
      if (lane == 0) mbar_arrive(&accempty[acc]);
      const int cell = t * kTile + row;
      const bool cv = cell < P.cells;
#pragma unroll
      for (int o = 0; o < kFuseHeadOut; ++o) v[o] += hb[o];
      if (cv) {
        float4* ho = reinterpret_cast<float4*>(P.head_out + (size_t)cell * kFuseHeadOut);
#pragma unroll
        for (int q = 0; q < 4; ++q) ho[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
      }
#pragma unroll
      for (int o = 0; o < kFuseHeadOut; ++o) {
        if (o < P.anchors) {
          const bool keep = cv && v[o] >= P.cls_thresh;
          const uint32_t key = keep ? ord_desc(v[o]) : 0xFFFFFFFFu;
          if (cv) P.keys[(size_t)cell * P.anchors + o] = key;
          hist_add(P.hist0, keep, key, lane);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  span_end(P.span);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 32);
  }
}

}  // namespace

int fuse_tc_chunk(int C, int K) {
  if (C % 32 != 0 || C > kMaxC || K < 1 || K > RTCC_MAX_AGENTS) return 0;
  // 64-channel chunks while at least 3 stages of K agent chunks fit, else 32
  if (C % 64 == 0 && 3 * K * kTile * 64 * 2 <= stage_area(64)) return 64;
  return 2 * K * kTile * 32 * 2 <= stage_area(32) ? 32 : 0;
}

int fuse_tc_stages(int C, int K) {
  const int bkc = fuse_tc_chunk(C, K);
  if (bkc == 0) return 0;
  const int n = stage_area(bkc) / (K * kTile * bkc * 2);
  return n < kMaxStages ? n : kMaxStages;
}

cudaError_t launch_fuse_max_head(const FuseTcParams& p, bool bf16, cudaStream_t st) {
  if (p.bkc != fuse_tc_chunk(p.C, p.K) || p.stages != fuse_tc_stages(p.C, p.K) || p.stages < 2 ||
      p.anchors < 1 || p.anchors > kFuseHeadOut || p.cells < 1)
    return cudaErrorInvalidValue;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int tiles = (p.cells + kTile - 1) / kTile;
  const int blocks = tiles < sms ? tiles : sms;
  auto kern = bf16 ? k_fuse_max_head<__nv_bfloat16> : k_fuse_max_head<__half>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(blocks), dim3(kThreads), kSmem, st, p);
}

}  // namespace rtcc

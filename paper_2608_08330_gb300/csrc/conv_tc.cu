// Implicit-GEMM convolutions of the encoder backbone and neck on the
// 5th-generation tensor cores (tcgen05, accumulator in tensor memory), fed by
// TMA tiled loads.  Used for every 3x3 conv (stride 1 and 2, zero padding 1)
// and every transposed conv with kernel = stride (the PointPillars neck), all
// followed by bias + ReLU (Sec. III-B: the per-agent encoder E_k).
//
// GEMM view, one CTA per (128-pixel tile, BN output channels):
//   D[m][n] = sum_k A[m][k] * B[n][k],  m = pixel, n = output channel,
//   k = (tap, input channel), tap-major.
// A (activations, NHWC) is never materialised: for each tap the producer warp
// issues a TMA box load of the input shifted by the tap's offset; TMA fills
// out-of-image elements with zeros, which is exactly the zero padding.  Stride
// 2 uses a 5-D view of the same tensor, (2C, W/2, 2, H/2, 1), in which the
// stride-2 gather becomes a unit-stride box at a tap-dependent (channel half,
// column, row parity, row) offset.  B (weights) is pre-packed K-major.
//
// Roles (192 threads): warp 0 = TMA producer, warp 1 = tensor-memory owner and
// MMA issuer, warps 2..5 = epilogue (tensor memory -> registers -> bias, ReLU,
// 16-bit, staged in shared memory and written by TMA tensor stores).  Every mbarrier wait is bounded; a wait that runs out sets a
// bit in the error word and the CTA winds down without hanging.
#include <mutex>
#include <type_traits>

#include "common.cuh"
#include "kernels.h"

namespace rtcc {

namespace {

constexpr int TW = 32;            // tile width in pixels
constexpr int TH = 4;             // tile height
constexpr int BM = TW * TH;       // 128 = MMA M
constexpr int kThreads = 192;
constexpr int kSmemBudget = 160 * 1024;

struct ConvArgs {
  const float* bias;
  void* out;
  int gw, gh;          // extent of the M grid
  int out_w;           // output map width (pixels)
  int ldc, choff;
  int cin, cout, s;
  int tiles_x;
  int splits;          // K split across gridDim.z CTAs (1 = none)
  float* ws;           // [splits][tiles][BN/4][BM][4] fp32 partials (splits > 1)
  int* counters;       // [tiles] arrivals per tile, 0 between launches
  int* err;
};

template <int BN, int BK>
struct Geo {
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int STAGES = (kSmemBudget / STAGE_BYTES) > 8 ? 8 : (kSmemBudget / STAGE_BYTES);
  static constexpr int SMEM = STAGES * STAGE_BYTES + 1024 + 256;
  static constexpr int TMEM_COLS = BN < 32 ? 32 : BN;
  static constexpr uint32_t SWZ = (BK == 64) ? 2u : 4u;     // 128B : 64B swizzle
  static constexpr uint32_t SBO = 8 * BK * 2;               // bytes between 8-row atoms
};

// bias + ReLU of 16 fp32 columns [c0, c0+16) of tile row `row`, packed to
// 16 bits and written to the staging tile.  Channels are staged in groups of
// SG (64 or 32): group g is a [BM][SG] block with SG*2-byte rows in the
// 128-byte (SG = 64) or 64-byte (SG = 32) swizzle of the store tensor map, so
// a warp's 16-byte writes spread over all banks.
template <typename T, int SG>
__device__ __forceinline__ void stage16(uint8_t* stage, int row, int c0, const float* v,
                                        const float* bias) {
  uint32_t pk[8];
#pragma unroll
  for (int j = 0; j < 8; ++j)
    pk[j] = Store<T>::pack2(relu_f(v[2 * j] + bias[2 * j]), relu_f(v[2 * j + 1] + bias[2 * j + 1]));
  constexpr int RB = SG * 2;                           // bytes per staged row
  uint8_t* base = stage + (c0 / SG) * (BM * RB) + row * RB;
  const int j0 = (c0 % SG) / 8;                        // 16-byte chunk within the row
  const int x = (SG == 64) ? (row & 7) : ((row >> 1) & 3);
  *reinterpret_cast<uint4*>(base + ((j0 ^ x) << 4)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
  *reinterpret_cast<uint4*>(base + (((j0 + 1) ^ x) << 4)) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
}

// barrier among the 4 epilogue warps only (named barrier 1, 128 threads)
__device__ __forceinline__ void epilogue_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

template <int KIND, int BN, int BK, typename T>
__global__ void __launch_bounds__(kThreads, 1)
k_conv_tc(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
          const __grid_constant__ CUtensorMap mapC, const ConvArgs a) {
  using G = Geo<BN, BK>;
  constexpr int STAGES = G::STAGES;
  constexpr int SG = BN < 64 ? BN : 64;          // channels per staged output group
  static_assert(STAGES * G::A_BYTES >= BM * BN * 2, "staging tile must fit the A buffers");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * G::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + STAGES * G::B_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* accum = empty + STAGES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int tile = blockIdx.x;
  const int x0 = (tile % a.tiles_x) * TW;
  const int y0 = (tile / a.tiles_x) * TH;
  const int n0 = blockIdx.y * BN;
  const int ncb = a.cin / BK;
  const int total_kb = (KIND == DECONV ? 1 : 9) * ncb;
  // this CTA's slice of the K loop (all of it without split-K)
  const int z = blockIdx.z;
  const int kb_begin = (z * total_kb) / a.splits;
  const int num_kb = ((z + 1) * total_kb) / a.splits - kb_begin;

  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&mapA);
    tma_prefetch_desc(&mapB);
    tma_prefetch_desc(&mapC);
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accum, 1);
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, G::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // the prologue above overlapped the previous layer; from here on this CTA
  // reads its input and writes its output
  pdl_trigger();
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      for (int it = 0; it < num_kb; ++it) {
        const int s = it % STAGES;
        const uint32_t ph = (it / STAGES) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1)) {
          atomicOr(a.err, ERR_WAIT_PRODUCER);
          break;
        }
        const int kb = kb_begin + it;
        const int tap = kb / ncb;
        const int cb = kb - tap * ncb;
        mbar_arrive_expect_tx(&full[s], G::STAGE_BYTES);
        void* dA = sA + s * G::A_BYTES;
        void* dB = sB + s * G::B_BYTES;
        if (KIND == CONV3_S1) {
          const int dy = tap / 3, dx = tap - 3 * (tap / 3);
          tma_load_4d(dA, &mapA, &full[s], cb * BK, x0 + dx - 1, y0 + dy - 1, 0);
        } else if (KIND == CONV3_S2) {
          // input x = 2*ox + dx - 1 = 2*j + p; input y = 2*oy + dy - 1 = 2*i + q
          const int dy = tap / 3, dx = tap - 3 * (tap / 3);
          const int j = x0 + (dx == 0 ? -1 : 0);
          const int p = (dx == 1) ? 0 : 1;
          const int i = y0 + (dy == 0 ? -1 : 0);
          const int q = (dy == 1) ? 0 : 1;
          tma_load_5d(dA, &mapA, &full[s], p * a.cin + cb * BK, j, q, i, 0);
        } else {
          tma_load_4d(dA, &mapA, &full[s], cb * BK, x0, y0, 0);
        }
        tma_load_2d(dB, &mapB, &full[s], tap * a.cin + cb * BK, n0);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      constexpr uint32_t IDESC = idesc_f16(BM, BN, std::is_same<T, __nv_bfloat16>::value);
      for (int kb = 0; kb < num_kb; ++kb) {
        const int s = kb % STAGES;
        const uint32_t ph = (kb / STAGES) & 1;
        if (!mbar_wait(&full[s], ph)) {
          atomicOr(a.err, ERR_WAIT_MMA);
          break;
        }
        tc_fence_after();
        const uint32_t aa = smem_u32(sA + s * G::A_BYTES);
        const uint32_t bb = smem_u32(sB + s * G::B_BYTES);
#pragma unroll
        for (int k = 0; k < BK / 16; ++k) {
          umma_f16(tmem, smem_desc(aa + k * 32, G::SBO, G::SWZ),
                   smem_desc(bb + k * 32, G::SBO, G::SWZ), IDESC, (kb | k) != 0);
        }
        umma_commit(&empty[s]);
      }
      umma_commit(accum);
    }
  } else {
    // ---------------- epilogue ----------------
    // accumulator -> bias + ReLU -> 16-bit, staged in shared memory in the
    // store map's swizzled layout, then written by TMA tensor stores (full
    // lines; rows outside the image are clipped by the store)
    const int qd = warp & 3;                 // tensor-memory lane quarter of this warp
    const int row = qd * 32 + lane;          // pixel within the tile
    const bool ok = mbar_wait(accum, 0);
    if (!ok && lane == 0) atomicOr(a.err, ERR_WAIT_EPILOGUE);
    tc_fence_after();
    const float* bias = a.bias + (KIND == DECONV ? 0 : n0);
    const uint32_t taddr = tmem + (static_cast<uint32_t>(qd * 32) << 16);
    uint8_t* stage = sA;                     // pipeline buffers are idle once the MMAs are done
    bool store = true;
    if (a.splits == 1) {
#pragma unroll
      for (int c0 = 0; c0 < BN; c0 += 16) {
        float v[16];
        tmem_ld16(taddr + c0, v);
        stage16<T, SG>(stage, row, c0, v, bias + c0);
      }
    } else {
      // split-K: publish this slice's fp32 partial, then the last CTA of the
      // tile sums the slices in slice order (deterministic) and stores
      // workspace layout per (slice, tile): [BN/4 column quads][BM rows][4],
      // so a warp's float4 stores cover 512 contiguous bytes
      const int tiles = gridDim.x * gridDim.y;
      const int tile_id = blockIdx.y * gridDim.x + blockIdx.x;
      float4* mine = reinterpret_cast<float4*>(a.ws + (size_t)(z * tiles + tile_id) * BM * BN) + row;
#pragma unroll
      for (int c0 = 0; c0 < BN; c0 += 16) {
        float v[16];
        tmem_ld16(taddr + c0, v);
#pragma unroll
        for (int q = 0; q < 4; ++q)
          mine[(c0 / 4 + q) * BM] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
      }
      __threadfence();
      epilogue_sync();
      __shared__ int s_last;
      if (row == 0) {
        const int old = atomicAdd(&a.counters[tile_id], 1);
        s_last = (old == a.splits - 1);
      }
      epilogue_sync();
      store = s_last != 0;
      if (store) {
        __threadfence();
#pragma unroll
        for (int c0 = 0; c0 < BN; c0 += 16) {
          float acc[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) acc[j] = 0.f;
          for (int zz = 0; zz < a.splits; ++zz) {
            float v[16];
            if (zz == z) {
              tmem_ld16(taddr + c0, v);
            } else {
              const float4* src =
                  reinterpret_cast<const float4*>(a.ws + (size_t)(zz * tiles + tile_id) * BM * BN) +
                  row;
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const float4 f = __ldcg(src + (c0 / 4 + q) * BM);
                v[4 * q] = f.x; v[4 * q + 1] = f.y; v[4 * q + 2] = f.z; v[4 * q + 3] = f.w;
              }
            }
#pragma unroll
            for (int j = 0; j < 16; ++j) acc[j] += v[j];
          }
          stage16<T, SG>(stage, row, c0, acc, bias + c0);
        }
        if (row == 0) a.counters[tile_id] = 0;       // ready for the next launch
      }
    }
    if (store) {                                     // uniform over the epilogue warps
      fence_async_smem();
      epilogue_sync();
      if (row == 0 && ok) {
        constexpr int GB = BM * SG * 2;              // bytes of one staged channel group
        if (KIND == DECONV) {
          const int sub = n0 / a.cout;
          const int sy = sub / a.s, sx = sub - sy * a.s;
#pragma unroll
          for (int g = 0; g < BN / SG; ++g)
            tma_store_5d(&mapC, stage + g * GB, a.choff + g * SG, sx, x0, sy, y0);
        } else {
#pragma unroll
          for (int g = 0; g < BN / SG; ++g) tma_store_3d(&mapC, stage + g * GB, n0 + g * SG, x0, y0);
        }
        bulk_commit();
        bulk_wait_all();
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    // every MMA this CTA issued has retired before its accumulator is freed
    mbar_wait(accum, 0);
    tc_fence_after();
    tmem_dealloc(tmem, G::TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------

using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                              const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                              const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                              CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn encode_fn() {
  static EncodeFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFn>(p);
  });
  return fn;
}

template <int KIND, int BN, int BK, typename T>
cudaError_t launch_t(const ConvLayer& L, int* err, cudaStream_t st) {
  using G = Geo<BN, BK>;
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [] {
    attr_err = cudaFuncSetAttribute(k_conv_tc<KIND, BN, BK, T>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, G::SMEM);
  });
  if (attr_err != cudaSuccess) return attr_err;
  ConvArgs a;
  a.bias = L.bias;
  a.out = L.out;
  a.gw = L.gw;
  a.gh = L.gh;
  a.out_w = L.out_w;
  a.ldc = L.ldc;
  a.choff = L.choff;
  a.cin = L.cin;
  a.cout = L.cout;
  a.s = L.s;
  a.tiles_x = (L.gw + TW - 1) / TW;
  a.splits = L.splits < 1 ? 1 : L.splits;
  a.ws = L.ws;
  a.counters = L.counters;
  a.err = err;
  const int tiles_y = (L.gh + TH - 1) / TH;
  dim3 grid(a.tiles_x * tiles_y, L.n_tiles_n, a.splits);
  return launch_pdl(k_conv_tc<KIND, BN, BK, T>, grid, dim3(kThreads), G::SMEM, st, L.mapA, L.mapB,
                    L.mapC, a);
}

template <int KIND, typename T>
cudaError_t launch_kind(const ConvLayer& L, int* err, cudaStream_t st) {
  if (L.bk == 64) {
    if (L.bn == 128) return launch_t<KIND, 128, 64, T>(L, err, st);
    if (L.bn == 64) return launch_t<KIND, 64, 64, T>(L, err, st);
    if (L.bn == 32) return launch_t<KIND, 32, 64, T>(L, err, st);
  } else if (L.bk == 32) {
    if (L.bn == 128) return launch_t<KIND, 128, 32, T>(L, err, st);
    if (L.bn == 64) return launch_t<KIND, 64, 32, T>(L, err, st);
    if (L.bn == 32) return launch_t<KIND, 32, 32, T>(L, err, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

int conv_tile_w() { return TW; }
int conv_tile_h() { return TH; }
int conv_tile_m() { return BM; }

cudaError_t conv_make_maps(ConvLayer& L, bool bf16) {
  EncodeFn enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  const CUtensorMapDataType dt =
      bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
  const CUtensorMapSwizzle sw =
      (L.bk == 64) ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
  const cuuint64_t C = (cuuint64_t)L.cin, W = (cuuint64_t)L.in_w, H = (cuuint64_t)L.in_h;
  CUresult r;
  if (L.kind == CONV3_S2) {
    if ((L.in_w & 1) || (L.in_h & 1)) return cudaErrorInvalidValue;
    cuuint64_t dims[5] = {2 * C, W / 2, 2, H / 2, 1};
    cuuint64_t strides[4] = {2 * C * 2, W * C * 2, 2 * W * C * 2, H * W * C * 2};
    cuuint32_t box[5] = {(cuuint32_t)L.bk, (cuuint32_t)TW, 1, (cuuint32_t)TH, 1};
    cuuint32_t es[5] = {1, 1, 1, 1, 1};
    r = enc(&L.mapA, dt, 5, const_cast<void*>(L.in), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  } else {
    cuuint64_t dims[4] = {C, W, H, 1};
    cuuint64_t strides[3] = {C * 2, W * C * 2, H * W * C * 2};
    cuuint32_t box[4] = {(cuuint32_t)L.bk, (cuuint32_t)TW, (cuuint32_t)TH, 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    r = enc(&L.mapA, dt, 4, const_cast<void*>(L.in), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  }
  if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  const cuuint64_t K = (cuuint64_t)((L.kind == DECONV ? 1 : 9) * L.cin);
  const cuuint64_t rows = (cuuint64_t)((L.kind == DECONV ? L.s * L.s : 1) * L.cout);
  cuuint64_t bdims[2] = {K, rows};
  cuuint64_t bstr[1] = {K * 2};
  cuuint32_t bbox[2] = {(cuuint32_t)L.bk, (cuuint32_t)L.bn};
  cuuint32_t bes[2] = {1, 1};
  r = enc(&L.mapB, dt, 2, const_cast<void*>(L.wpacked), bdims, bstr, bbox, bes,
          CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  // output store map: conv [out_h][out_w][ldc]; deconv viewed as
  // [in_h][s][in_w][s][ldc] so one sub-pixel position of a tile is one box
  const int sg = L.bn < 64 ? L.bn : 64;
  const CUtensorMapSwizzle osw = (sg == 64) ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
  const cuuint64_t LD = (cuuint64_t)L.ldc;
  if (L.kind == DECONV) {
    const cuuint64_t S = (cuuint64_t)L.s, IW = (cuuint64_t)L.in_w, IH = (cuuint64_t)L.in_h;
    const cuuint64_t OW = (cuuint64_t)L.out_w;
    cuuint64_t dims[5] = {LD, S, IW, S, IH};
    cuuint64_t strides[4] = {LD * 2, S * LD * 2, OW * LD * 2, S * OW * LD * 2};
    cuuint32_t box[5] = {(cuuint32_t)sg, 1, (cuuint32_t)TW, 1, (cuuint32_t)TH};
    cuuint32_t es[5] = {1, 1, 1, 1, 1};
    r = enc(&L.mapC, dt, 5, L.out, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, osw,
            CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  } else {
    cuuint64_t dims[3] = {LD, (cuuint64_t)L.out_w, (cuuint64_t)L.out_h};
    cuuint64_t strides[2] = {LD * 2, (cuuint64_t)L.out_w * LD * 2};
    cuuint32_t box[3] = {(cuuint32_t)sg, (cuuint32_t)TW, (cuuint32_t)TH};
    cuuint32_t es[3] = {1, 1, 1};
    r = enc(&L.mapC, dt, 3, L.out, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, osw,
            CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  }
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t launch_conv(const ConvLayer& L, bool bf16, int* err, cudaStream_t st) {
  if (L.cin % L.bk || (L.kind != DECONV && L.cout % L.bn) ||
      (L.kind == DECONV && L.bn != L.cout))
    return cudaErrorInvalidValue;
  const int total_kb = (L.kind == DECONV ? 1 : 9) * (L.cin / L.bk);
  if (L.splits > 1 && (!L.ws || !L.counters || L.splits > total_kb)) return cudaErrorInvalidValue;
  if (bf16) {
    switch (L.kind) {
      case CONV3_S1: return launch_kind<CONV3_S1, __nv_bfloat16>(L, err, st);
      case CONV3_S2: return launch_kind<CONV3_S2, __nv_bfloat16>(L, err, st);
      case DECONV: return launch_kind<DECONV, __nv_bfloat16>(L, err, st);
    }
  } else {
    switch (L.kind) {
      case CONV3_S1: return launch_kind<CONV3_S1, __half>(L, err, st);
      case CONV3_S2: return launch_kind<CONV3_S2, __half>(L, err, st);
      case DECONV: return launch_kind<DECONV, __half>(L, err, st);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace rtcc

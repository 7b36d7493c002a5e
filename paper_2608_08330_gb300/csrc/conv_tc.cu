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
// 16-bit store).  Every mbarrier wait is bounded; a wait that runs out sets a
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

template <int KIND, int BN, int BK, typename T>
__global__ void __launch_bounds__(kThreads, 1)
k_conv_tc(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
          const ConvArgs a) {
  using G = Geo<BN, BK>;
  constexpr int STAGES = G::STAGES;
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
  const int num_kb = (KIND == DECONV ? 1 : 9) * ncb;

  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&mapA);
    tma_prefetch_desc(&mapB);
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

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      for (int kb = 0; kb < num_kb; ++kb) {
        const int s = kb % STAGES;
        const uint32_t ph = (kb / STAGES) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1)) {
          atomicOr(a.err, ERR_WAIT_PRODUCER);
          break;
        }
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
    const int qd = warp & 3;                 // tensor-memory lane quarter of this warp
    const int row = qd * 32 + lane;          // pixel within the tile
    const bool ok = mbar_wait(accum, 0);
    if (!ok && lane == 0) atomicOr(a.err, ERR_WAIT_EPILOGUE);
    tc_fence_after();
    const int gx = x0 + (row % TW);
    const int gy = y0 + (row / TW);
    const bool valid = ok && gx < a.gw && gy < a.gh;
    size_t off;
    const float* bias;
    if (KIND == DECONV) {
      const int sub = n0 / a.cout;
      const int oy = gy * a.s + sub / a.s;
      const int ox = gx * a.s + sub % a.s;
      off = ((size_t)oy * a.out_w + ox) * a.ldc + a.choff;
      bias = a.bias;
    } else {
      off = ((size_t)gy * a.out_w + gx) * a.ldc + a.choff + n0;
      bias = a.bias + n0;
    }
    T* out = static_cast<T*>(a.out) + off;
    const uint32_t taddr = tmem + (static_cast<uint32_t>(qd * 32) << 16);
#pragma unroll
    for (int c0 = 0; c0 < BN; c0 += 16) {
      float v[16];
      tmem_ld16(taddr + c0, v);
      if (valid) {
        uint32_t pk[8];
#pragma unroll
        for (int j = 0; j < 8; ++j)
          pk[j] = Store<T>::pack2(relu_f(v[2 * j] + bias[c0 + 2 * j]),
                                  relu_f(v[2 * j + 1] + bias[c0 + 2 * j + 1]));
        uint4* dst = reinterpret_cast<uint4*>(out + c0);
        dst[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        dst[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
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
  a.err = err;
  const int tiles_y = (L.gh + TH - 1) / TH;
  dim3 grid(a.tiles_x * tiles_y, L.n_tiles_n);
  k_conv_tc<KIND, BN, BK, T><<<grid, kThreads, G::SMEM, st>>>(L.mapA, L.mapB, a);
  return cudaGetLastError();
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
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t launch_conv(const ConvLayer& L, bool bf16, int* err, cudaStream_t st) {
  if (L.cin % L.bk || (L.kind != DECONV && L.cout % L.bn) ||
      (L.kind == DECONV && L.bn != L.cout))
    return cudaErrorInvalidValue;
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

// Post-join fusion of the agents' BEV feature slots and the 1x1 detection head
// (the shared subgraph after the all-agent join, Sec. III-B / Sec. IV-D).
//
// One warp per BEV cell.  Each lane owns a fixed set of C/32 channels and
// reads them from every present agent's slot with 8/16-byte loads; the warp
// reads each slot's cell vector exactly once (the kernel is bound by HBM/L2
// bandwidth).  Fusion, in agent-index order over present agents:
//   max:        F = max_k X_k (elementwise)
//   attention:  s_k = <X_0, X_k> / sqrt(C) (ego agent 0 is the query),
//               w = softmax_k(s), F = sum_k w_k X_k
// The fused vector stays in registers and feeds the head
//   out[o] = b[o] + sum_c W[o][c] F[c],  o < 8A = 16,
// whose 16 partial sums are reduced across the warp with a reduce-scatter
// butterfly (16 shuffles).  Every reduction has a fixed order, so the output is
// bit-reproducible and independent of when or in what order the branches ran.
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace rtcc {

namespace {

constexpr unsigned kFull = 0xFFFFFFFFu;
constexpr int kHeadOut = 16;

template <int C>
struct Lanes {
  static constexpr int CPL = C / 32;          // channels per lane
  // channel of the lane's j-th value
  static __host__ __device__ int chan(int lane, int j) {
    if (C == 384) return j < 8 ? 8 * lane + j : 256 + 4 * lane + (j - 8);
    return lane * CPL + j;
  }
};

template <typename T, int N>
__device__ __forceinline__ void load_vals(const T* p, float* x) {
  // N contiguous 16-bit values at p (N in {1, 2, 4, 8})
  if (N == 8) {
    const uint4 u = *reinterpret_cast<const uint4*>(p);
    float2 f;
    f = Store<T>::unpack2(u.x); x[0] = f.x; x[1] = f.y;
    f = Store<T>::unpack2(u.y); x[2] = f.x; x[3] = f.y;
    f = Store<T>::unpack2(u.z); x[4] = f.x; x[5] = f.y;
    f = Store<T>::unpack2(u.w); x[6] = f.x; x[7] = f.y;
  } else if (N == 4) {
    const uint2 u = *reinterpret_cast<const uint2*>(p);
    float2 f;
    f = Store<T>::unpack2(u.x); x[0] = f.x; x[1] = f.y;
    f = Store<T>::unpack2(u.y); x[2] = f.x; x[3] = f.y;
  } else if (N == 2) {
    const float2 f = Store<T>::unpack2(*reinterpret_cast<const uint32_t*>(p));
    x[0] = f.x; x[1] = f.y;
  } else {
    x[0] = Store<T>::to_f(*p);
  }
}

template <typename T, int C>
__device__ __forceinline__ void load_cell(const T* row, int lane, float* x) {
  if (C == 384) {
    load_vals<T, 8>(row + 8 * lane, x);
    load_vals<T, 4>(row + 256 + 4 * lane, x + 8);
  } else {
    load_vals<T, Lanes<C>::CPL>(row + lane * Lanes<C>::CPL, x);
  }
}

template <typename T, int C>
__device__ __forceinline__ void store_cell(T* row, int lane, const float* x) {
#pragma unroll
  for (int j = 0; j < Lanes<C>::CPL; ++j) row[Lanes<C>::chan(lane, j)] = Store<T>::from_f(x[j]);
}

template <typename T, int C, bool ATTN>
__global__ void __launch_bounds__(256)
k_fuse_head(const void* const* __restrict__ feats, const int* __restrict__ present, int K,
            int cells, float inv_sqrt_c, const float* __restrict__ head_wp,
            const float* __restrict__ head_b, float* __restrict__ head_out, T* __restrict__ fused) {
  constexpr int CPL = Lanes<C>::CPL;
  extern __shared__ float sw[];               // [16][CPL][32] permuted head weights
  for (int i = threadIdx.x; i < kHeadOut * C; i += blockDim.x) sw[i] = head_wp[i];
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int warps = blockDim.x >> 5;
  unsigned pres = 0;
  for (int k = 0; k < K; ++k) pres |= (present[k] ? 1u : 0u) << k;
  const T* slot[RTCC_MAX_AGENTS];
#pragma unroll
  for (int k = 0; k < RTCC_MAX_AGENTS; ++k)
    slot[k] = (k < K) ? static_cast<const T*>(feats[k]) : nullptr;
  const float hb = head_b[lane >> 1];

  for (int cell = blockIdx.x * warps + (threadIdx.x >> 5); cell < cells;
       cell += gridDim.x * warps) {
    float x[RTCC_MAX_AGENTS][CPL];
#pragma unroll
    for (int k = 0; k < RTCC_MAX_AGENTS; ++k)
      if (k < K && ((pres >> k) & 1u)) load_cell<T, C>(slot[k] + (size_t)cell * C, lane, x[k]);
    float F[CPL];
    if (!ATTN) {
      bool first = true;
#pragma unroll
      for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
        if (k < K && ((pres >> k) & 1u)) {
#pragma unroll
          for (int j = 0; j < CPL; ++j) F[j] = first ? x[k][j] : (x[k][j] > F[j] ? x[k][j] : F[j]);
          first = false;
        }
      }
    } else {
      float s[RTCC_MAX_AGENTS];
      float m = -INFINITY;
#pragma unroll
      for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
        s[k] = -INFINITY;
        if (k < K && ((pres >> k) & 1u)) {
          float d = 0.f;
#pragma unroll
          for (int j = 0; j < CPL; ++j) d = fmaf(x[0][j], x[k][j], d);
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) d += __shfl_xor_sync(kFull, d, o);
          s[k] = d * inv_sqrt_c;
          m = fmaxf(m, s[k]);
        }
      }
      float den = 0.f;
#pragma unroll
      for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
        if (k < K && ((pres >> k) & 1u)) {
          s[k] = expf(s[k] - m);
          den += s[k];
        }
      }
#pragma unroll
      for (int j = 0; j < CPL; ++j) F[j] = 0.f;
#pragma unroll
      for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
        if (k < K && ((pres >> k) & 1u)) {
          const float w = s[k] / den;
#pragma unroll
          for (int j = 0; j < CPL; ++j) F[j] = fmaf(w, x[k][j], F[j]);
        }
      }
    }
    if (fused) store_cell<T, C>(fused + (size_t)cell * C, lane, F);
    // head: 16 partial dot products over the lane's channels
    float acc[kHeadOut];
#pragma unroll
    for (int o = 0; o < kHeadOut; ++o) {
      float a = 0.f;
#pragma unroll
      for (int j = 0; j < CPL; ++j) a = fmaf(F[j], sw[(o * CPL + j) * 32 + lane], a);
      acc[o] = a;
    }
    // reduce-scatter: after offsets 16, 8, 4, 2 lane l holds output l >> 1 over
    // the 16 lanes sharing its bit 0; the last exchange adds the other half.
    int n = kHeadOut;
#pragma unroll
    for (int off = 16; off >= 2; off >>= 1) {
      const int h = n >> 1;
      const bool upper = (lane & off) != 0;
#pragma unroll
      for (int i = 0; i < kHeadOut / 2; ++i) {
        if (i < h) {
          const float send = upper ? acc[i] : acc[i + h];
          const float keep = upper ? acc[i + h] : acc[i];
          acc[i] = keep + __shfl_xor_sync(kFull, send, off);
        }
      }
      n = h;
    }
    const float tot = acc[0] + __shfl_xor_sync(kFull, acc[0], 1);
    if ((lane & 1) == 0) head_out[(size_t)cell * kHeadOut + (lane >> 1)] = tot + hb;
  }
}

template <typename T, int C>
cudaError_t launch_c(const FuseArgs& a, cudaStream_t st) {
  const size_t smem = sizeof(float) * kHeadOut * C;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int blocks = (a.cells + 7) / 8;
  const int cap = sms * 8;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  const float isc = 1.0f / sqrtf((float)C);
  T* fused = static_cast<T*>(a.fused);
  if (a.attention) {
    if (smem > 48 * 1024)
      cudaFuncSetAttribute(k_fuse_head<T, C, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem);
    k_fuse_head<T, C, true><<<blocks, 256, smem, st>>>(a.feats, a.present, a.K, a.cells, isc,
                                                       a.head_wp, a.head_b, a.head_out, fused);
  } else {
    if (smem > 48 * 1024)
      cudaFuncSetAttribute(k_fuse_head<T, C, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem);
    k_fuse_head<T, C, false><<<blocks, 256, smem, st>>>(a.feats, a.present, a.K, a.cells, isc,
                                                        a.head_wp, a.head_b, a.head_out, fused);
  }
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_t(const FuseArgs& a, cudaStream_t st) {
  switch (a.C) {
    case 32: return launch_c<T, 32>(a, st);
    case 64: return launch_c<T, 64>(a, st);
    case 128: return launch_c<T, 128>(a, st);
    case 256: return launch_c<T, 256>(a, st);
    case 384: return launch_c<T, 384>(a, st);
  }
  return cudaErrorInvalidValue;
}

template <int C>
void permute_c(const float* w, float* out) {
  constexpr int CPL = Lanes<C>::CPL;
  for (int o = 0; o < kHeadOut; ++o)
    for (int j = 0; j < CPL; ++j)
      for (int l = 0; l < 32; ++l) out[(o * CPL + j) * 32 + l] = w[o * C + Lanes<C>::chan(l, j)];
}

}  // namespace

cudaError_t launch_fuse_head(const FuseArgs& a, bool bf16, cudaStream_t st) {
  if (a.K < 1 || a.K > RTCC_MAX_AGENTS) return cudaErrorInvalidValue;
  return bf16 ? launch_t<__nv_bfloat16>(a, st) : launch_t<__half>(a, st);
}

void permute_head_weights(const float* w, int C, float* out) {
  switch (C) {
    case 32: permute_c<32>(w, out); break;
    case 64: permute_c<64>(w, out); break;
    case 128: permute_c<128>(w, out); break;
    case 256: permute_c<256>(w, out); break;
    case 384: permute_c<384>(w, out); break;
  }
}

}  // namespace rtcc

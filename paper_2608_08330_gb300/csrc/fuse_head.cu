// Post-join fusion of the agents' BEV feature slots and the 1x1 detection head
// (the shared subgraph after the all-agent join, Sec. III-B / Sec. IV-D).
//
// Each warp handles a few BEV cells per pass, persistent over cells.  Each lane
// owns a fixed set of C/32 channels and reads them from every present agent's
// slot with 16/8-byte loads, so each slot's cell vector is read exactly once;
// the kernel is bound by HBM/L2 bandwidth.  Agent vectors stay packed in
// 16-bit pairs.
// Fusion, in agent-index order over present agents:
//   max:        F = max_k X_k elementwise (exact in the 16-bit domain; the slots
//               hold ReLU outputs, so the running max starts at +0)
//   attention:  s_k = <X_0, X_k> / sqrt(C) (ego agent 0 is the query),
//               w = softmax_k(s), F = sum_k w_k X_k   (fp32)
// The fused vector feeds the head out[o] = b[o] + sum_c W[o][c] F[c], o < 16,
// whose partial sums are reduced across the warp with a reduce-scatter
// butterfly.  The kernel also writes, per anchor, the 32-bit key the decode
// selects on: the class logit mapped to an unsigned integer whose ascending
// order is descending logit order, or 0xFFFFFFFF below the threshold.  Every
// reduction has a fixed order, so the output is bit-reproducible.
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace rtcc {

namespace {

constexpr unsigned kFull = 0xFFFFFFFFu;
constexpr int kHeadOut = 16;
constexpr int kThreads = 384;

template <int C>
struct Lanes {
  static constexpr int CPL = C / 32;                   // channels per lane
  static constexpr int NW = CPL < 2 ? 1 : CPL / 2;     // 32-bit words per lane
  // channel of the lane's j-th value
  static __host__ __device__ int chan(int lane, int j) {
    if (C == 384) return j < 8 ? 8 * lane + j : 256 + 4 * lane + (j - 8);
    return lane * CPL + j;
  }
};

// The lane's channels of one cell, as packed 16-bit pairs.
template <typename T, int C>
__device__ __forceinline__ void load_raw(const T* row, int lane, uint32_t* r) {
  if (C == 384) {
    const uint4 a = *reinterpret_cast<const uint4*>(row + 8 * lane);
    const uint2 b = *reinterpret_cast<const uint2*>(row + 256 + 4 * lane);
    r[0] = a.x; r[1] = a.y; r[2] = a.z; r[3] = a.w; r[4] = b.x; r[5] = b.y;
  } else if (Lanes<C>::CPL == 8) {
    const uint4 a = *reinterpret_cast<const uint4*>(row + 8 * lane);
    r[0] = a.x; r[1] = a.y; r[2] = a.z; r[3] = a.w;
  } else if (Lanes<C>::CPL == 4) {
    const uint2 a = *reinterpret_cast<const uint2*>(row + 4 * lane);
    r[0] = a.x; r[1] = a.y;
  } else if (Lanes<C>::CPL == 2) {
    r[0] = *reinterpret_cast<const uint32_t*>(row + 2 * lane);
  } else {
    r[0] = *reinterpret_cast<const uint16_t*>(row + lane);
  }
}

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

template <typename T, int C>
__device__ __forceinline__ void unpack(const uint32_t* r, float* x) {
  if (Lanes<C>::CPL == 1) {
    x[0] = Store<T>::to_f(*reinterpret_cast<const T*>(&r[0]));
  } else {
#pragma unroll
    for (int i = 0; i < Lanes<C>::NW; ++i) {
      const float2 f = Store<T>::unpack2(r[i]);
      x[2 * i] = f.x;
      x[2 * i + 1] = f.y;
    }
  }
}

// ascending unsigned order of the result == descending float order; -0 -> +0
__device__ __forceinline__ uint32_t ord_desc(float f) {
  f = f + 0.0f;
  const uint32_t u = __float_as_uint(f);
  const uint32_t asc = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ~asc;
}

// The fused vector of one cell for this lane's channels.
template <typename T, int C, bool ATTN>
__device__ __forceinline__ void fuse_cell(const T* const* slot, unsigned pres, int K, int cell,
                                          int lane, float inv_sqrt_c, float* F) {
  constexpr int CPL = Lanes<C>::CPL;
  constexpr int NW = Lanes<C>::NW;
  if (!ATTN) {
    // every slot holds ReLU outputs (>= +0), so a running max started at +0
    // equals the max over the present agents
    uint32_t m[NW];
#pragma unroll
    for (int i = 0; i < NW; ++i) m[i] = 0u;
#pragma unroll
    for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
      if (k < K && ((pres >> k) & 1u)) {
        uint32_t r[NW];
        load_raw<T, C>(slot[k] + (size_t)cell * C, lane, r);
#pragma unroll
        for (int i = 0; i < NW; ++i) m[i] = max2<T>(m[i], r[i]);
      }
    }
    unpack<T, C>(m, F);
  } else {
    uint32_t raw[RTCC_MAX_AGENTS][NW];
#pragma unroll
    for (int k = 0; k < RTCC_MAX_AGENTS; ++k)
      if (k < K && ((pres >> k) & 1u)) load_raw<T, C>(slot[k] + (size_t)cell * C, lane, raw[k]);
    float x0[CPL];
    unpack<T, C>(raw[0], x0);
    float s[RTCC_MAX_AGENTS];
    float mx = -INFINITY;
#pragma unroll
    for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
      s[k] = -INFINITY;
      if (k < K && ((pres >> k) & 1u)) {
        float xk[CPL];
        unpack<T, C>(raw[k], xk);
        float d = 0.f;
#pragma unroll
        for (int j = 0; j < CPL; ++j) d = fmaf(x0[j], xk[j], d);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) d += __shfl_xor_sync(kFull, d, o);
        s[k] = d * inv_sqrt_c;
        mx = fmaxf(mx, s[k]);
      }
    }
    float den = 0.f;
#pragma unroll
    for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
      if (k < K && ((pres >> k) & 1u)) {
        s[k] = expf(s[k] - mx);
        den += s[k];
      }
    }
#pragma unroll
    for (int j = 0; j < CPL; ++j) F[j] = 0.f;
#pragma unroll
    for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
      if (k < K && ((pres >> k) & 1u)) {
        const float wk = s[k] / den;
        float xk[CPL];
        unpack<T, C>(raw[k], xk);
#pragma unroll
        for (int j = 0; j < CPL; ++j) F[j] = fmaf(wk, xk[j], F[j]);
      }
    }
  }
}

// Cells a warp handles per pass: each head weight read from shared memory is
// applied to all of them, and their loads are in flight together.
template <int C, bool ATTN>
struct Group {
  static constexpr int NC = (ATTN || C > 256) ? 2 : 4;
};

template <typename T, int C, bool ATTN>
__global__ void __launch_bounds__(kThreads, 1)
k_fuse_head(const void* const* __restrict__ feats, const int* present, int K,
            int cells, float inv_sqrt_c, const float* __restrict__ head_wp,
            const float* __restrict__ head_b, float* __restrict__ head_out, T* __restrict__ fused,
            uint32_t* __restrict__ keys, uint32_t* __restrict__ hist0, float cls_thresh,
            int anchors, unsigned long long* span) {
  constexpr int CPL = Lanes<C>::CPL;
  constexpr int NC = Group<C, ATTN>::NC;
  extern __shared__ float sw[];               // [16][CPL][32] permuted head weights
  __shared__ const T* slot[RTCC_MAX_AGENTS];
  pdl_trigger();
  for (int i = threadIdx.x; i < kHeadOut * C; i += blockDim.x) sw[i] = head_wp[i];  // constant
  pdl_wait();
  span_begin(span);
  if (threadIdx.x < RTCC_MAX_AGENTS)
    slot[threadIdx.x] = threadIdx.x < K ? static_cast<const T*>(feats[threadIdx.x]) : nullptr;
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int warps = blockDim.x >> 5;
  unsigned pres = 0;
  for (int k = 0; k < K; ++k) pres |= (present[k] ? 1u : 0u) << k;
  const float hb = head_b[lane >> 1];
  const int groups = (cells + NC - 1) / NC;

  for (int gi = blockIdx.x * warps + (threadIdx.x >> 5); gi < groups; gi += gridDim.x * warps) {
    const int cell0 = gi * NC;
    float F[NC][CPL];
#pragma unroll
    for (int c = 0; c < NC; ++c) {
      const int cell = min(cell0 + c, cells - 1);    // a short last group repeats a cell
      fuse_cell<T, C, ATTN>(slot, pres, K, cell, lane, inv_sqrt_c, F[c]);
    }
    if (fused) {
#pragma unroll
      for (int c = 0; c < NC; ++c) {
        if (cell0 + c < cells) {
          T* row = fused + (size_t)(cell0 + c) * C;
#pragma unroll
          for (int j = 0; j < CPL; ++j) row[Lanes<C>::chan(lane, j)] = Store<T>::from_f(F[c][j]);
        }
      }
    }
    // head: 16 partial dot products over the lane's channels, for NC cells
    float acc[NC][kHeadOut];
#pragma unroll
    for (int o = 0; o < kHeadOut; ++o) {
#pragma unroll
      for (int c = 0; c < NC; ++c) acc[c][o] = 0.f;
#pragma unroll
      for (int j = 0; j < CPL; ++j) {
        const float wv = sw[(o * CPL + j) * 32 + lane];
#pragma unroll
        for (int c = 0; c < NC; ++c) acc[c][o] = fmaf(F[c][j], wv, acc[c][o]);
      }
    }
#pragma unroll
    for (int c = 0; c < NC; ++c) {
      // reduce-scatter: after offsets 16, 8, 4, 2 lane l holds output l >> 1
      // over the 16 lanes sharing its bit 0; the last exchange adds the rest
      int n = kHeadOut;
#pragma unroll
      for (int off = 16; off >= 2; off >>= 1) {
        const int h = n >> 1;
        const bool upper = (lane & off) != 0;
#pragma unroll
        for (int i = 0; i < kHeadOut / 2; ++i) {
          if (i < h) {
            const float send = upper ? acc[c][i] : acc[c][i + h];
            const float keep = upper ? acc[c][i + h] : acc[c][i];
            acc[c][i] = keep + __shfl_xor_sync(kFull, send, off);
          }
        }
        n = h;
      }
      const float out = acc[c][0] + __shfl_xor_sync(kFull, acc[c][0], 1) + hb;
      const int cell = cell0 + c;
      const int o = lane >> 1;
      const bool mine = (lane & 1) == 0 && cell < cells;
      if (mine) head_out[(size_t)cell * kHeadOut + o] = out;
      const bool keep = mine && o < anchors && out >= cls_thresh;
      const uint32_t key = keep ? ord_desc(out) : 0xFFFFFFFFu;
      if (mine && o < anchors) keys[(size_t)cell * anchors + o] = key;
      // lanes sharing a histogram bin add their count with one atomic (valid
      // logits crowd into a few dozen bins)
      const uint32_t bin = keep ? (key >> 20) : 0xFFFFFFFFu;
      const unsigned peers = __match_any_sync(kFull, bin);
      if (keep && lane == __ffs(peers) - 1) atomicAdd(&hist0[bin], (uint32_t)__popc(peers));
    }
  }
  if (span) {
    __syncthreads();
    span_end(span);
  }
}

template <typename T, int C>
cudaError_t launch_c(const FuseArgs& a, cudaStream_t st) {
  const size_t smem = sizeof(float) * kHeadOut * C;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int warps = kThreads / 32;
  constexpr int NC = 4;
  int blocks = (a.cells + warps * NC - 1) / (warps * NC);
  if (blocks > sms) blocks = sms;
  if (blocks < 1) blocks = 1;
  const float isc = 1.0f / sqrtf((float)C);
  T* fused = static_cast<T*>(a.fused);
  auto kern = a.attention ? k_fuse_head<T, C, true> : k_fuse_head<T, C, false>;
  if (smem > 48 * 1024)
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  return launch_pdl(kern, dim3(blocks), dim3(kThreads), smem, st, a.feats, a.present, a.K,
                    a.cells, isc, a.head_wp, a.head_b, a.head_out, fused, a.keys, a.hist0,
                    a.cls_thresh, a.anchors, a.span);
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
  if (a.K < 1 || a.K > RTCC_MAX_AGENTS || a.anchors < 1 || a.anchors > kHeadOut) return cudaErrorInvalidValue;
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

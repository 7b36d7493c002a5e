// Cross-agent fusion of every backbone block's output, the first step of the
// shared post-join subgraph when the multi-scale maps are fused before the
// neck (the fusion/upsampling/concatenation placement of Sec. IV-A and the
// agent-indexed slots of Sec. IV-D): for each block b and each of its BEV
// cells, the present agents' C_b-channel vectors are fused -- per-channel max,
// or scaled dot-product attention with the ego agent 0 as the query -- and
// the fused vector is stored in the storage type.  The neck then runs once on
// the fused maps.
//
// Each thread owns 8 channels (16 bytes) of one cell, so the C_b / 8 threads
// of a cell read each agent's vector with one coalesced 16-byte load apiece
// and a warp covers 32 * 8 / C_b consecutive cells.  The kernel is bound by
// HBM bandwidth: every present agent's block outputs are read once and the
// fused maps written once.  One launch covers all blocks (warp tasks are
// numbered block after block).
//   max:        F = max_k X_k elementwise (exact in the 16-bit domain; the
//               block outputs are ReLU outputs, so a running max from +0
//               equals the max over the present agents)
//   attention:  s_k = <X_0, X_k> / sqrt(C_b), w = softmax over present k,
//               F = sum_k w_k X_k   (fp32; the dot product is each thread's
//               fused multiply-adds, then a butterfly over the cell's
//               threads, so every thread holds the same s_k; the softmax is
//               taken online in one pass over the agents)
// Every reduction has a fixed order: the result is bit-reproducible.
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace rtcc {

namespace {

constexpr unsigned kFull = 0xFFFFFFFFu;
constexpr int kThreads = 256;

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

__device__ __forceinline__ uint4 ld16(const void* p) { return *reinterpret_cast<const uint4*>(p); }

// One thread's 8 * NV channels (NV 16-byte vectors) of one cell.  G threads
// share the cell (C = 8 * NV * G); they are lanes [g0, g0 + G) of the warp.
template <typename T, bool ATTN, int G, int NV>
__device__ __forceinline__ void fuse_vec(const T* src, long long astride, const unsigned pres, int K,
                                         size_t off, float inv_sqrt_c, uint4* out) {
  if (!ATTN) {
#pragma unroll
    for (int v = 0; v < NV; ++v) out[v] = make_uint4(0u, 0u, 0u, 0u);
    for (int k = 0; k < K; ++k) {
      if (!((pres >> k) & 1u)) continue;
#pragma unroll
      for (int v = 0; v < NV; ++v) {
        const uint4 r = ld16(src + (size_t)k * astride + off + 8 * v);
        out[v].x = max2<T>(out[v].x, r.x);
        out[v].y = max2<T>(out[v].y, r.y);
        out[v].z = max2<T>(out[v].z, r.z);
        out[v].w = max2<T>(out[v].w, r.w);
      }
    }
  } else {
    // one pass over the present agents in index order, softmax online: a
    // running maximum m of the scores, the denominator and the weighted sum
    // rescaled by exp(m_old - m_new) when m grows (the ego agent 0, always
    // present, starts them).  The ego vector stays packed (16-bit pairs) for
    // the dot products, so each agent's vector is read once and few
    // registers stay live.
    constexpr int E = 8 * NV;
    uint32_t q[4 * NV];
#pragma unroll
    for (int v = 0; v < NV; ++v) {
      const uint4 r = ld16(src + off + 8 * v);
      q[4 * v] = r.x;
      q[4 * v + 1] = r.y;
      q[4 * v + 2] = r.z;
      q[4 * v + 3] = r.w;
    }
    float F[E], m = 0.f, den = 0.f;
#pragma unroll
    for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
      if (k < K && ((pres >> k) & 1u)) {
        uint32_t x[4 * NV];
        if (k == 0) {
#pragma unroll
          for (int i = 0; i < 4 * NV; ++i) x[i] = q[i];
        } else {
#pragma unroll
          for (int v = 0; v < NV; ++v) {
            const uint4 r = ld16(src + (size_t)k * astride + off + 8 * v);
            x[4 * v] = r.x;
            x[4 * v + 1] = r.y;
            x[4 * v + 2] = r.z;
            x[4 * v + 3] = r.w;
          }
        }
        float d = 0.f;
#pragma unroll
        for (int i = 0; i < 4 * NV; ++i) {
          const float2 a = Store<T>::unpack2(q[i]), b = Store<T>::unpack2(x[i]);
          d = fmaf(a.x, b.x, d);
          d = fmaf(a.y, b.y, d);
        }
#pragma unroll
        for (int o = G / 2; o > 0; o >>= 1) d += __shfl_xor_sync(kFull, d, o);
        const float sk = d * inv_sqrt_c;
        if (k == 0) {
          m = sk;
          den = 1.f;
#pragma unroll
          for (int i = 0; i < 4 * NV; ++i) {
            const float2 b = Store<T>::unpack2(x[i]);
            F[2 * i] = b.x;
            F[2 * i + 1] = b.y;
          }
        } else {
          const float mn = fmaxf(m, sk);
          const float sc = expf(m - mn), wk = expf(sk - mn);
          m = mn;
          den = fmaf(den, sc, wk);
#pragma unroll
          for (int i = 0; i < 4 * NV; ++i) {
            const float2 b = Store<T>::unpack2(x[i]);
            F[2 * i] = fmaf(F[2 * i], sc, wk * b.x);
            F[2 * i + 1] = fmaf(F[2 * i + 1], sc, wk * b.y);
          }
        }
      }
    }
    const float inv = 1.f / den;
#pragma unroll
    for (int v = 0; v < NV; ++v) {
      out[v].x = Store<T>::pack2(F[8 * v + 0] * inv, F[8 * v + 1] * inv);
      out[v].y = Store<T>::pack2(F[8 * v + 2] * inv, F[8 * v + 3] * inv);
      out[v].z = Store<T>::pack2(F[8 * v + 4] * inv, F[8 * v + 5] * inv);
      out[v].w = Store<T>::pack2(F[8 * v + 6] * inv, F[8 * v + 7] * inv);
    }
  }
}

// Warp task w of block b: cells [w * 32 / G, (w + 1) * 32 / G) of that block.
template <typename T, bool ATTN, int G, int NV>
__device__ __forceinline__ void block_task(const FuseBlocksArgs& a, int b, int w, int lane, unsigned pres) {
  constexpr int CPW = 32 / G;                       // cells per warp task
  const int cell = w * CPW + lane / G;
  const bool valid = cell < a.cells[b];
  // lanes of a cell past the end still join the butterfly (their data is a
  // clamped copy of the last cell and is not stored)
  const int c = valid ? cell : a.cells[b] - 1;
  const size_t off = (size_t)c * (8 * NV * G) + (size_t)(lane % G) * (8 * NV);
  uint4 v[NV];
  fuse_vec<T, ATTN, G, NV>(static_cast<const T*>(a.src[b]), a.astride[b], pres, a.K, off, a.inv_sqrt_c[b], v);
  if (valid) {
#pragma unroll
    for (int i = 0; i < NV; ++i) reinterpret_cast<uint4*>(static_cast<T*>(a.dst[b]) + off)[i] = v[i];
  }
}

static_assert(RTCC_MAX_BLOCKS == 3, "the task numbering below covers three blocks");

// WIDE: one 384-channel map (the single-scale 384-channel slots; 16 threads of
// 24 channels per cell); otherwise block maps of 32 to 256 channels.  The max
// of the block maps runs 5 blocks per SM (more loads in flight: stress8's
// three maps 12.8 -> 10.7 us against 3 blocks); attention keeps 3 (80
// registers).
template <typename T, bool ATTN, bool WIDE>
__global__ void __launch_bounds__(kThreads, (ATTN || WIDE) ? 3 : 5) k_fuse_blocks(const __grid_constant__ FuseBlocksArgs a) {
  pdl_trigger();
  pdl_wait();
  span_begin(a.span);
  unsigned pres = 0;
  for (int k = 0; k < a.K; ++k) pres |= (a.present[k] ? 1u : 0u) << k;
  const int lane = threadIdx.x & 31;
  const int warps = (int)(gridDim.x * blockDim.x) >> 5;
  // warp tasks of the blocks, numbered block after block
  const int e0 = a.tasks[0];
  const int e1 = e0 + (a.n > 1 ? a.tasks[1] : 0);
  const int e2 = e1 + (a.n > 2 ? a.tasks[2] : 0);
  for (int t = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5); t < e2; t += warps) {
    const int b = t < e0 ? 0 : (t < e1 ? 1 : 2);
    const int w = t - (b == 0 ? 0 : (b == 1 ? e0 : e1));
    if (WIDE) {
      block_task<T, ATTN, 16, 3>(a, b, w, lane, pres);
    } else {
      switch (a.ch[b]) {                             // warp-uniform
        case 32: block_task<T, ATTN, 4, 1>(a, b, w, lane, pres); break;
        case 64: block_task<T, ATTN, 8, 1>(a, b, w, lane, pres); break;
        case 128: block_task<T, ATTN, 16, 1>(a, b, w, lane, pres); break;
        default: block_task<T, ATTN, 32, 1>(a, b, w, lane, pres); break;
      }
    }
  }
  if (a.span) {
    __syncthreads();
    span_end(a.span);
  }
}

}  // namespace

cudaError_t launch_fuse_blocks(FuseBlocksArgs a, bool bf16, cudaStream_t st) {
  if (a.K < 1 || a.K > RTCC_MAX_AGENTS || a.n < 1 || a.n > RTCC_MAX_BLOCKS) return cudaErrorInvalidValue;
  long long work = 0;
  const bool wide = a.ch[0] == 384;
  if (wide && a.n != 1) return cudaErrorInvalidValue;
  for (int b = 0; b < a.n; ++b) {
    if (!wide && a.ch[b] != 32 && a.ch[b] != 64 && a.ch[b] != 128 && a.ch[b] != 256)
      return cudaErrorInvalidValue;
    if (a.cells[b] < 1 || !a.src[b] || !a.dst[b] || a.astride[b] < (long long)a.cells[b] * a.ch[b])
      return cudaErrorInvalidValue;
    // 16-byte loads and stores: every base and the agent stride 16-byte aligned
    if ((reinterpret_cast<uintptr_t>(a.src[b]) | reinterpret_cast<uintptr_t>(a.dst[b])) & 15u ||
        (a.astride[b] * 2) % 16)
      return cudaErrorInvalidValue;
    const int cpw = wide ? 2 : 32 / (a.ch[b] / 8);   // cells per warp task
    a.tasks[b] = (a.cells[b] + cpw - 1) / cpw;
    a.inv_sqrt_c[b] = 1.0f / sqrtf((float)a.ch[b]);
    work += a.tasks[b];
  }
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long long per_block = kThreads / 32;
  long long blocks = (work + per_block - 1) / per_block;
  if (blocks > 8LL * sms) blocks = 8LL * sms;       // grid-stride beyond 8 blocks per SM
  if (blocks < 1) blocks = 1;
  const dim3 g((unsigned)blocks), t(kThreads);
  if (bf16) {
    if (wide)
      return a.attention ? launch_pdl(k_fuse_blocks<__nv_bfloat16, true, true>, g, t, 0, st, a)
                         : launch_pdl(k_fuse_blocks<__nv_bfloat16, false, true>, g, t, 0, st, a);
    return a.attention ? launch_pdl(k_fuse_blocks<__nv_bfloat16, true, false>, g, t, 0, st, a)
                       : launch_pdl(k_fuse_blocks<__nv_bfloat16, false, false>, g, t, 0, st, a);
  }
  if (wide)
    return a.attention ? launch_pdl(k_fuse_blocks<__half, true, true>, g, t, 0, st, a)
                       : launch_pdl(k_fuse_blocks<__half, false, true>, g, t, 0, st, a);
  return a.attention ? launch_pdl(k_fuse_blocks<__half, true, false>, g, t, 0, st, a)
                     : launch_pdl(k_fuse_blocks<__half, false, false>, g, t, 0, st, a);
}

}  // namespace rtcc

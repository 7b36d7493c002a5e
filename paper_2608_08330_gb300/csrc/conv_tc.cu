// Persistent implicit-GEMM backbone of one encoder branch on the 5th-
// generation tensor cores (tcgen05, accumulators in tensor memory), fed by TMA.
// One launch runs every 3x3 conv (stride 1 and 2, zero padding 1) and every
// transposed conv with kernel = stride (the PointPillars neck) of a branch,
// each followed by bias + ReLU (Sec. III-B: the per-agent encoder E_k).
//
// GEMM view of a layer, one work item per (128-pixel tile, BN output
// channels, K slice):
//   D[m][n] = sum_k A[m][k] * B[n][k],  m = pixel, n = output channel,
//   k = (tap, input channel), tap-major.
// A (activations, NHWC) is never materialised: for each tap the producer
// issues a TMA box load of the input shifted by the tap's offset; TMA fills
// out-of-image elements with zeros, which is exactly the zero padding.  Stride
// 2 uses a 5-D view of the same tensor, (2C, W/2, 2, H/2, 1), in which the
// stride-2 gather becomes a unit-stride box at a tap-dependent (channel half,
// column, row parity, row) offset.  B (weights) is pre-packed K-major.
//
// The grid is one CTA per SM, co-resident (cooperative launch).  Work items of
// a layer are dealt round-robin over the CTAs; each CTA counts itself in the
// layer's arrival counter once its part of the layer is written, and a layer
// whose input another CTA writes starts once the counter of the layer it
// depends on shows every CTA (one counter per layer: a CTA with no work in
// some layers runs ahead and must not be counted for a layer it has not
// reached in the others' order).  Keeping the CTAs resident replaces
// sixteen kernel boundaries (each a full drain and relaunch) by counter waits,
// and lets the TMA/MMA pipeline and the tensor-memory allocation carry across
// tiles and layers.
//
// Roles (192 threads): warp 0 = TMA producer, warp 1 = tensor-memory owner and
// MMA issuer, warps 2..5 = epilogue.  Tensor memory holds two 128-column
// accumulators, so the epilogue of one tile overlaps the MMAs of the next.
// The epilogue adds bias, applies ReLU, rounds to 16 bits and writes each
// pixel's channels from registers (16-byte stores; a CTA's stores are then
// published by one release-ordered count).  Split-K slices of a tile are
// summed in slice order (through distributed shared memory, else global
// memory), so results do not depend on timing.  Every
// wait is bounded; one that runs out sets a bit in the error word and the CTA
// winds down instead of hanging.
#include <algorithm>
#include <cstring>
#include <mutex>
#include <type_traits>
#include <vector>

#include "common.cuh"
#include "kernels.h"

namespace rtcc {

namespace {

constexpr int TW = 8;                        // tile width in pixels: one 8-row MMA atom per image row
constexpr int TH = 16;                       // tile height
constexpr int kTallTH = 2 * TH;              // height of a tall tile: two MMA row blocks
constexpr int kWideTW = 2 * TW;              // wide tile of a tap-box layer: 16 x 8 = BM pixels,
constexpr int kWideTH = TH / 2;              // two MMA atoms per image row of its dense boxes
constexpr int BM = TW * TH;                  // 128 = MMA M
// warps: 0 TMA producer, 1 MMA issuer, 2..5 epilogue, 6..7 more TMA producers
constexpr int kThreads = 256;
constexpr int kProducers = 3;
constexpr int kFirstExtraProducer = 6;
constexpr int kStages = 5;
constexpr int kABytes = BM * 64 * 2;         // A slot (BK <= 64)
constexpr int kBBytes = 128 * 64 * 2;        // B slot (BN <= 128, BK <= 64)
// taps of 64 channels one B slot holds at N tile bn (a halo layer's stage)
__host__ __device__ constexpr int kStageTaps(int bn) { return kBBytes / (bn * 128); }
// Halo tiles (3x3 stride-1 convs with 64-channel k-blocks): the (TW+2) x
// (th+2) input pixels of a tile for one 64-channel chunk, 128 bytes each in
// the 128-byte swizzle; kHalo slots (sized for a tall tile) reuse the A area.
constexpr int kHaloW = TW + 2, kHaloH = TH + 2, kHaloHTall = kTallTH + 2;
constexpr int kHaloBytes = kHaloW * kHaloH * 128;
constexpr int kHaloBytesTall = kHaloW * kHaloHTall * 128;
constexpr int kHaloSlot = 44 * 1024;         // 1024-byte aligned (128-byte swizzle atoms)
constexpr int kHalo = 2;
// the lower row block of a tall tile starts TH halo rows further in (16-byte units)
constexpr uint32_t kTallHalfDesc = (uint32_t)(TH * kHaloW * 128 / 16);
constexpr int kAArea = 88 * 1024;            // A area: kStages tap-box slots or kHalo halo slots
constexpr int kBOff = kAArea;                // the A area, then the B slots
static_assert(kStages * kABytes <= kAArea, "tap-box slots must fit the A area");
static_assert(kHaloBytesTall <= kHaloSlot && kHalo * kHaloSlot <= kAArea, "halo slots must fit the A area");
constexpr int kStagingBytes = 56 * 1024;     // DSMEM split-K exchange: the outgoing slots
                                             // (4 x 128 x 16 fp32) and the receive slots
                                             // (3 x 128 x 16 fp32); deconvs: the output
                                             // tile (128 x 128 channels, 16-bit)
constexpr int kSmem = kAArea + kStages * kBBytes + kStagingBytes + 1024 + 256;
// two accumulators of 256 columns: a tall tile's row blocks at +0 and +128
constexpr uint32_t kAccStride = 256;
constexpr uint32_t kTmemCols = 2 * kAccStride;

// bias + ReLU of 16 fp32 values, packed to 16 bits and written as two
// 16-byte stores to dst (16-byte aligned: the channel offset is a multiple of
// 16 and the pixel stride a multiple of 8 channels); nothing for a pixel
// outside the image (dst null).
template <typename T>
__device__ __forceinline__ void store16(T* dst, const float* v, const float* bias) {
  if (!dst) return;
  uint32_t pk[8];
#pragma unroll
  for (int j = 0; j < 8; ++j)
    pk[j] = Store<T>::pack2(relu_f(v[2 * j] + bias[2 * j]), relu_f(v[2 * j + 1] + bias[2 * j + 1]));
  uint4* o = reinterpret_cast<uint4*>(dst);
  o[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
  o[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
}

// bias + ReLU of 16 fp32 columns [c0, c0+16) of tile row `row`, packed to
// 16 bits and written to the staging tile: a [BM][64]-channel block per 64
// columns, 128-byte rows in the 128-byte swizzle of the deconv store map, so
// a warp's 16-byte writes spread over all banks.
template <typename T>
__device__ __forceinline__ void stage16(uint8_t* stage, int row, int c0, const float* v, const float* bias) {
  uint32_t pk[8];
#pragma unroll
  for (int j = 0; j < 8; ++j)
    pk[j] = Store<T>::pack2(relu_f(v[2 * j] + bias[2 * j]), relu_f(v[2 * j + 1] + bias[2 * j + 1]));
  uint8_t* base = stage + (c0 / 64) * (BM * 128) + row * 128;
  const int j0 = (c0 % 64) / 8;                        // 16-byte chunk within the row
  const int x = row & 7;
  *reinterpret_cast<uint4*>(base + ((j0 ^ x) << 4)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
  *reinterpret_cast<uint4*>(base + (((j0 + 1) ^ x) << 4)) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
}

// The epilogue threads that issue a deconv item's TMA box stores: the first
// thread of each of the bn / 64 first epilogue warps (one 64-channel box each).
__device__ __forceinline__ bool deconv_storer(int row, int bn) { return (row & 31) == 0 && row < bn / 2; }

// barrier among the 4 epilogue warps only (named barrier 1, 128 threads)
__device__ __forceinline__ void epilogue_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// Release-ordered additions to a grid-wide counter: the writes this thread
// made before are visible to any thread that reads the new value with acquire
// semantics.  The reduction form does not wait for the old value.
__device__ __forceinline__ void red_add_release_gpu(unsigned* ctr, unsigned v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(ctr), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned atom_add_release_gpu(unsigned* ctr, unsigned v) {
  unsigned old;
  asm volatile("atom.release.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(ctr), "r"(v) : "memory");
  return old;
}

// Wait until the grid-wide arrival counter reaches `target` (bounded).
__device__ __forceinline__ bool grid_wait(const unsigned* ctr, unsigned target, long long budget) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
  if (v >= target) return true;
  const long long t0 = clock64();
  while (true) {
    __nanosleep(64);
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
    if (v >= target) return true;
    if (clock64() - t0 > budget) return false;
  }
}

// The scalars of one layer, read once per layer into registers.  The layer
// table lives in kernel parameter space and is indexed by the (dynamic) layer
// number; re-reading its fields inside the k-loops (every asm statement with a
// memory clobber forces a reload) costs a constant-cache round trip each.
struct LayerScalars {
  const float* bias;
  float* ws;
  int* counters;
  int kind, cin, cout, s, bn, bk, splits;
  int tiles_x, m_tiles, n_tiles, choff, wait_layers;
  int n_items, total_kb;
  int ncb_log2;            // log2(cin / bk): k-block kb = (tap << ncb_log2) + channel block
  int dsm;                 // split-K slices reduced through distributed shared memory
  int cta_lo, cta_hi;      // CTAs the items are dealt to
  int wait_items;          // target of the awaited layer's counter
  int halo;                // A from halo tiles; k-blocks chunk-major (kb = 9 chunk + tap)
  int tall;                // halo layers: tiles of TW x kTallTH pixels (two MMA row blocks
                           // sharing every weight box) instead of TW x TH
  int tw_log2, th;         // tile width (a power of two) and height in tile coordinates
  int tr;                  // tile coordinates transposed: tile x runs along the image's
                           // rows (H), tile y along W (halo layers)
  int kpb;                 // k-blocks per pipeline stage: halo layers put the weight boxes of
                           // kBBytes / (bn * 128) taps into one stage, others 1 (A + B)
  int spc;                 // halo layers: stages per 64-channel chunk (a stage never spans
                           // two chunks)
  void* out;               // output [agent][.][ow][ldc], 16-bit
  long long out_astride;   // elements between agents in out
  int ow, ldc, gw, gh;     // output row length (pixels), pixel stride (channels), tile grid extent
  int ipa;                 // items per agent
  int deconv_idx;
  int n_batch;
};
__device__ __forceinline__ LayerScalars layer_scalars(const LayerDesc& D, int n_batch) {
  LayerScalars S;
  S.bias = D.bias;
  S.ws = D.ws;
  S.counters = D.counters;
  S.kind = D.kind;
  S.cin = D.cin;
  S.cout = D.cout;
  S.s = D.s;
  S.bn = D.bn;
  S.bk = D.bk;
  S.splits = D.splits;
  S.tiles_x = D.tiles_x;
  S.m_tiles = D.m_tiles;
  S.n_tiles = D.n_tiles;
  S.choff = D.choff;
  S.wait_layers = D.wait_layers;
  S.dsm = D.dsm;
  S.cta_lo = D.cta_lo;
  S.cta_hi = D.cta_hi;
  S.wait_items = D.wait_items;
  S.halo = D.halo;
  S.tall = D.tall;
  S.tw_log2 = __ffs(D.tw) - 1;
  S.th = D.th;
  S.tr = D.tr;
  S.out = D.out;
  S.out_astride = D.out_astride;
  S.ipa = D.ipa;
  S.deconv_idx = D.deconv_idx;
  S.n_batch = n_batch;
  S.ow = D.ow;
  S.ldc = D.ldc;
  S.gw = D.gw;
  S.gh = D.gh;
  S.kpb = S.halo ? kStageTaps(S.bn) : 1;
  S.spc = (9 + S.kpb - 1) / S.kpb;
  S.n_items = n_batch * S.ipa;
  S.ncb_log2 = __ffs(S.cin / S.bk) - 1;            // cin / bk is a power of two
  S.total_kb = (S.kind == DECONV ? 1 : 9) << S.ncb_log2;
  return S;
}

// This CTA's first item of a layer (-1: none); its later items follow every
// cta_hi - cta_lo items.
__device__ __forceinline__ int first_item(const LayerScalars& S) {
  const int b = (int)blockIdx.x;
  if (b < S.cta_lo || b >= S.cta_hi) return -1;
  return b - S.cta_lo < S.n_items ? b - S.cta_lo : -1;
}

// Work item t of a layer -> (batch slot j, tile = (m tile, n tile), K slice
// z), its agent, its tile origin and its k-block range [kb0, kb1).  Items
// run agent-major, and within an agent the slice index runs fastest, so the
// slices of a tile are consecutive items: with one item per CTA and a grid of
// clusters of kMaxSplits CTAs they share a cluster, slice z on rank z (an
// agent's item count is a multiple of the slice count).
struct Item {
  int x0, y0, n0, z, tile, kb0, kb1, slot, agent;
};
__device__ __forceinline__ Item item_of(const LayerScalars& S, int t, const int* agents) {
  Item it;
  it.slot = t / S.ipa;
  it.agent = agents[it.slot];
  t -= it.slot * S.ipa;
  it.z = t % S.splits;
  it.tile = t / S.splits;
  const int mt = it.tile % S.m_tiles;
  const int nt = it.tile / S.m_tiles;
  it.x0 = (mt % S.tiles_x) << S.tw_log2;
  it.y0 = (mt / S.tiles_x) * (S.tall ? kTallTH : S.th);
  it.n0 = nt * S.bn;
  it.kb0 = (it.z * S.total_kb) / S.splits;
  it.kb1 = ((it.z + 1) * S.total_kb) / S.splits;
  return it;
}

// Pipeline stages of an item and the k-blocks [*k0, *k0 + *n) of its stage j.
// Tap-box layers: one k-block per stage.  Halo layers: the item holds whole
// 64-channel chunks, each split into spc stages of up to kpb taps.
__device__ __forceinline__ int item_stages(const LayerScalars& S, const Item& I) {
  return S.halo ? (I.kb1 - I.kb0) / 9 * S.spc : I.kb1 - I.kb0;
}
__device__ __forceinline__ void stage_kbs(const LayerScalars& S, const Item& I, int j, int* k0, int* n) {
  if (!S.halo) {
    *k0 = I.kb0 + j;
    *n = 1;
    return;
  }
  const int c = j / S.spc, q = j - c * S.spc;
  *k0 = I.kb0 + 9 * c + q * S.kpb;
  *n = min(S.kpb, 9 - q * S.kpb);
}

// TMA load of the activation (A) box of k-block kb of item I.
__device__ __forceinline__ void load_a(const LayerScalars& S, const CUtensorMap* map, uint8_t* dA,
                                       uint64_t* bar, const Item& I, int kb) {
  const int tap = kb >> S.ncb_log2;
  const int cb = kb - (tap << S.ncb_log2);
  if (S.kind == CONV3_S1) {
    const int dy = tap / 3, dx = tap - 3 * (tap / 3);
    tma_load_4d(dA, map, bar, cb * S.bk, I.x0 + dx - 1, I.y0 + dy - 1, I.agent);
  } else if (S.kind == CONV3_S2) {
    // input x = 2*ox + dx - 1 = 2*j + p; input y = 2*oy + dy - 1 = 2*i + q
    const int dy = tap / 3, dx = tap - 3 * (tap / 3);
    const int j = I.x0 + (dx == 0 ? -1 : 0);
    const int p = (dx == 1) ? 0 : 1;
    const int i = I.y0 + (dy == 0 ? -1 : 0);
    const int q = (dy == 1) ? 0 : 1;
    tma_load_5d(dA, map, bar, p * S.cin + cb * S.bk, j, q, i, I.agent);
  } else {
    tma_load_4d(dA, map, bar, cb * S.bk, I.x0, I.y0, I.agent);
  }
}

// TMA load of the weight (B) box starting at k-block kb of item I.  Conv
// weights are packed tap-major, [tap][Cout][Cin], and mapped as a 3-D tensor
// (Cin, Cout, tap): the box (bk channels, bn rows, taps) at (cb * bk, n0, tap)
// lands as one bn x bk operand per tap, bn * bk * 2 bytes apart (a halo
// layer's stage loads its kpb consecutive taps of one chunk in one box; map
// decides the tap count).  Deconv weights stay [(sub-position, Cout)][Cin].
__device__ __forceinline__ void load_b(const LayerScalars& S, const CUtensorMap* map, uint8_t* dB,
                                       uint64_t* bar, const Item& I, int kb) {
  if (S.kind == DECONV) {
    tma_load_2d(dB, map, bar, kb * S.bk, I.n0);
  } else if (S.halo) {
    const int cb = kb / 9, tap = kb - 9 * cb;
    tma_load_3d(dB, map, bar, cb * 64, I.n0, tap);
  } else {
    const int tap = kb >> S.ncb_log2;
    const int cb = kb - (tap << S.ncb_log2);
    tma_load_3d(dB, map, bar, cb * S.bk, I.n0, tap);
  }
}

// TMA load of the halo tile of 64-channel chunk cb of item I: input pixels
// [x0 - 1, x0 + TW] x [y0 - 1, y0 + TH]; out-of-image pixels read as zero,
// which is the zero padding.  Tap (dy, dx) of the tile is then the A operand
// starting (dy * kHaloW + dx) rows into it, with kHaloW rows between the
// 8-row atoms: the hardware applies the 128-byte swizzle to the final shared
// memory address, so a start at any 128-byte row matches the TMA placement.
__device__ __forceinline__ void load_halo(const CUtensorMap* map, uint8_t* dH, uint64_t* bar,
                                          const Item& I, int cb) {
  tma_load_4d(dH, map, bar, cb * 64, I.x0 - 1, I.y0 - 1, I.agent);
}

// One k-block of MMAs (BK = 64 or 32 -> 4 or 2 MMAs of K = 16).  The
// issuing thread cannot issue an MMA before the tensor pipe takes the
// previous one, so every instruction between them adds to the k-block's time;
// one asm statement keeps that to one add per operand.  The descriptors come
// as 32-bit halves: advancing K by 16 elements = 32 bytes is +2 in the
// 16-byte address field of the low half (the start stays inside its stage,
// so the field does not overflow), and the high half (stride, swizzle) is the
// same for every MMA of an operand.
__device__ __forceinline__ void mma_kblock(uint32_t d_tmem, uint32_t a_lo, uint32_t a_hi, uint32_t b_lo,
                                           uint32_t b_hi, uint32_t idesc, uint32_t acc0, bool bk64) {
  if (bk64) {
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t.reg .b64 a, b;\n\t.reg .b32 al, bl;\n\t"
        "setp.ne.b32 p, %5, 0;\n\t"
        "setp.eq.b32 q, %5, %5;\n\t"
        "mov.b64 a, {%1, %2};\n\tmov.b64 b, {%3, %4};\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %6, p;\n\t"
        "add.u32 al, %1, 2;\n\tadd.u32 bl, %3, 2;\n\t"
        "mov.b64 a, {al, %2};\n\tmov.b64 b, {bl, %4};\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %6, q;\n\t"
        "add.u32 al, %1, 4;\n\tadd.u32 bl, %3, 4;\n\t"
        "mov.b64 a, {al, %2};\n\tmov.b64 b, {bl, %4};\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %6, q;\n\t"
        "add.u32 al, %1, 6;\n\tadd.u32 bl, %3, 6;\n\t"
        "mov.b64 a, {al, %2};\n\tmov.b64 b, {bl, %4};\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %6, q;\n\t}" ::"r"(d_tmem),
        "r"(a_lo), "r"(a_hi), "r"(b_lo), "r"(b_hi), "r"(acc0), "r"(idesc));
  } else {
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t.reg .b64 a, b;\n\t.reg .b32 al, bl;\n\t"
        "setp.ne.b32 p, %5, 0;\n\t"
        "setp.eq.b32 q, %5, %5;\n\t"
        "mov.b64 a, {%1, %2};\n\tmov.b64 b, {%3, %4};\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %6, p;\n\t"
        "add.u32 al, %1, 2;\n\tadd.u32 bl, %3, 2;\n\t"
        "mov.b64 a, {al, %2};\n\tmov.b64 b, {bl, %4};\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %6, q;\n\t}" ::"r"(d_tmem),
        "r"(a_lo), "r"(a_hi), "r"(b_lo), "r"(b_hi), "r"(acc0), "r"(idesc));
  }
}

// The MMAs of one 64-channel chunk of a halo layer's item: the 9 taps fully
// unrolled, so every descriptor offset is an immediate and the MMAs issue
// back to back; a stage of kpb taps (km = kpb - 1) starts with a wait on its
// weight box and ends with a commit that frees it.  TALL: the tile's lower
// row block (accumulator columns +128) takes the same weight box with the A
// rows TH halo rows further down.  TR: the halo tile is stored in transposed
// tile coordinates (tile x along the image's H), so image tap (dy, dx) starts
// dx * kHaloW + dy rows into it instead of dy * kHaloW + dx.  False if a wait
// runs out.
template <bool TALL, bool TR>
__device__ __forceinline__ bool halo_chunk_mma(uint32_t d_tmem, uint32_t a_lo, uint32_t a_hi, uint32_t b_lo0,
                                               uint32_t b_hi, uint32_t idesc, int km, uint32_t bstep,
                                               bool accumulate, uint64_t* full, uint64_t* empty, uint32_t& it,
                                               long long budget) {
  uint32_t b_lo = 0;
  int s = 0;
#pragma unroll
  for (int tap = 0; tap < 9; ++tap) {
    if ((tap & km) == 0) {
      s = it % kStages;
      if (!mbar_wait(&full[s], (it / kStages) & 1, budget)) return false;
      tc_fence_after();
      b_lo = b_lo0 + (uint32_t)(s * (kBBytes >> 4));
    }
    const int tap_y = TR ? tap % 3 : tap / 3, tap_x = TR ? tap / 3 : tap % 3;
    const uint32_t a_tap = a_lo + (uint32_t)((tap_y * kHaloW + tap_x) * 8);
    const uint32_t b_tap = b_lo + (uint32_t)(tap & km) * bstep;
    const uint32_t accum = (accumulate || tap > 0) ? 1u : 0u;
    mma_kblock(d_tmem, a_tap, a_hi, b_tap, b_hi, idesc, accum, true);
    if (TALL) mma_kblock(d_tmem + 128, a_tap + kTallHalfDesc, a_hi, b_tap, b_hi, idesc, accum, true);
    if (((tap + 1) & km) == 0 || tap == 8) {
      umma_commit(&empty[s]);
      ++it;
    }
  }
  return true;
}

template <typename T>
__global__ void __launch_bounds__(kThreads, 1) k_backbone(const __grid_constant__ BackboneParams P) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* stage = smem + kAArea + kStages * kBBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(stage + kStagingBytes);
  uint64_t* empty = full + kStages;
  uint64_t* accfull = empty + kStages;         // [2]
  uint64_t* accempty = accfull + 2;            // [2]
  uint64_t* recvbar = accempty + 2;            // partials received through DSMEM
  uint64_t* hfull = recvbar + 1;               // [kHalo] halo tiles
  uint64_t* hempty = hfull + kHalo;            // [kHalo]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(hempty + kHalo);
  __shared__ int s_last;
  __shared__ float s_bias[2][128];             // bias of the tile in each accumulator
  __shared__ int s_agents[RTCC_MAX_AGENTS];    // the launch's agents (batch slot -> agent)
  const long long budget = P.wait_budget;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // The DSMEM reduction needs the launch to be in clusters of kMaxSplits CTAs;
  // the cluster size is read from the hardware, not trusted from the
  // parameters, and without such clusters split layers reduce through global
  // memory (the workspace exists for every split layer).
  const uint32_t ncl = cluster_nctarank();
  const bool clustered = ncl == (uint32_t)kMaxSplits;

  if (threadIdx.x < RTCC_MAX_AGENTS) s_agents[threadIdx.x] = P.agents[threadIdx.x];
  if (warp == 0 && lane == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&accfull[a], 1);
      mbar_init(&accempty[a], 4);              // one arrival per epilogue warp
    }
    mbar_init(recvbar, 1);                     // the owner's arrival + the peers' bytes
    for (int h = 0; h < kHalo; ++h) {
      mbar_init(&hfull[h], 1);
      mbar_init(&hempty[h], 1);
    }
    fence_barrier_init();
    if (ncl > 1) fence_mbar_init_cluster();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  if (ncl > 1) cluster_sync_all();            // peers' barriers are initialised
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();
  // the pseudo-image is the previous kernel's output; the producers wait for
  // it only after they have issued layer 0's weight boxes
  const bool producer_warp = warp == 0 || warp >= kFirstExtraProducer;
  if (!producer_warp) pdl_wait();

  if (producer_warp) {
    if (lane == 0) {
      // ---------------- TMA producers (one thread in each of kProducers warps) ----------------
      // One thread's TMA boxes complete one after another, each in about the
      // same time whatever its size (measured on GB300: ~600 clocks), so a
      // single issuing thread cannot keep the tensor pipe fed.  The boxes are
      // dealt over kProducers threads: pipeline stage u (its A and B boxes,
      // or a halo layer's one weight box of kpb taps) to thread
      // u % kProducers, and a chunk's halo tile to the thread of the chunk's
      // first stage, issued just before that stage.  Every thread walks the
      // same sequence of layers, items and stages and issues only its own.
      const uint32_t pid = (warp == 0) ? 0u : (uint32_t)(warp - kFirstExtraProducer + 1);
      uint32_t it = 0, hc = 0;                   // stages (B ring) and halo tiles so far
      int a_mode = 0;                            // last user of the A area: 1 tap boxes, 2 halo tiles
      bool alive = true, waited_pdl = false;
      // test hook: one wait for an item that never comes (read once)
      unsigned stall = (P.stall && *P.stall != 0) ? 1u : 0u;
      for (int l = 0; l < P.n_layers && alive; ++l) {
        const LayerDesc& D = P.L[l];
        const LayerScalars S = layer_scalars(D, P.n_batch);
        const CUtensorMap* mapA = &D.mapA;
        const CUtensorMap* mapB = &D.mapB;
        const CUtensorMap* mapB1 = &D.mapB1;
        tma_prefetch_desc(mapA);
        tma_prefetch_desc(mapB);
        if (S.halo) tma_prefetch_desc(mapB1);
        // bytes landing on a stage's barrier: the tap box and the weight box,
        // or for a layer that reads halo tiles (they have their own barriers)
        // the weight box of the stage's taps
        const uint32_t bbox = (uint32_t)S.bn * S.bk * 2;       // one tap's weight rows
        const uint32_t bytes = (uint32_t)(BM * S.bk * 2) + bbox;
        // The weights do not depend on the previous layer: load the B boxes
        // of the first stages of this CTA's first item before waiting for
        // the layer's input, so only the A boxes remain after the wait.
        const int t0 = first_item(S), tstep = S.cta_hi - S.cta_lo;
        if (t0 < 0) continue;                    // no items here: no wait, no count
        const Item I0 = item_of(S, t0, s_agents);
        int npre = item_stages(S, I0);
        if (npre > kStages) npre = kStages;
        for (int j = 0; j < npre; ++j) {
          const uint32_t u = it + j;
          if (u % kProducers != pid) continue;
          const int s = u % kStages;
          if (!mbar_wait(&empty[s], ((u / kStages) & 1) ^ 1, budget)) {
            atomicOr(P.err, ERR_WAIT_PRODUCER);
            alive = false;
            break;
          }
          int k0, n;
          stage_kbs(S, I0, j, &k0, &n);
          mbar_arrive_expect_tx(&full[s], S.halo ? bbox * n : bytes);
          load_b(S, (S.halo && n < S.kpb) ? mapB1 : mapB, smem + kBOff + s * kBBytes, &full[s], I0, k0);
        }
        if (!alive) break;
        if (!waited_pdl) {                       // the pseudo-image is the previous kernel's output
          pdl_wait();
          waited_pdl = true;
        }
        if (S.wait_layers > 0) {
          // every item of the layer this one reads has been stored
          if (!grid_wait(&P.grid_bar[S.wait_layers - 1], (unsigned)S.wait_items + stall, budget)) {
            atomicOr(P.err, ERR_WAIT_PRODUCER);
            alive = false;
            break;
          }
          stall = 0;
          fence_async_global();
        }
        // Tap boxes and halo tiles share the A area: before it changes use,
        // the MMAs that read it must be done.  The issuer commits every stage
        // after its MMAs, halo tiles included, so the release of the last stage
        // implies the rest.  This thread may get here before another producer
        // has even issued the last stages, so it waits for the releases of the
        // last kStages stages in order: each wait then finds its barrier's
        // previous phase complete, and the phase parity cannot alias.
        const int mode = S.halo ? 2 : 1;
        if (a_mode != 0 && a_mode != mode && it > 0) {
          for (uint32_t x = it > (uint32_t)kStages ? it - kStages : 0u; x < it && alive; ++x) {
            if (!mbar_wait(&empty[x % kStages], (x / kStages) & 1, budget)) {
              atomicOr(P.err, ERR_WAIT_PRODUCER);
              alive = false;
            }
          }
          if (!alive) break;
        }
        a_mode = mode;
        if (P.stamps && t0 == 0 && pid == 0) P.stamps[l] = global_ns();
        if (S.halo) {
          // Halo tiles in the order the MMAs use them: this CTA's items, chunk
          // by chunk, tile k + kHalo in the slot of tile k once tile k's MMAs
          // are done.  The layer's first tile goes out right after the
          // dependency wait; tile k + 1 goes out with the trigger stage of
          // chunk k (its 5th, or its last if shorter), from that stage's
          // thread: that thread has just seen the release of the stage 5
          // earlier, so chunk k - 1 is done (tile k + 1's slot is free) and
          // the tile has a chunk of MMAs to land.
          const int nch = (I0.kb1 - I0.kb0) / 9;       // chunks per item (the same for all)
          const int n_halos = ((S.n_items - 1 - t0) / tstep + 1) * nch;
          const uint32_t hbytes = S.tall ? (uint32_t)kHaloBytesTall : (uint32_t)kHaloBytes;
          const int trig = S.spc < 5 ? S.spc - 1 : 4;
          const uint32_t hc0 = hc;
          // tile k of this layer (the threads take turns, so each works out
          // the tile's item itself)
          auto issue_halo = [&](int k) -> bool {
            const uint32_t hk = hc0 + (uint32_t)k;
            const int h = hk % kHalo;
            if (!mbar_wait(&hempty[h], ((hk / kHalo) & 1) ^ 1, budget)) return false;
            const int i = k / nch, c = k - i * nch;
            const Item In = (i == 0) ? I0 : item_of(S, t0 + i * tstep, s_agents);
            mbar_arrive_expect_tx(&hfull[h], hbytes);
            load_halo(mapA, smem + h * kHaloSlot, &hfull[h], In, In.kb0 / 9 + c);
            return true;
          };
          if (it % kProducers == pid && !issue_halo(0)) {
            atomicOr(P.err, ERR_WAIT_PRODUCER);
            break;
          }
          int k = 0;                                    // chunk index in this layer
          for (int t = t0; t < S.n_items && alive; t += tstep) {
            const Item I = (t == t0) ? I0 : item_of(S, t, s_agents);
            for (int c = 0; c < nch && alive; ++c, ++k) {
              for (int q = 0; q < S.spc && alive; ++q, ++it) {
                if (it % kProducers != pid) continue;
                const int j = c * S.spc + q;
                if (!(t == t0 && j < npre)) {           // weights not already in flight
                  int k0, n;
                  stage_kbs(S, I, j, &k0, &n);
                  const int s = it % kStages;
                  if (!mbar_wait(&empty[s], ((it / kStages) & 1) ^ 1, budget)) {
                    atomicOr(P.err, ERR_WAIT_PRODUCER);
                    alive = false;
                    break;
                  }
                  mbar_arrive_expect_tx(&full[s], bbox * n);
                  load_b(S, n < S.kpb ? mapB1 : mapB, smem + kBOff + s * kBBytes, &full[s], I, k0);
                }
                if (q == trig && k + 1 < n_halos && !issue_halo(k + 1)) {
                  atomicOr(P.err, ERR_WAIT_PRODUCER);
                  alive = false;
                  break;
                }
              }
            }
          }
          hc = hc0 + (uint32_t)n_halos;
        } else {
          for (int t = t0; t < S.n_items && alive; t += tstep) {
            const Item I = (t == t0) ? I0 : item_of(S, t, s_agents);
            for (int kb = I.kb0; kb < I.kb1; ++kb, ++it) {
              if (it % kProducers != pid) continue;
              const int s = it % kStages;
              uint8_t* dA = smem + s * kABytes;
              if (t == t0 && kb - I.kb0 < npre) {
                load_a(S, mapA, dA, &full[s], I, kb);         // B already in flight
                continue;
              }
              if (!mbar_wait(&empty[s], ((it / kStages) & 1) ^ 1, budget)) {
                atomicOr(P.err, ERR_WAIT_PRODUCER);
                alive = false;
                break;
              }
              mbar_arrive_expect_tx(&full[s], bytes);
              load_a(S, mapA, dA, &full[s], I, kb);
              load_b(S, mapB, smem + kBOff + s * kBBytes, &full[s], I, kb);
            }
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer (one thread) ----------------
      uint32_t it = 0, tc = 0, hc = 0;
      bool alive = true;
      const uint32_t smem0 = smem_u32(smem);
      for (int l = 0; l < P.n_layers && alive; ++l) {
        const LayerScalars S = layer_scalars(P.L[l], P.n_batch);
        const uint32_t idesc = idesc_f16(BM, S.bn, std::is_same<T, __nv_bfloat16>::value);
        const bool bk64 = S.bk == 64;
        const uint32_t swz = bk64 ? 2u : 4u;            // 128B : 64B swizzle
        const uint32_t sbo = 8u * S.bk * 2u;            // bytes between 8-row atoms
        // descriptor halves of the first A and B slots (the slots of a stage
        // s are kABytes / kBBytes further on) and of the halo slots
        const uint64_t ad0 = smem_desc(smem0, sbo, swz), bd0 = smem_desc(smem0 + kBOff, sbo, swz);
        const uint32_t a_lo0 = (uint32_t)ad0, a_hi = (uint32_t)(ad0 >> 32);
        const uint32_t b_lo0 = (uint32_t)bd0, b_hi = (uint32_t)(bd0 >> 32);
        const uint32_t a_hi_halo = (uint32_t)(smem_desc(smem0, kHaloW * 128, 2u) >> 32);
        const int t0 = first_item(S), tstep = S.cta_hi - S.cta_lo;
        for (int t = t0; t >= 0 && t < S.n_items && alive; t += tstep, ++tc) {
          const Item I = item_of(S, t, s_agents);
          const int acc = tc & 1;
          if (!mbar_wait(&accempty[acc], ((tc >> 1) & 1) ^ 1, budget)) {
            atomicOr(P.err, ERR_WAIT_MMA);
            alive = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem + acc * kAccStride;
          if (S.halo) {
            // Chunk by chunk: wait for the halo tile, then the 9 taps fully
            // unrolled, so every descriptor offset is an immediate and the
            // MMAs issue back to back; a stage of kpb taps starts with a wait
            // on its weight boxes and ends with a commit that frees it.  A
            // tall tile's lower row block (accumulator columns +128) takes the
            // same weight box with the A rows TH halo rows further down.
            const bool tall = S.tall != 0;
            const int nch = (I.kb1 - I.kb0) / 9;
            const int km = S.kpb - 1;
            const uint32_t bstep = (uint32_t)(S.bn * 8);        // one weight box, 16-byte units
            for (int c = 0; c < nch && alive; ++c) {
              const int h = hc % kHalo;
              if (!mbar_wait(&hfull[h], (hc / kHalo) & 1, budget)) {
                atomicOr(P.err, ERR_WAIT_MMA);
                alive = false;
                break;
              }
              ++hc;
              const uint32_t a_lo = (uint32_t)smem_desc(smem0 + h * kHaloSlot, kHaloW * 128, 2u);
              const bool acc_in = c > 0;
              const bool ok =
                  tall ? (S.tr ? halo_chunk_mma<true, true>(d_tmem, a_lo, a_hi_halo, b_lo0, b_hi, idesc, km, bstep,
                                                            acc_in, full, empty, it, budget)
                               : halo_chunk_mma<true, false>(d_tmem, a_lo, a_hi_halo, b_lo0, b_hi, idesc, km,
                                                             bstep, acc_in, full, empty, it, budget))
                       : (S.tr ? halo_chunk_mma<false, true>(d_tmem, a_lo, a_hi_halo, b_lo0, b_hi, idesc, km,
                                                             bstep, acc_in, full, empty, it, budget)
                               : halo_chunk_mma<false, false>(d_tmem, a_lo, a_hi_halo, b_lo0, b_hi, idesc, km,
                                                              bstep, acc_in, full, empty, it, budget));
              if (!ok) {
                atomicOr(P.err, ERR_WAIT_MMA);
                alive = false;
                break;
              }
              umma_commit(&hempty[h]);
            }
          } else {
            for (int kb = I.kb0; kb < I.kb1; ++kb, ++it) {
              const int s = it % kStages;
              if (!mbar_wait(&full[s], (it / kStages) & 1, budget)) {
                atomicOr(P.err, ERR_WAIT_MMA);
                alive = false;
                break;
              }
              tc_fence_after();
              mma_kblock(d_tmem, a_lo0 + (uint32_t)(s * (kABytes >> 4)), a_hi,
                         b_lo0 + (uint32_t)(s * (kBBytes >> 4)), b_hi, idesc, kb > I.kb0 ? 1u : 0u, bk64);
              umma_commit(&empty[s]);
            }
          }
          umma_commit(&accfull[acc]);
        }
      }
    }
  } else {
    // ---------------- epilogue ----------------
    const int qd = warp & 3;                   // tensor-memory lane quarter of this warp
    const int row = qd * 32 + lane;            // pixel within the tile
    // The four epilogue warps meet at named barriers, so they never leave the
    // loops early: after a wait runs out they skip further waits (the values
    // are then garbage, the error word says so) but keep the same sequence of
    // barriers and grid arrivals.
    uint32_t tc = 0, dsm_phase = 0;
    bool alive = true;
    for (int l = 0; l < P.n_layers; ++l) {
      const LayerScalars S = layer_scalars(P.L[l], P.n_batch);
      const int t0 = first_item(S), tstep = S.cta_hi - S.cta_lo;
      if (t0 < 0) continue;                    // no items here: no count
      int mine = 0;
      for (int t = t0; t < S.n_items; t += tstep, ++tc, ++mine) {
        const Item I = item_of(S, t, s_agents);
        const int acc = tc & 1;
        // bias of this tile, read while the MMAs run (the slot was last read
        // two tiles ago, before the barriers in between)
        if (row < S.bn) s_bias[acc][row] = S.bias[(S.kind == DECONV ? 0 : I.n0) + row];
        if (alive && !mbar_wait(&accfull[acc], (tc >> 1) & 1, budget)) {
          if (lane == 0) atomicOr(P.err, ERR_WAIT_EPILOGUE);
          alive = false;
        }
        tc_fence_after();
        const float* bias = s_bias[acc];
        const uint32_t taddr = tmem + acc * kAccStride + (static_cast<uint32_t>(qd * 32) << 16);
        // This row's output pixel (the tile's row-th pixel; for a deconv one
        // sub-pixel position of its input pixel), written straight from
        // registers: channels [n0, n0 + bn) of a conv, [choff, choff + cout)
        // of a deconv.  Null outside the image (ragged tiles).
        T* orow = nullptr;
        {
          const int px = I.x0 + (row & ((1 << S.tw_log2) - 1)), py = I.y0 + (row >> S.tw_log2);
          if (px < S.gw && py < S.gh) {
            size_t pix;
            int c0;
            if (S.kind == DECONV) {
              const int sub = I.n0 / S.cout;
              const int sy = sub / S.s, sx = sub - sy * S.s;
              pix = (size_t)(py * S.s + sy) * S.ow + (size_t)(px * S.s + sx);
              c0 = S.choff;
            } else {
              pix = S.tr ? (size_t)px * S.ow + py : (size_t)py * S.ow + px;
              c0 = S.choff + I.n0;
            }
            orow = static_cast<T*>(S.out) + (size_t)I.agent * S.out_astride + pix * S.ldc + c0;
          }
        }
        // the previous item's bulk copies (DSMEM exchange) or tile stores
        // (deconv) must have read the shared memory they came from
        if ((S.dsm && row == 0) || (S.kind == DECONV && deconv_storer(row, S.bn))) bulk_wait_read_all();
        epilogue_sync();
        if (S.splits == 1) {
          // up to 64 columns per round: issue all TMEM loads, wait once; a
          // tall tile's lower row block (TH image rows further down) follows
          // from accumulator columns +128
          const int halves = S.tall ? 2 : 1;
          for (int hh = 0; hh < halves; ++hh) {
            T* o = orow;
            if (hh > 0) {
              // tall tiles are TW wide
              const int px = I.x0 + row % TW, py = I.y0 + TH + row / TW;
              const size_t pix = S.tr ? (size_t)px * S.ow + py : (size_t)py * S.ow + px;
              o = (px < S.gw && py < S.gh)
                      ? static_cast<T*>(S.out) + (size_t)I.agent * S.out_astride + pix * S.ldc + S.choff + I.n0
                      : nullptr;
            }
            const uint32_t ta = taddr + (uint32_t)(hh * 128);
            for (int c0 = 0; c0 < S.bn; c0 += 64) {
              const int ng = (S.bn - c0) / 16 < 4 ? (S.bn - c0) / 16 : 4;   // uniform
              uint32_t r[4][16];
#pragma unroll
              for (int g = 0; g < 4; ++g)
                if (g < ng) tmem_ld16_issue(ta + c0 + 16 * g, r[g]);
              tmem_ld_wait();
#pragma unroll
              for (int g = 0; g < 4; ++g) {
                if (g < ng) {
                  tmem_reg_fence(r[g]);
                  float v[16];
#pragma unroll
                  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[g][i]);
                  if (S.kind == DECONV)
                    stage16<T>(stage, row, c0 + 16 * g, v, bias + c0 + 16 * g);
                  else
                    store16<T>(o ? o + c0 + 16 * g : nullptr, v, bias + c0 + 16 * g);
                }
              }
            }
          }
        } else if (S.dsm && clustered) {
          // The Sp = splits (2 or 4) K-slices of this 64-wide tile sit on Sp
          // consecutive ranks of this cluster of four, slice z on rank gb + z.
          // Reduce-scatter through distributed shared memory: slice z owns the
          // CW = 64 / Sp output channels [CW z, CW (z + 1)).  Every rank writes
          // its 64 partial columns into its own shared memory by owner; one
          // bulk copy per peer moves the peer's slot into the peer's receive
          // slot (counted on the peer's mbarrier); each owner sums the slices in
          // slice order and stores its channels in 16-channel TMA boxes.  The
          // slots are rewritten only after the next item's bulk_wait_read_all.
          const int Sp = S.splits;
          const int CW = 64 / Sp, G16 = CW / 16;
          const int z = I.z;
          const uint32_t rank = cluster_ctarank();
          const uint32_t gb = rank & ~static_cast<uint32_t>(Sp - 1);
          if (row == 0 && (rank & static_cast<uint32_t>(Sp - 1)) != (uint32_t)z) atomicOr(P.err, ERR_BOUNDS);
          const int SLOT = BM * CW * 4;                          // one owner's channels, fp32
          uint8_t* own = stage;                                  // [Sp][BM][CW] fp32, by owner (32 KB)
          uint8_t* recv = stage + Sp * SLOT;                     // [Sp-1][BM][CW] fp32, from peers
          if (row == 0) mbar_arrive_expect_tx(recvbar, (uint32_t)((Sp - 1) * SLOT));
          // the row's 64 columns in one round of TMEM loads, into the owner slots
          uint32_t rq[4][16];
#pragma unroll
          for (int g = 0; g < 4; ++g) tmem_ld16_issue(taddr + 16 * g, rq[g]);
          tmem_ld_wait();
#pragma unroll
          for (int g = 0; g < 4; ++g) {
            tmem_reg_fence(rq[g]);
            const int q = g / G16, h = g - q * G16;
            uint4* o = reinterpret_cast<uint4*>(own + q * SLOT + (row * CW + h * 16) * 4);
#pragma unroll
            for (int j = 0; j < 4; ++j)
              o[j] = make_uint4(rq[g][4 * j], rq[g][4 * j + 1], rq[g][4 * j + 2], rq[g][4 * j + 3]);
          }
          fence_async_smem();                      // generic writes -> the bulk copies
          epilogue_sync();
          if (row == 0) {
            const uint32_t my_recv = smem_u32(recv), my_bar = smem_u32(recvbar);
            for (int q = 0; q < Sp; ++q) {
              if (q == z) continue;
              const int slot = z < q ? z : z - 1;  // this slice's receive slot at owner q
              bulk_copy_to_peer(mapa_shared(my_recv + (uint32_t)(slot * SLOT), gb + q), own + q * SLOT,
                                (uint32_t)SLOT, mapa_shared(my_bar, gb + q));
            }
            bulk_commit();
          }
          if (alive && !mbar_wait(recvbar, dsm_phase, budget)) {
            if (lane == 0) atomicOr(P.err, ERR_WAIT_EPILOGUE);
            alive = false;
          }
          dsm_phase ^= 1u;
          for (int h = 0; h < G16; ++h) {
            float sum[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) sum[j] = 0.f;
            for (int zz = 0; zz < Sp; ++zz) {
              const uint8_t* src = (zz == z) ? own + z * SLOT : recv + (zz < z ? zz : zz - 1) * SLOT;
              const float4* f4 = reinterpret_cast<const float4*>(src + (row * CW + h * 16) * 4);
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const float4 f = f4[q];
                sum[4 * q] += f.x;
                sum[4 * q + 1] += f.y;
                sum[4 * q + 2] += f.z;
                sum[4 * q + 3] += f.w;
              }
            }
            // bias + ReLU, 16-bit, the owner's 16 channels of this row
            store16<T>(orow ? orow + z * CW + h * 16 : nullptr, sum, bias + z * CW + h * 16);
          }
        } else {
          // publish this slice's fp32 partial ([bn/4][BM][4] per (slice, tile),
          // so a warp's float4 stores cover 512 contiguous bytes), then the
          // last slice of the tile sums the slices in slice order (tiles of
          // the batch's agents numbered slot-major)
          const int tiles = S.n_batch * S.m_tiles * S.n_tiles;
          const int tile_id = I.slot * S.m_tiles * S.n_tiles + I.tile;
          float4* mine =
              reinterpret_cast<float4*>(S.ws + (size_t)(I.z * tiles + tile_id) * BM * S.bn) + row;
          for (int c0 = 0; c0 < S.bn; c0 += 16) {
            float v[16];
            tmem_ld16(taddr + c0, v);
#pragma unroll
            for (int q = 0; q < 4; ++q)
              mine[(c0 / 4 + q) * BM] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          }
          __threadfence();
          epilogue_sync();
          if (row == 0) {
            const int old = atomicAdd(&S.counters[tile_id], 1);
            s_last = (old == S.splits - 1);
          }
          epilogue_sync();
          if (s_last != 0) {
            __threadfence();
            for (int c0 = 0; c0 < S.bn; c0 += 16) {
              // all other slices' loads of this column group in flight at once
              float4 f[kMaxSplits][4];
#pragma unroll
              for (int zz = 0; zz < kMaxSplits; ++zz) {
                if (zz < S.splits && zz != I.z) {
                  const float4* src =
                      reinterpret_cast<const float4*>(S.ws + (size_t)(zz * tiles + tile_id) * BM * S.bn) +
                      row;
#pragma unroll
                  for (int q = 0; q < 4; ++q) f[zz][q] = __ldcg(src + (c0 / 4 + q) * BM);
                }
              }
              float v[16];
              tmem_ld16(taddr + c0, v);
              float sum[16];
#pragma unroll
              for (int j = 0; j < 16; ++j) sum[j] = 0.f;
#pragma unroll
              for (int zz = 0; zz < kMaxSplits; ++zz) {
                if (zz < S.splits) {
                  if (zz == I.z) {
#pragma unroll
                    for (int j = 0; j < 16; ++j) sum[j] += v[j];
                  } else {
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                      sum[4 * q] += f[zz][q].x;
                      sum[4 * q + 1] += f[zz][q].y;
                      sum[4 * q + 2] += f[zz][q].z;
                      sum[4 * q + 3] += f[zz][q].w;
                    }
                  }
                }
              }
              store16<T>(orow ? orow + c0 : nullptr, sum, bias + c0);
            }
            if (row == 0) S.counters[tile_id] = 0;     // ready for the next launch
          }
        }
        // the accumulator has been read: hand it back to the MMA issuer
        tc_fence_before();
        if (lane == 0) mbar_arrive(&accempty[acc]);
        if (S.kind == DECONV) {
          // A deconv row is 128 channels at a strided sub-pixel position:
          // one 5-D TMA box store per 64 channels beats 16 stores per thread.
          // A thread's TMA operations complete one after another, so box g
          // goes out from the first thread of epilogue warp g.
          fence_async_smem();
          epilogue_sync();
          if (deconv_storer(row, S.bn)) {
            const int g = row / 32;
            const int sub = I.n0 / S.cout;
            const int sy = sub / S.s, sx = sub - sy * S.s;
            const CUtensorMap* mapC = &P.mapC[S.deconv_idx][I.agent];
            tma_store_5d(mapC, stage + g * BM * 128, S.choff + g * 64, sx, I.x0, sy, I.y0);
            bulk_commit();
          }
        }
      }
      // This CTA's items of layer l are stored: count them.  The epilogue
      // threads' stores are ordered before the count by the barrier and the
      // count's release semantics (cumulative over what the barrier made
      // visible to this thread), so a consumer that acquires the counter
      // sees them.  (With TMA stores, waiting for their completion and a
      // full __threadfence here cost about a microsecond per layer.)
      if (S.kind == DECONV && deconv_storer(row, S.bn)) {   // TMA stores: complete, then ordered
        bulk_wait_all();
        fence_async_global();
      }
      epilogue_sync();
      if (row == 0) {
        if (P.stamps) {
          const unsigned before = atom_add_release_gpu(&P.grid_bar[l], (unsigned)mine);
          // the CTA completing the layer's count stamps its end
          if (before + (unsigned)mine == (unsigned)S.n_items) P.stamps[P.n_layers + l] = global_ns();
        } else {
          red_add_release_gpu(&P.grid_bar[l], (unsigned)mine);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (ncl > 1) cluster_sync_all();            // no peer still writes into this CTA
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  // The last CTA to leave zeroes the counters for the next launch that uses
  // them (every other CTA is past its last wait and count) and reports the
  // launch's end to the host.
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned old = atomicAdd(&P.grid_bar[kMaxLayers], 1u);
    if (old == gridDim.x - 1) {
      for (int l = 0; l < P.n_layers; ++l) P.grid_bar[l] = 0u;
      P.grid_bar[kMaxLayers] = 0u;
      if (P.done_word) {
        __threadfence_system();
        *P.done_word = 1;
      }
    }
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

}  // namespace

cudaError_t tmap_2d(CUtensorMap* m, const void* base, bool bf16, uint64_t inner, uint64_t outer,
                    uint32_t box_inner, uint32_t box_outer, int swizzle_bytes) {
  EncodeFn enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  const CUtensorMapDataType dt =
      bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
  const CUtensorMapSwizzle sw = swizzle_bytes == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                                : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                      : CU_TENSOR_MAP_SWIZZLE_NONE;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  const CUresult r = enc(m, dt, 2, const_cast<void*>(base), dims, strides, box, es,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t tmap_3d(CUtensorMap* m, const void* base, bool bf16, uint64_t inner, uint64_t mid,
                    uint64_t outer, uint32_t box_inner, uint32_t box_mid, uint32_t box_outer,
                    int swizzle_bytes) {
  EncodeFn enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  const CUtensorMapDataType dt =
      bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
  const CUtensorMapSwizzle sw = swizzle_bytes == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                                : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                      : CU_TENSOR_MAP_SWIZZLE_NONE;
  cuuint64_t dims[3] = {inner, mid, outer};
  cuuint64_t strides[2] = {inner * 2, inner * mid * 2};
  cuuint32_t box[3] = {box_inner, box_mid, box_outer};
  cuuint32_t es[3] = {1, 1, 1};
  const CUresult r = enc(m, dt, 3, const_cast<void*>(base), dims, strides, box, es,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

int conv_tile_w() { return TW; }
int conv_tile_h() { return TH; }
int conv_tile_m() { return BM; }
// The tile grid of layer L: tile width and height, and the extent the tiles
// cover in tile coordinates (the image's W x H, or H x W when transposed).
static void tile_grid(const ConvLayer& L, int* tw, int* th, int* gx, int* gy) {
  *tw = L.wide ? kWideTW : TW;
  *th = L.tall ? kTallTH : L.wide ? kWideTH : TH;
  *gx = L.tr ? L.gh : L.gw;
  *gy = L.tr ? L.gw : L.gh;
}
int conv_m_tiles(const ConvLayer& L) {
  int tw, th, gx, gy;
  tile_grid(L, &tw, &th, &gx, &gy);
  return ((gx + tw - 1) / tw) * ((gy + th - 1) / th);
}
bool conv_shape_ok(const ConvLayer& L) {
  const bool halo = conv_uses_halo(L);
  if (L.tall && (!halo || L.splits != 1)) return false;
  if (L.tr && (!halo || L.splits != 1 || L.wide)) return false;
  if (L.wide && (L.kind == DECONV || halo || L.splits != 1)) return false;
  return true;
}

cudaError_t conv_make_maps(ConvLayer& L, bool bf16) {
  EncodeFn enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  const CUtensorMapDataType dt =
      bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
  const CUtensorMapSwizzle sw =
      (L.bk == 64) ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
  const cuuint64_t C = (cuuint64_t)L.cin, W = (cuuint64_t)L.in_w, H = (cuuint64_t)L.in_h;
  // the agents' inputs are one tensor, agent outermost
  const cuuint64_t NA = (cuuint64_t)(L.n_agents > 0 ? L.n_agents : 1);
  const cuuint64_t AS = (cuuint64_t)L.in_astride * 2;
  if (L.n_agents < 1 || L.n_agents > RTCC_MAX_AGENTS || L.in_astride < (long long)(C * W * H) ||
      (L.kind == DECONV && L.out_astride < (long long)L.out_w * L.out_h * L.ldc))
    return cudaErrorInvalidValue;
  CUresult r;
  if (!conv_shape_ok(L)) return cudaErrorInvalidValue;
  const cuuint32_t tw = (cuuint32_t)(L.wide ? kWideTW : TW), th = (cuuint32_t)(L.wide ? kWideTH : TH);
  if (L.kind == CONV3_S2) {
    if ((L.in_w & 1) || (L.in_h & 1)) return cudaErrorInvalidValue;
    cuuint64_t dims[5] = {2 * C, W / 2, 2, H / 2, NA};
    cuuint64_t strides[4] = {2 * C * 2, W * C * 2, 2 * W * C * 2, AS};
    cuuint32_t box[5] = {(cuuint32_t)L.bk, tw, 1, th, 1};
    cuuint32_t es[5] = {1, 1, 1, 1, 1};
    r = enc(&L.mapA, dt, 5, const_cast<void*>(L.in), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  } else {
    // transposed halo layers walk the image with H as the tile's x: the same
    // NHWC tensor described with its two pixel dimensions swapped
    cuuint64_t dims[4] = {C, L.tr ? H : W, L.tr ? W : H, NA};
    cuuint64_t strides[3] = {L.tr ? W * C * 2 : C * 2, L.tr ? C * 2 : W * C * 2, AS};
    const bool halo = conv_uses_halo(L);
    cuuint32_t box[4] = {(cuuint32_t)L.bk, (cuuint32_t)(halo ? kHaloW : tw),
                         (cuuint32_t)(halo ? (L.tall ? kHaloHTall : kHaloH) : th), 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    r = enc(&L.mapA, dt, 4, const_cast<void*>(L.in), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  }
  if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  if (L.kind == DECONV) {
    const cuuint64_t K = (cuuint64_t)L.cin;
    const cuuint64_t rows = (cuuint64_t)(L.s * L.s * L.cout);
    cuuint64_t bdims[2] = {K, rows};
    cuuint64_t bstr[1] = {K * 2};
    cuuint32_t bbox[2] = {(cuuint32_t)L.bk, (cuuint32_t)L.bn};
    cuuint32_t bes[2] = {1, 1};
    r = enc(&L.mapB, dt, 2, const_cast<void*>(L.wpacked), bdims, bstr, bbox, bes,
            CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    L.mapB1 = L.mapB;
  } else {
    // tap-major weights [9][Cout][Cin] as (Cin, Cout, tap): mapB carries a
    // halo layer's kpb taps per box (one tap otherwise), mapB1 one tap
    const int kpb = conv_uses_halo(L) ? kStageTaps(L.bn) : 1;
    if (kpb < 1) return cudaErrorInvalidValue;
    cuuint64_t bdims[3] = {(cuuint64_t)L.cin, (cuuint64_t)L.cout, 9};
    cuuint64_t bstr[2] = {(cuuint64_t)L.cin * 2, (cuuint64_t)L.cin * L.cout * 2};
    cuuint32_t bes[3] = {1, 1, 1};
    cuuint32_t bbox[3] = {(cuuint32_t)L.bk, (cuuint32_t)L.bn, (cuuint32_t)kpb};
    r = enc(&L.mapB, dt, 3, const_cast<void*>(L.wpacked), bdims, bstr, bbox, bes,
            CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    bbox[2] = 1;
    r = enc(&L.mapB1, dt, 3, const_cast<void*>(L.wpacked), bdims, bstr, bbox, bes,
            CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  }
  if (L.kind == DECONV) {
    // output store map of each agent: [in_h][s][in_w][s][ldc] view of its
    // output, so one sub-pixel position of a tile is one box of 64 channels
    // (a ragged tile's rows past in_h are clipped by the map, which an agent
    // dimension folded into in_h would not do)
    if (L.bn % 64) return cudaErrorInvalidValue;
    const cuuint64_t LD = (cuuint64_t)L.ldc, S = (cuuint64_t)L.s;
    const cuuint64_t IW = (cuuint64_t)L.in_w, IH = (cuuint64_t)L.in_h, OW = (cuuint64_t)L.out_w;
    cuuint64_t dims[5] = {LD, S, IW, S, IH};
    cuuint64_t strides[4] = {LD * 2, S * LD * 2, OW * LD * 2, S * OW * LD * 2};
    cuuint32_t box[5] = {64, 1, (cuuint32_t)TW, 1, (cuuint32_t)TH};
    cuuint32_t es[5] = {1, 1, 1, 1, 1};
    for (int k = 0; k < L.n_agents; ++k) {
      void* base = static_cast<uint8_t*>(L.out) + (size_t)k * (size_t)L.out_astride * 2;
      r = enc(&L.mapC[k], dt, 5, base, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    }
  }
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t backbone_fill(const std::vector<ConvLayer>& layers, int n_batch, unsigned* grid_bar,
                          int* err, unsigned long long* stamps, bool allow_clusters,
                          long long wait_budget, BackboneParams* P) {
  if (layers.empty() || layers.size() > (size_t)kMaxLayers) return cudaErrorInvalidValue;
  if (n_batch < 1 || n_batch > RTCC_MAX_AGENTS || n_batch > layers[0].n_agents || wait_budget < 1)
    return cudaErrorInvalidValue;
  std::memset(P, 0, sizeof(*P));
  P->n_layers = (int)layers.size();
  P->n_batch = n_batch;
  for (int j = 0; j < n_batch; ++j) P->agents[j] = j;
  P->grid_bar = grid_bar;
  P->err = err;
  P->stamps = stamps;
  P->wait_budget = wait_budget;
  const int grid_sm = backbone_grid(1), grid_cl = allow_clusters ? backbone_grid(kMaxSplits) : 0;
  if (grid_sm < 1) return cudaErrorInvalidValue;
  bool any_dsm = false;
  int n_deconv = 0;
  for (size_t i = 0; i < layers.size(); ++i) {
    const ConvLayer& L = layers[i];
    if (L.n_agents != layers[0].n_agents) return cudaErrorInvalidValue;
    const int ncb = L.bk > 0 ? L.cin / L.bk : 0;
    if (L.bk < 1 || L.cin % L.bk || ncb < 1 || (ncb & (ncb - 1)) ||   // a power of two
        (L.kind != DECONV && L.cout % L.bn) || (L.kind == DECONV && L.bn != L.cout) ||
        L.bn > 128 || L.bk > 64 || L.bn % 32)
      return cudaErrorInvalidValue;
    const int total_kb = (L.kind == DECONV ? 1 : 9) * (L.cin / L.bk);
    if (L.splits < 1 || L.splits > kMaxSplits || L.splits > total_kb || (L.splits > 1 && (!L.ws || !L.counters)))
      return cudaErrorInvalidValue;
    LayerDesc& D = P->L[i];
    D.mapA = L.mapA;
    D.mapB = L.mapB;
    D.mapB1 = L.mapB1;
    D.deconv_idx = -1;
    if (L.kind == DECONV) {
      if (n_deconv >= kMaxDeconv) return cudaErrorInvalidValue;
      D.deconv_idx = n_deconv;
      for (int k = 0; k < L.n_agents; ++k) P->mapC[n_deconv][k] = L.mapC[k];
      ++n_deconv;
    }
    D.bias = L.bias;
    D.ws = L.ws;
    D.counters = L.counters;
    D.kind = L.kind;
    D.cin = L.cin;
    D.cout = L.cout;
    D.s = L.s;
    D.bn = L.bn;
    D.bk = L.bk;
    D.splits = L.splits;
    if (!conv_shape_ok(L)) return cudaErrorInvalidValue;
    int tw, th, gx, gy;
    tile_grid(L, &tw, &th, &gx, &gy);
    D.tiles_x = (gx + tw - 1) / tw;
    D.m_tiles = conv_m_tiles(L);
    D.tall = L.tall ? 1 : 0;
    D.tw = tw;
    D.th = L.wide ? kWideTH : TH;
    D.tr = L.tr ? 1 : 0;
    D.n_tiles = L.n_tiles_n;
    D.choff = L.choff;
    D.wait_layers = L.wait_layers;
    D.out = L.out;
    D.out_astride = L.out_astride;
    D.ipa = D.m_tiles * D.n_tiles * L.splits;
    D.ow = L.out_w;
    D.ldc = L.ldc;
    D.gw = gx;
    D.gh = gy;
    D.halo = conv_uses_halo(L) ? 1 : 0;
    // a split of a 64-wide tile into 2 or kMaxSplits slices, one item per
    // CTA, reduces its slices through distributed shared memory within a
    // cluster of kMaxSplits CTAs
    D.dsm = (L.kind != DECONV && (L.splits == 2 || L.splits == kMaxSplits) && L.bn == 64 && grid_cl > 0 &&
             n_batch * D.ipa <= grid_cl)
                ? 1
                : 0;
    any_dsm = any_dsm || D.dsm;
  }
  P->cluster = any_dsm ? kMaxSplits : 1;
  P->grid = any_dsm ? grid_cl : grid_sm;
  // Item ranges.  Every layer's items are dealt round-robin over all CTAs,
  // except the deconvs of the shallower blocks (those that do not read the
  // deepest block): when the conv layers that can run at the same time as
  // such a deconv (those after the layer it reads) leave at least 8 CTAs
  // without items, those CTAs take the deconv, which then runs alongside the
  // deeper conv blocks instead of after them (a CTA with no items in a layer
  // skips it without waiting).  A layer waits for the items of the one layer
  // it reads.
  int last_conv = -1;
  for (int i = 0; i < P->n_layers; ++i)
    if (P->L[i].kind != DECONV) last_conv = i;
  for (int i = 0; i < P->n_layers; ++i) {
    LayerDesc& D = P->L[i];
    D.cta_lo = 0;
    D.cta_hi = P->grid;
    if (D.kind == DECONV && D.wait_layers >= 1 && D.wait_layers - 1 != last_conv) {
      int conc_max = 0;                            // conv items beside this deconv
      for (int j = D.wait_layers; j < P->n_layers; ++j)
        if (P->L[j].kind != DECONV) conc_max = std::max(conc_max, n_batch * P->L[j].ipa);
      if (P->grid - conc_max >= 8) D.cta_lo = conc_max;
    }
    if (D.wait_layers > P->n_layers || D.wait_layers > (int)i) return cudaErrorInvalidValue;
    D.wait_items = 0;
    if (D.wait_layers > 0) {
      const LayerDesc& W = P->L[D.wait_layers - 1];
      D.wait_items = n_batch * W.ipa;
    }
  }
  return cudaSuccess;
}

int backbone_grid(int cluster) {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
    return 0;
  if (cluster <= 1) return sms;
  static std::mutex mu;
  static int cached[64][2] = {};                  // per device: cluster size, grid
  std::lock_guard<std::mutex> lk(mu);
  if (dev < 64 && cached[dev][0] == cluster) return cached[dev][1];
  if (cudaFuncSetAttribute(k_backbone<__half>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           kSmem) != cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(sms - sms % cluster);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, k_backbone<__half>, &cfg) != cudaSuccess || n < 1) {
    (void)cudaGetLastError();
    return 0;
  }
  if (dev < 64) {
    cached[dev][0] = cluster;
    cached[dev][1] = n * cluster;
  }
  return n * cluster;
}

cudaError_t launch_backbone(const BackboneParams& P, bool bf16, cudaStream_t st) {
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [] {
    attr_err = cudaFuncSetAttribute(k_backbone<__half>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    kSmem);
    if (attr_err == cudaSuccess)
      attr_err = cudaFuncSetAttribute(k_backbone<__nv_bfloat16>,
                                      cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  });
  if (attr_err != cudaSuccess) return attr_err;
  if (P.grid < 1 || (P.cluster > 1 && P.grid % P.cluster)) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(P.grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmem;
  cfg.stream = st;
  cudaLaunchAttribute attr[3];
  int na = 0;
  attr[na].id = cudaLaunchAttributeCooperative;  // every CTA resident: grid barriers are safe
  attr[na++].val.cooperative = 1;
  // programmatic dependent launch: CTAs are scheduled while the pillar chain
  // drains and run their prologue (barriers, TMEM, cluster sync, first weight
  // boxes) before griddepcontrol.wait
  attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[na++].val.programmaticStreamSerializationAllowed = 1;
  if (P.cluster > 1) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = (unsigned)P.cluster;
    attr[na].val.clusterDim.y = 1;
    attr[na++].val.clusterDim.z = 1;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  if (bf16) return cudaLaunchKernelEx(&cfg, k_backbone<__nv_bfloat16>, P);
  return cudaLaunchKernelEx(&cfg, k_backbone<__half>, P);
}

}  // namespace rtcc

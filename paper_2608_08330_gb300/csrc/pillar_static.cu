// Allocation-free variant of the pillarisation + PFN + scatter pass.
//
// Some callers cannot allocate device memory at the point where they need
// this pass: code that runs while a CUDA stream is being captured into a graph
// (cudaMalloc is not a capturable operation), hosts that hand a plugin only
// pre-planned memory and no allocator, and latency-critical loops that must not
// risk the implicit device synchronisation an allocation can cause.  For them
// this entry point takes its scratch from one fixed array in device global
// memory that the library reserves when it is loaded, instead of calling any
// allocator.  The array is sized for grids up to 65,536 cells, payloads up to
// 131,072 points, 16,384 pillars of up to 32 points and 64 PFN channels (about
// 11.8 MB, held on every GPU that loads the library until the process exits).
//
// The kernels are the ones rtcc_payload_complete runs (launch_pillarise); only
// the scratch pointers differ.  All calls share the one array: a call clears
// what must start at zero (per-cell counters and first-point indices, the
// caller's stats) before it runs, and calls that overlap on the GPU -- on
// different streams, or from different host threads -- race on the array and
// must be serialised by the caller.
#include <mutex>

#include "kernels.h"
#include "rtcc.h"

namespace rtcc {
namespace {

constexpr int kMaxCells = 65536;
constexpr int kMaxPoints = 131072;
constexpr int kMaxPillars = 16384;
constexpr int kMaxCh = 64;
constexpr int kMaxPts = 32;
constexpr int kMaxTiles = (kMaxPoints + kScanTileMin - 1) / kScanTileMin;
constexpr size_t kPad = (kMaxPoints + kScanPadUnit - 1) / kScanPadUnit * kScanPadUnit + kScanPadUnit;

constexpr size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

constexpr size_t kOffN = 0;
constexpr size_t kOffCellOf = align256(kOffN + 16);
constexpr size_t kOffSlot = align256(kOffCellOf + 4ull * kPad);
constexpr size_t kOffList = align256(kOffSlot + 4ull * kPad);
constexpr size_t kOffTouched = align256(kOffList + 4ull * kMaxPoints);
constexpr size_t kOffBucket = align256(kOffTouched + 4ull * kMaxPoints);
constexpr size_t kOffCnt = align256(kOffBucket + 16ull * kMaxPillars * kMaxPts);
constexpr size_t kOffFirst = align256(kOffCnt + 4ull * kMaxCells);
constexpr size_t kOffLoc = align256(kOffFirst + 4ull * kMaxCells);
constexpr size_t kOffAgg = align256(kOffLoc + 8ull * kMaxCells);
constexpr size_t kOffPrec = align256(kOffAgg + 8ull * kMaxTiles * kAggStride);
constexpr size_t kOffNp = align256(kOffPrec + 16ull * kMaxPillars);
constexpr size_t kOffNt = align256(kOffNp + 16);
constexpr size_t kStaticBytes = align256(kOffNt + 16);

static __device__ __align__(256) unsigned char g_pillar_scratch[kStaticBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
unsigned char* g_addr[kMaxDevices] = {};

// Device address of the static array on the current device, looked up once
// per device (the symbol's host-side name is not a device address).
rtcc_status scratch_address(unsigned char** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return RTCC_E_CUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_pillar_scratch) != cudaSuccess || !p) return RTCC_E_CUDA;
    g_addr[dev] = static_cast<unsigned char*>(p);
  }
  *out = g_addr[dev];
  return RTCC_OK;
}

__global__ void k_static_reset(int n, int cells, int* __restrict__ n_slot,
                               int* __restrict__ cnt_cell, int* __restrict__ first_cell,
                               int* __restrict__ stats) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i == 0) *n_slot = n;
  if (i < 8) stats[i] = 0;
  for (int c = i; c < cells; c += gridDim.x * blockDim.x) {
    cnt_cell[c] = 0;
    first_cell[c] = kFirstInit;
  }
}

}  // namespace
}  // namespace rtcc

using namespace rtcc;

extern "C" rtcc_status rtcc_pillarise_noalloc(const rtcc_model_config* cfg, const float* d_points,
                                              int32_t n_points, const float* d_pfn_w,
                                              const float* d_pfn_b, int32_t* d_cell2pillar,
                                              int32_t* d_pillar_cell, int32_t* d_count,
                                              int32_t* d_stats, void* d_image, void* stream) {
  if (!cfg || !d_pfn_w || !d_pfn_b || !d_cell2pillar || !d_pillar_cell || !d_count ||
      !d_stats || !d_image || (n_points > 0 && !d_points))
    return RTCC_E_ARG;
  const long long cells = (long long)cfg->grid_w * cfg->grid_h;
  if (cfg->grid_w < 1 || cfg->grid_h < 1 || cells > kMaxCells) return RTCC_E_ARG;
  if (n_points < 0 || n_points > kMaxPoints) return RTCC_E_ARG;
  if (cfg->max_pillars < 1 || cfg->max_pillars > kMaxPillars) return RTCC_E_ARG;
  if (cfg->max_pts < 1 || cfg->max_pts > kMaxPts) return RTCC_E_ARG;
  if (cfg->pfn_ch != 32 && cfg->pfn_ch != kMaxCh) return RTCC_E_ARG;
  if (cfg->dtype != RTCC_FP16 && cfg->dtype != RTCC_BF16) return RTCC_E_ARG;
  if (!(cfg->pillar > 0.f)) return RTCC_E_ARG;
  if (!grid_coords_ok(cfg->x_min, cfg->y_min, cfg->z_min, cfg->z_max, cfg->pillar, cfg->grid_w,
                      cfg->grid_h))
    return RTCC_E_ARG;
  // The kernels read the points as float4 and clear the image with 16-byte
  // stores; a sub-view that is not so aligned is refused here instead of
  // faulting on the device.
  auto misaligned = [](const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) != 0; };
  if ((n_points > 0 && misaligned(d_points, 16)) || misaligned(d_image, 16) || misaligned(d_pfn_w, 4) ||
      misaligned(d_pfn_b, 4) || misaligned(d_cell2pillar, 4) || misaligned(d_pillar_cell, 4) ||
      misaligned(d_count, 4) || misaligned(d_stats, 4))
    return RTCC_E_ARG;
  unsigned char* base = nullptr;
  rtcc_status s = scratch_address(&base);
  if (s != RTCC_OK) return s;
  cudaStream_t st = static_cast<cudaStream_t>(stream);

  PillarBufs b{};
  b.pts = reinterpret_cast<const float4*>(d_points);
  b.n_hdr = reinterpret_cast<const int*>(base + kOffN);
  b.cell_of = reinterpret_cast<int*>(base + kOffCellOf);
  b.slot_of = reinterpret_cast<int*>(base + kOffSlot);
  b.cnt_cell = reinterpret_cast<int*>(base + kOffCnt);
  b.first_cell = reinterpret_cast<int*>(base + kOffFirst);
  b.cell_loc = reinterpret_cast<int2*>(base + kOffLoc);
  b.tile_agg = reinterpret_cast<unsigned long long*>(base + kOffAgg);
  b.pillar_rec = reinterpret_cast<int4*>(base + kOffPrec);
  b.touched = reinterpret_cast<int*>(base + kOffTouched);
  b.ntouched = reinterpret_cast<int*>(base + kOffNt);
  b.list = reinterpret_cast<int*>(base + kOffList);
  b.bucket = reinterpret_cast<float4*>(base + kOffBucket);
  b.np_prev = reinterpret_cast<int*>(base + kOffNp);
  b.pillar_cell = d_pillar_cell;
  b.pcount = d_count;
  b.stats = d_stats;
  b.zero_words = d_stats;                       // the first kernel clears the stats
  b.n_zero = 8;
  b.cell2pillar = d_cell2pillar;
  b.image = d_image;
  b.cap = n_points;
  b.P = cfg->max_pillars;
  b.N = cfg->max_pts;
  b.C = cfg->pfn_ch;
  b.clear_all = 1;                              // the caller's image and cell2pillar: unknown content

  int blocks = (int)((cells + 255) / 256);
  if (blocks < 1) blocks = 1;
  // cudaLaunchKernelEx reports this launch's own error; an error state the
  // caller's earlier work left on the thread is neither returned nor cleared
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3(blocks);
  lc.blockDim = dim3(256);
  lc.stream = st;
  if (cudaLaunchKernelEx(&lc, k_static_reset, n_points, (int)cells, reinterpret_cast<int*>(base + kOffN),
                         b.cnt_cell, b.first_cell, d_stats) != cudaSuccess)
    return RTCC_E_CUDA;
  GridGeom g{cfg->x_min, cfg->y_min, cfg->z_min, cfg->z_max, cfg->pillar, cfg->grid_w,
             cfg->grid_h};
  if (launch_pillarise(b, g, d_pfn_w, d_pfn_b, cfg->dtype == RTCC_BF16, st) !=
      cudaSuccess)
    return RTCC_E_CUDA;
  return RTCC_OK;
}

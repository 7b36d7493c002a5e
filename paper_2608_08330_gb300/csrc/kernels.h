// Host-side launch interface of the RTCC kernels (internal to the library).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "rtcc.h"

namespace rtcc {

// Pillar grid geometry (float32, as the points are).
struct GridGeom {
  float x_min, y_min, z_min, z_max, v;
  int W, H;
};

// Buffers of one pillarisation + PFN + scatter pass.  `cap` is the payload
// capacity in points; P = P_max, N = N_max, C = C_p.
struct PillarBufs {
  const float4* pts;     // [cap] device payload (x, y, z, intensity)
  const int* n_hdr;      // device: number of valid points
  // scratch
  int* cell_of;          // [cap]   cell of each point, -1 out of range
  int* cnt_cell;         // [H*W]   points per cell (0 between passes)
  int* first_cell;       // [H*W]   first point index per cell (kFirstInit between passes)
  int* c2p;              // [H*W]   pillar id of a cell (valid where cnt_cell > 0)
  int2* blocksum;        // [nblk]  per-tile (#first points, #points of their cells)
  int* pcnt_raw;         // [P]     points of the pillar's cell before the N_max cap
  int* poff;             // [P]     offset of the pillar's point list
  int* cursor;           // [P]     fill cursor
  int* list;             // [cap]   point indices grouped by pillar
  void* feat;            // [P][C]  pillar features (storage type)
  // outputs
  int* pillar_cell;      // [P]
  int* pcount;           // [P]     kept points
  int* stats;            // [8]     n, in_range, n_pillars, kept, 0, 0, ncap drops,
                         //         points of kept pillars before the N_max cap
  int* cell2pillar;      // [H*W]
  void* image;           // [H][W][C] storage type
  int cap, P, N, C;
};

constexpr int kFirstInit = 0x7F7F7F7F;   // memset byte 0x7F
constexpr int kScanTile = 4096;          // points per scan block
inline int scan_blocks(int cap) { return (cap + kScanTile - 1) / kScanTile; }

// Enqueue the 6 pillar kernels (cells, block sums, scan, fill, PFN, scatter).
cudaError_t launch_pillarise(const PillarBufs& b, const GridGeom& g, const float* pfn_w,
                             const float* pfn_b, bool bf16, int* err, cudaStream_t st);

// ---------------------------------------------------------------------------
// implicit-GEMM convolution on tcgen05 (3x3 stride 1/2 and deconv k = s)
// ---------------------------------------------------------------------------

enum ConvKind { CONV3_S1 = 0, CONV3_S2 = 1, DECONV = 2 };

struct ConvLayer {
  ConvKind kind;
  int cin, cout;         // conv: Cout; deconv: Cout per sub-position
  int s;                 // deconv stride (= kernel); 1 for convs
  int in_w, in_h;        // input map
  int out_w, out_h;      // output map
  int gw, gh;            // M grid the tiles cover (conv: output; deconv: input)
  int ldc, choff;        // output pixel stride (channels) and channel offset
  int bn, bk;            // N tile (output channels per CTA), K chunk (channels)
  int n_tiles_n;         // grid.y
  const void* in;        // device [in_h][in_w][cin]
  void* out;             // device [out_h][out_w][ldc]
  const void* wpacked;   // device, K-major: conv [Cout][9][Cin]; deconv [s*s*Cout][Cin]
  const float* bias;     // device [Cout]
  CUtensorMap mapA, mapB;
};

// Encode the layer's tensor maps (input activations and packed weights).
cudaError_t conv_make_maps(ConvLayer& L, bool bf16);
cudaError_t launch_conv(const ConvLayer& L, bool bf16, int* err, cudaStream_t st);
int conv_tile_w();
int conv_tile_h();

// ---------------------------------------------------------------------------
// post-join: fusion + head, decode
// ---------------------------------------------------------------------------

struct FuseArgs {
  const void* const* feats;  // device array [K] of slot pointers [H'W'][C]
  const int* present;        // device [K]
  int K, C, cells;
  int attention;             // 0 = max, 1 = ego-query attention
  const float* head_wp;      // device, permuted head weights (see fuse_head.cu)
  const float* head_b;       // device [16]
  float* head_out;           // device [cells][16]
  void* fused;               // device [cells][C] or null
};
cudaError_t launch_fuse_head(const FuseArgs& a, bool bf16, cudaStream_t st);
// Head weight permutation expected by the fusion kernel (host side).
void permute_head_weights(const float* w /*[16][C]*/, int C, float* out /*[16*C]*/);

struct DecodeArgs {
  const float* head;         // [cells][16]
  int feat_w, feat_h, anchors;
  float x_min, y_min, x_max, y_max;
  float cls_thresh;
  int max_boxes;
  unsigned long long* cand;  // [n_chunks][kDecodeKeep] keys, then [n_chunks] int counts
  const int* err;            // device error word, copied into the result header
  void* out;                 // device result block: DetResultHeader + rtcc_box[max_boxes]
};
constexpr int kDecodeChunk = 4096;
constexpr int kDecodeKeep = 512;     // >= max_boxes
int decode_chunks(int n_anchors);
cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t st);

// Result block the post-join graph copies to pinned host memory.
struct DetResultHeader {
  int n_boxes;
  int err;
  int pad[2];
};

}  // namespace rtcc

// Host-side launch interface of the RTCC kernels (internal to the library).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

#include "rtcc.h"

namespace rtcc {

// Launch `kern` on `st` with programmatic stream serialisation, so that it may
// begin while the previous kernel in the stream finishes (the kernel itself
// calls pdl_wait before touching shared data).  Captured into a graph, this
// becomes a programmatic dependency edge.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// Pillar grid geometry (float32, as the points are).
struct GridGeom {
  float x_min, y_min, z_min, z_max, v;
  int W, H;
  // fixed-point scales of the PFN's means (powers of two, set by
  // launch_pillarise): 32 x v x qxy and 32 x (z_max - z_min) x qz <= 2^30
  float qxy, qz, qxy_inv, qz_inv;
};

// Buffers of one pillarisation + PFN + scatter pass.  `cap` is the payload
// capacity in points; P = P_max, N = N_max, C = C_p.
struct PillarBufs {
  const float4* pts;     // [cap] device payload (x, y, z, intensity)
  const int* n_hdr;      // device: number of valid points
  // scratch
  int* cell_of;          // [scan_pad(cap)] cell of each point, -1 out of range
  int* slot_of;          // [scan_pad(cap)] the point's slot in its cell's list
  int* cnt_cell;         // [H*W]   points per cell (0 between passes)
  int* first_cell;       // [H*W]   first point index per cell (kFirstInit between passes)
  int2* cell_loc;        // [H*W]   per cell the pass opened: (tile << 12 | pillar rank
                         //         in the tile, list offset in the tile)
  unsigned long long* tile_agg;   // [scan_tiles(cap) * kAggStride] the scan's published tile
                                  // aggregates, one per 128-byte line
  int4* pillar_rec;      // [P]     (cell, points before the N_max cap, list offset,
                         //         column | row << 16)
  int* touched;          // [cap]   cell of every pillar id of the pass, kept or not
  int* ntouched;         // [1]     pillar ids of the pass
  int* list;             // [cap]   point indices grouped by pillar (pillars over N_max points)
  float4* bucket;        // [P][N]  the points of each pillar of at most N_max points
  int* np_prev;          // [1]     pillars the previous pass wrote into image and
                         //         cell2pillar (0 at allocation)
  int* err;              // optional: error word (a scan wait ran out: bit 32)
  // outputs
  int* pillar_cell;      // [P]
  int* pcount;           // [P]     kept points
  int* stats;            // [8]     n, in_range, n_pillars, kept, 0, 0, ncap drops,
                         //         points of kept pillars before the N_max cap
  int* zero_words;       // [n_zero] words the pass's first kernel clears; begins with
  int n_zero;            //         the 8 stats words (zero_words == stats, n_zero >= 8)
  int* cell2pillar;      // [H*W]     -1 where no kept pillar
  void* image;           // [H][W][C] storage type, zeros where no kept pillar
  int* present_flag;     // optional: set to 1 by the pass (the agent's slot is filled)
  unsigned long long* pfn_span;   // optional [3]: the PFN kernel's span stamps (span_begin)
  // optional zero-copy payload: the first kernel reads the header and points
  // from src_* (e.g. pinned host memory) and writes them to dst_* (= n_hdr,
  // pts) for the later kernels
  const int* src_hdr;
  const float4* src_pts;
  int* dst_hdr;
  float4* dst_pts;
  int cap, P, N, C;
  int clear_all;         // 1: the pass clears all of image and cell2pillar (their
                         // content is unknown); 0: they hold the previous pass's
                         // output, and only its np_prev pillar cells are cleared
};

constexpr int kFirstInit = 0x7F7F7F7F;   // memset byte 0x7F
// The scan takes tiles of 4 points per thread, 256 to 1024 threads.
constexpr int kScanTileMin = 1024;
constexpr int kAggStride = 16;           // words between two tiles' aggregates (one line each)
constexpr int kScanPadUnit = 4096;
// Most tiles a pass over cap points has; points the per-point scratch holds.
inline int scan_tiles(int cap) { return cap > 0 ? (cap + kScanTileMin - 1) / kScanTileMin : 1; }
inline size_t scan_pad(int cap) {   // whole tiles of any size up to 4096 points
  return ((size_t)(cap > 0 ? cap : 1) + kScanPadUnit - 1) / kScanPadUnit * kScanPadUnit +
         kScanPadUnit;
}
// Grid bounds the PFN's fixed-point means accept: every bound within 2^20
// pillar edges of 0 (and z within 2^20 z-ranges), so that float32 rounding
// keeps a point within one edge of its pillar's centre.
inline bool grid_coords_ok(double x_min, double y_min, double z_min, double z_max, double v,
                           int W, int H) {
  const double lim = v * 1048576.0, zlim = (z_max - z_min) * 1048576.0;
  auto in = [](double a, double l) { return a >= -l && a <= l; };
  return in(x_min, lim) && in(x_min + W * v, lim) && in(y_min, lim) && in(y_min + H * v, lim) &&
         in(z_min, zlim) && in(z_max, zlim);
}

// Enqueue the 3 pillar kernels (cells; scan + list fill; PFN, which writes
// each pillar's vector into the BEV pseudo-image).  The first kernel clears
// b.zero_words, so the caller needs no memset per pass.
cudaError_t launch_pillarise(const PillarBufs& b, const GridGeom& g, const float* pfn_w,
                             const float* pfn_b, bool bf16, cudaStream_t st);

// ---------------------------------------------------------------------------
// implicit-GEMM convolution on tcgen05 (3x3 stride 1/2 and deconv k = s)
// ---------------------------------------------------------------------------

enum ConvKind { CONV3_S1 = 0, CONV3_S2 = 1, DECONV = 2 };

struct ConvLayer {
  ConvKind kind;
  // Every agent's tensors of a layer live in one allocation, agent-major with
  // a fixed stride, so one tensor map covers all agents (the agent index is
  // the map's outermost coordinate) and a launch may run any set of agents.
  int n_agents;          // agents the buffers hold
  long long in_astride;  // elements between agents in `in`
  long long out_astride; // elements between agents in `out`
  int cin, cout;         // conv: Cout; deconv: Cout per sub-position
  int s;                 // deconv stride (= kernel); 1 for convs
  int in_w, in_h;        // input map
  int out_w, out_h;      // output map
  int gw, gh;            // M grid the tiles cover (conv: output; deconv: input)
  int ldc, choff;        // output pixel stride (channels) and channel offset
  int bn, bk;            // N tile (output channels per item), K chunk (channels)
  int n_tiles_n;         // N tiles
  int splits;            // split-K factor; 1 = none
  int tall;              // halo layers without split-K: tiles of 8 x 32 pixels, two
                         // 128-row MMAs per weight box (0: 8 x 16 pixels)
  int tr;                // halo layers without split-K: tiles walk the image transposed,
                         // 8 pixels along H by 16 (tall: 32) along W
  int wide;              // tap-box convs without split-K: tiles of 16 x 8 pixels
  int wait_layers;       // this layer reads outputs of layers [0, wait_layers)
  float* ws;             // split-K partials [batch][splits][m_tiles * n_tiles][128][bn] fp32
  int* counters;         // split-K arrivals per tile [batch][m_tiles * n_tiles], zero-initialised
  const void* in;        // device [agent][in_h][in_w][cin]
  void* out;             // device [agent][out_h][out_w][ldc]
  const void* wpacked;   // device, K-major: conv [9][Cout][Cin]; deconv [s*s*Cout][Cin]
  const float* bias;     // device [Cout]
  CUtensorMap mapA, mapB;         // input (tap boxes or halo tiles; outermost
                                  // coordinate = agent), packed weights (a halo
                                  // layer: boxes of a stage's taps)
  CUtensorMap mapB1;              // packed weights, one tap per box
  CUtensorMap mapC[RTCC_MAX_AGENTS];  // deconvs: output store map of each agent
};

// Encode the layer's tensor maps (input activations, packed weights).
cudaError_t conv_make_maps(ConvLayer& L, bool bf16);
// Whether the layer reads its A operand as halo tiles (one box per tile and
// 64-channel chunk, shared by the 9 taps) instead of one box per tap: 3x3
// stride-1 convs with 64-channel k-blocks whose K slices hold whole chunks.
inline bool conv_uses_halo(const ConvLayer& L) {
  return L.kind == CONV3_S1 && L.bk == 64 && L.splits >= 1 && (L.cin / 64) % L.splits == 0;
}
int conv_tile_w();
int conv_tile_h();                 // rows of a tile (a tall tile has twice as many)
int conv_tile_m();
// M tiles of layer L's grid with its tile shape
int conv_m_tiles(const ConvLayer& L);
// Whether L's tile shape flags (tall, tr, wide) fit its kind and split.
bool conv_shape_ok(const ConvLayer& L);

// One layer of the persistent backbone kernel (kernel-parameter layout).
constexpr int kMaxLayers = 20;
constexpr int kMaxDeconv = 3;     // neck deconvs (one per block)
constexpr int kMaxSplits = 4;     // split-K slices per tile (the reducing slice keeps one load per slice in flight)
struct alignas(128) LayerDesc {   // CUtensorMap is 128-byte aligned
  CUtensorMap mapA, mapB, mapB1;
  const float* bias;
  float* ws;
  int* counters;
  int kind, cin, cout, s, bn, bk, splits;
  int tiles_x, m_tiles, n_tiles, choff;
  int wait_layers;
  int dsm;                       // split-K slices reduced through distributed shared memory
  int cta_lo, cta_hi;            // the CTAs this layer's items are dealt to (round-robin)
  int wait_items;                // items of layer wait_layers - 1 (its counter's target)
  int halo;                      // 3x3 stride-1 with 64-channel k-blocks: A from halo tiles
  int tall;                      // halo layers: tiles two MMA row blocks high (see ConvLayer)
  int tw, th;                    // tile width and height (one MMA row block) in pixels
  int tr;                        // tile x along the image's H (see ConvLayer)
  void* out;                     // output [agent][out_h][ow][ldc], channels from choff
  long long out_astride;         // elements between agents in `out`
  int ow, ldc, gw, gh;           // output row length, pixel stride, tile grid extent
  int ipa;                       // items per agent (m_tiles * n_tiles * splits)
  int deconv_idx;                // deconvs: index into BackboneParams::mapC
};
struct BackboneParams {
  LayerDesc L[kMaxLayers];
  CUtensorMap mapC[kMaxDeconv][RTCC_MAX_AGENTS];   // deconv output store maps per agent
  int n_layers;
  int n_batch;                   // agents this launch runs
  int agents[RTCC_MAX_AGENTS];   // their indices, ascending (the agent coordinate of the maps)
  unsigned* grid_bar;            // [kMaxLayers + 1] per-layer counts of finished items, then
                                 // the CTA exit count; zero before a launch (the last CTA to
                                 // leave zeroes them again)
  int* err;
  unsigned long long* stamps;    // optional [2 * n_layers] global-timer ns: layer starts
                                 // (first item's wait passed), then layer ends (last item counted)
  volatile int* done_word;       // optional (pinned host): the last CTA to leave writes 1
  const volatile int* stall;     // optional test hook: when *stall != 0 the first layer that
                                 // waits for another waits for one item too many (the wait
                                 // runs out, the error word is set, the kernel winds down)
  long long wait_budget;         // cycles after which a wait gives up
  int cluster;                   // 1, or kMaxSplits when some layer reduces through DSMEM
  int grid;                      // CTAs of the launch
};

// Fill the kernel parameters of a backbone launch over `n_batch` agents from
// the layer list (whose bn fields are the N tiles for that batch size);
// grid_bar holds kMaxLayers + 1 counters.  The agent list is set by the
// caller (agents[0 .. n_batch)).
cudaError_t backbone_fill(const std::vector<ConvLayer>& layers, int n_batch, unsigned* grid_bar,
                          int* err, unsigned long long* stamps, bool allow_clusters,
                          long long wait_budget, BackboneParams* P);
// One cooperative launch (one CTA per SM) running every layer.
cudaError_t launch_backbone(const BackboneParams& P, bool bf16, cudaStream_t st);
// CTAs of a backbone launch: every SM (cluster = 1), or as many CTAs as can be
// co-resident in clusters of `cluster` CTAs; 0 on error.
int backbone_grid(int cluster);

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
  uint32_t* keys;            // device [cells][anchors] decode keys (see fuse_head.cu)
  uint32_t* hist0;           // device [4096] histogram of the keys' top 12 bits
  float cls_thresh;
  int anchors;
  unsigned long long* span;  // device [3] kernel span stamps (see span_begin), or null
};
cudaError_t launch_fuse_head(const FuseArgs& a, bool bf16, cudaStream_t st);

// Cross-agent fusion of the backbone blocks' outputs (fuse_blocks.cu): the
// multi-scale placement, where each block's map is fused before the neck.
struct FuseBlocksArgs {
  const void* src[RTCC_MAX_BLOCKS];     // block b's outputs, agent-major [K][cells][C_b]
  long long astride[RTCC_MAX_BLOCKS];   // elements between agents
  void* dst[RTCC_MAX_BLOCKS];           // fused map of block b [cells][C_b]
  int cells[RTCC_MAX_BLOCKS];           // cells of block b's grid
  int ch[RTCC_MAX_BLOCKS];              // C_b: 32, 64, 128 or 256
  int tasks[RTCC_MAX_BLOCKS];           // set by the launcher (warp tasks per block)
  float inv_sqrt_c[RTCC_MAX_BLOCKS];    // set by the launcher
  int n;                                // blocks
  const int* present;                   // device [K] presence flags
  int K;
  int attention;                        // 0 = max, 1 = ego-query attention
  unsigned long long* span;             // device [3] kernel span stamps, or null
};
cudaError_t launch_fuse_blocks(FuseBlocksArgs a, bool bf16, cudaStream_t st);

// Max fusion + head on the tensor cores (fuse_tc.cu).
constexpr int kFuseHeadOut = 16;
struct FuseTcParams {
  CUtensorMap feat[RTCC_MAX_AGENTS];  // agent k's slot [cells][C], box (bkc, 128), swizzled
  CUtensorMap feat_all;               // the K slots as one [K][cells][C] tensor, box (bkc, 128, K)
  CUtensorMap wmap;                   // head weights [16][C] in the storage type, box (bkc, 16)
  const int* present;                 // device [K]
  int K, C, cells, bkc, stages;
  const float* head_b;                // device [16]
  float* head_out;                    // device [cells][16]
  void* fused;                        // device [cells][C] or null
  uint32_t* keys;                     // device [cells][anchors] decode keys
  uint32_t* hist0;                    // device [4096] top-12-bit key histogram
  float cls_thresh;
  int anchors;
  int* err;                           // device error word
  unsigned long long* span;           // device [3] kernel span stamps, or null
};
// Channel chunk (64 or 32) the kernel stages for C channels and K agent slots,
// 0 if it cannot run that shape.
int fuse_tc_chunk(int C, int K);
int fuse_tc_stages(int C, int K);   // pipeline stages for that chunk
cudaError_t launch_fuse_max_head(const FuseTcParams& p, bool bf16, cudaStream_t st);

// Row-major 2-D 16-bit tensor map [outer][inner] with a box of
// box_inner x box_outer elements and the given swizzle span (128, 64 or 0
// bytes); OOB elements read as zero.
cudaError_t tmap_2d(CUtensorMap* m, const void* base, bool bf16, uint64_t inner, uint64_t outer,
                    uint32_t box_inner, uint32_t box_outer, int swizzle_bytes);
// The same for a 3-D tensor [outer][mid][inner], dense.
cudaError_t tmap_3d(CUtensorMap* m, const void* base, bool bf16, uint64_t inner, uint64_t mid,
                    uint64_t outer, uint32_t box_inner, uint32_t box_mid, uint32_t box_outer,
                    int swizzle_bytes);
// Head weight permutation expected by the fusion kernel (host side).
void permute_head_weights(const float* w /*[16][C]*/, int C, float* out /*[16*C]*/);

struct DecodeArgs {
  const float* head;         // [cells][16]
  const uint32_t* keys;      // [cells][anchors] from the fusion kernel, padded with
                             // 0xFFFFFFFF to decode_key_capacity() entries
  uint32_t* hist0;           // [4096] top-12-bit histogram of the valid keys; the
                             // decode clears it after reading
  int feat_w, feat_h, anchors;
  float x_min, y_min, x_max, y_max;
  int max_boxes;
  const int* err;            // device error word, copied into the result header
  void* out;                 // result block DetResultHeader + rtcc_box[max_boxes], in
                             // pinned host memory (written directly by the kernel)
  int* present;              // device [K] per-agent presence flags: cleared for the next frame
  int K;
  volatile int* done;        // pinned host word: set to 1 once `out` is complete
  rtcc_box* dev_boxes;       // non-null when NMS follows: the boxes and their count go
  int* dev_n;                // to these device buffers instead, and neither `out` nor
                             // `done` is written
};
constexpr int kDecodeKeep = 512;     // largest supported max_boxes
constexpr int kDecodeHistBins = 4096;
int decode_key_chunk4(int n_anchors);
inline size_t decode_key_capacity(int n_anchors) {
  return (size_t)decode_key_chunk4(n_anchors) * 4 * 1024;
}
cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t st);

// Result block the decode (or NMS) kernel writes into pinned host memory.
struct DetResultHeader {
  int n_boxes;
  int err;
  int pad[2];
};

// Rotated BEV NMS of the decoded boxes (see nms.cu).
struct NmsArgs {
  const rtcc_box* in;        // device [max_boxes] decoded boxes in rank order
  const int* n_in;           // device: their count
  uint32_t* mask;            // device scratch, nms_mask_words(max_boxes) words
  unsigned* ticket;          // device counter, 0 between launches
  int max_boxes;
  float iou;                 // suppress when IoU > iou, 0 <= iou <= 1
  const int* err;            // device error word, copied into the result header
  void* out;                 // pinned host result block DetResultHeader + rtcc_box[max_boxes]
  volatile int* done;        // pinned host word: set to 1 once `out` is complete
};
size_t nms_mask_words(int max_boxes);
cudaError_t launch_nms(const NmsArgs& a, cudaStream_t st);

}  // namespace rtcc

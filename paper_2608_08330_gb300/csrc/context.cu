// RTCC runtime context: the offline stage (weights, buffers, per-branch CUDA
// graphs; Sec. IV-A) and the online release path (Sec. IV-C..F):
//
//   completion event e_k --validate--> RELEASED --(pinned H2D on the transfer
//   stream, cudaEvent)--> branch graph on the branch's compute stream, writing
//   the agent-indexed slot k --(cudaEvent)--> post-join graph once every
//   branch is resolved (fusion + head + decode + D2H of the detections).
//
// Barrier mode holds every release until the last branch resolves and then
// dispatches all present branches in index order (Sec. V).  Both modes launch
// the same graphs on the same inputs, so outputs are bit-identical.
#include <algorithm>
#include <atomic>
#include <chrono>
#include <cmath>
#include <condition_variable>
#include <cstring>
#include <mutex>
#include <new>
#include <thread>
#include <vector>

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "controller.h"
#include "kernels.h"
#include "rtcc.h"

using namespace rtcc;

namespace {

double now_ms() {
  using clk = std::chrono::steady_clock;
  return std::chrono::duration<double, std::milli>(clk::now().time_since_epoch()).count();
}

constexpr size_t kHdrBytes = 16;   // payload header: int32 n, padding to 16 bytes

struct Branch {
  float* staging = nullptr;        // pinned [kHdrBytes][cap][4]
  uint8_t* in_dev = nullptr;       // device [kHdrBytes][cap][4]
  PillarBufs pb{};
  void* feat = nullptr;            // agent-indexed feature slot [H'][W'][C_feat] (a view
                                   // into the context's feature slots)
  float* splitk_ws = nullptr;      // split-K partials of this branch's own launches
  int* splitk_cnt = nullptr;       // split-K per-tile arrival counters
  unsigned* grid_bar = nullptr;      // inside frame_zero: per-layer counters + exit count
  void* frame_zero = nullptr;         // [kFrameZeroBytes] cleared by every pass's first pillar kernel
  unsigned long long* stamps = nullptr;   // RTCC_FLAG_LAYER_TIMES: layer starts, then ends
  BackboneParams* bb = nullptr;    // backbone kernel parameters of this agent alone
  cudaStream_t st = nullptr;
  cudaGraphExec_t exec = nullptr;       // pillar chain + backbone, payload in the device slot
  cudaGraphExec_t exec_host = nullptr;  // the same, payload in the pinned staging buffer (zero-copy)
  cudaGraphExec_t pill = nullptr;       // pillar chain alone (the backbone runs in a batch)
  cudaGraphExec_t pill_host = nullptr;
  cudaEvent_t h2d_done = nullptr, done = nullptr, pill_done = nullptr;
  cudaEvent_t ev_start = nullptr, ev_bb0 = nullptr, ev_bb1 = nullptr, ev_end = nullptr;
  cudaEvent_t feat_ev = nullptr;   // this frame: the event after which the slot is written
  int stamp_src = -1;              // this frame: whose stamps buffer its launch wrote
  int launch_idx = -1;             // this frame: index of the backbone launch that ran it
  bool full_graph = false;         // this frame: ran as its own branch graph (event nodes)
  const float* pend_ptr = nullptr;
  int pend_n = 0;
  bool pend_resident = false;
  bool launched = false;
  bool resident_ok = false;
};

}  // namespace

struct rtcc_ctx {
  rtcc_model_config cfg{};
  bool bf16 = false;
  int K = 0, W = 0, H = 0, Cp = 0, P = 0, N = 0, cap = 0;
  int Wf = 0, Hf = 0, Cf = 0, n_conv = 0, n_deconv = 0;
  Controller ctrl;
  std::mutex mu;
  // weights
  float* pfn_w = nullptr;
  float* pfn_b = nullptr;
  std::vector<void*> wbufs;           // packed conv/deconv weights
  std::vector<float*> bbufs;          // conv/deconv biases
  float* head_wp = nullptr;
  float* head_b = nullptr;
  void* head_w16 = nullptr;   // head weights [16][C] in the storage type (tensor-core head)
  Branch br[RTCC_MAX_AGENTS];
  void* image_all = nullptr;          // pseudo-images [K][H][W][C_p]
  // Backbone tensors of all agents, agent-major with a fixed stride (one
  // tensor map covers every agent; a launch runs any subset)
  void* feat_all = nullptr;           // [K][H'][W'][C_feat]
  void* block_all[RTCC_MAX_BLOCKS][2] = {};   // ping-pong activations [K][H_b][W_b][C_b]
  std::vector<void*> layer_all;       // RTCC_FLAG_KEEP_LAYERS: every conv's output [K][...]
  std::vector<size_t> layer_elems;    // elements per agent
  void* block_out[RTCC_MAX_BLOCKS] = {};
  int block_w[RTCC_MAX_BLOCKS] = {}, block_h[RTCC_MAX_BLOCKS] = {};
  // RTCC_FLAG_MULTISCALE: the branches end at their blocks; the post-join
  // fuses each block's map across the agents, then runs the neck once
  bool ms = false;
  void* fblk[RTCC_MAX_BLOCKS] = {};   // fused block maps [H_b][W_b][C_b]
  void* neck_out = nullptr;           // neck of the fused blocks [H'][W'][C_feat]
  std::vector<ConvLayer> neck_layers; // its deconvs (one "agent")
  BackboneParams* neck_p = nullptr;
  unsigned* neck_bar = nullptr;       // [kMaxLayers + 1], zero between launches
  int* d_one = nullptr;               // [RTCC_MAX_AGENTS] = {1, 0, ...}: the head's one input
  int post_kernels = 0;               // kernels of the post-join graph
  size_t img_elems = 0, feat_elems = 0;
  std::vector<ConvLayer> layers;      // the layer list (N tiles of a one-agent launch)
  BackboneParams* bbt[RTCC_MAX_AGENTS + 1] = {};  // launch parameters per batch size
  long long wait_budget = 0;
  // batched backbone launches (agents released together)
  cudaStream_t bbst = nullptr;
  float* batch_ws = nullptr;
  int* batch_cnt = nullptr;
  unsigned* batch_bar = nullptr;      // [kMaxLayers + 1], zero between launches
  cudaEvent_t batch_ev[RTCC_MAX_AGENTS] = {}, batch_t0[RTCC_MAX_AGENTS] = {},
              batch_t1[RTCC_MAX_AGENTS] = {};
  BackboneParams* launch_p = nullptr; // scratch for one launch's parameters
  volatile int* done_words = nullptr; // pinned [2 * RTCC_MAX_AGENTS]: written 1 by the last
                                      // CTA of branch k's own backbone launch (k) or of
                                      // batched launch j (RTCC_MAX_AGENTS + j)
  int inflight = -1;                  // done word of the last backbone launched, -1 none
  int n_launches = 0;                 // backbone launches this frame
  int launch_size[RTCC_MAX_AGENTS] = {};
  int launch_word[RTCC_MAX_AGENTS] = {};
  std::vector<int> pending;           // released agents whose backbone waits for a batch
  std::atomic<double> t_hold{0.0};    // host time of the last release that left a batch open
  std::thread disp;                   // dispatcher of deferred batches
  std::condition_variable cv;
  bool stop = false;
  int dev = 0;
  volatile int* stall = nullptr;      // pinned test hook word (RTCC_FLAG_SHORT_WAITS)
  bool disp_err = false;              // the dispatcher failed to launch a batch
  size_t splitk_cnt_bytes = 0;        // split-K tile counters of one branch (batch: K x)
  cudaStream_t xfer = nullptr, post = nullptr;
  cudaGraphExec_t post_exec = nullptr;
  int* d_present = nullptr;           // [K] set by a branch's first kernel, cleared by the decode
  void** d_feat_ptrs = nullptr;
  float* head_out = nullptr;
  void* fused = nullptr;
  uint32_t* keys = nullptr;           // decode key per anchor (padded)
  uint32_t* hist0 = nullptr;          // decode level-0 histogram
  rtcc_box* dec_boxes = nullptr;      // NMS on: the decode's boxes (device), NMS input
  int* dec_n = nullptr;               //         and their count
  uint32_t* nms_mask = nullptr;       //         suppression bitmask scratch
  unsigned* nms_ticket = nullptr;     //         last-block counter
  unsigned long long* fuse_span = nullptr;   // RTCC_FLAG_TIMELINE: fusion kernel span stamps [3]
  uint8_t* det_host = nullptr;        // pinned; the decode (or NMS) kernel writes it directly
  size_t det_bytes = 0;
  volatile int* h_done = nullptr;     // pinned; the decode kernel sets it to 1 when det_host is complete
  bool present_dirty = false;         // a branch set its presence flag and no post-join cleared it
  int* d_err = nullptr;
  cudaEvent_t det_ready = nullptr;
  cudaEvent_t ev_post0 = nullptr, ev_fuse0 = nullptr, ev_fuse1 = nullptr, ev_post1 = nullptr;
  // frame bookkeeping
  bool post_launched = false;
  bool closed_pending = false;
  double t_last_event = 0.0;
  rtcc_frame_info info{};
  std::vector<void*> allocs;          // device allocations
  std::vector<void*> host_allocs;     // pinned allocations

  rtcc_ctx(int k, int cap_pts, bool ego) : ctrl(k, cap_pts, ego) {}
};

namespace {

#define CK(x)                                   \
  do {                                          \
    cudaError_t e_ = (x);                       \
    if (e_ != cudaSuccess) return RTCC_E_CUDA;  \
  } while (0)

template <typename T>
rtcc_status dalloc(rtcc_ctx* c, T** p, size_t bytes) {
  void* v = nullptr;
  if (cudaMalloc(&v, bytes ? bytes : 16) != cudaSuccess) return RTCC_E_NOMEM;
  c->allocs.push_back(v);
  *p = static_cast<T*>(v);
  return RTCC_OK;
}

template <typename T>
rtcc_status halloc(rtcc_ctx* c, T** p, size_t bytes) {
  void* v = nullptr;
  if (cudaHostAlloc(&v, bytes ? bytes : 16, cudaHostAllocDefault) != cudaSuccess)
    return RTCC_E_NOMEM;
  c->host_allocs.push_back(v);
  *p = static_cast<T*>(v);
  return RTCC_OK;
}

#define RS(x)                          \
  do {                                 \
    rtcc_status s_ = (x);              \
    if (s_ != RTCC_OK) return s_;      \
  } while (0)

// Round to the storage type and back (float value exactly representable).
float round_store(float v, bool bf16) {
  return bf16 ? __bfloat162float(__float2bfloat16_rn(v)) : __half2float(__float2half_rn(v));
}
uint16_t bits_store(float v, bool bf16) {
  if (bf16) {
    __nv_bfloat16 h = __float2bfloat16_rn(v);
    uint16_t u;
    std::memcpy(&u, &h, 2);
    return u;
  }
  __half h = __float2half_rn(v);
  uint16_t u;
  std::memcpy(&u, &h, 2);
  return u;
}

bool pow2_in(int v, std::initializer_list<int> allowed) {
  for (int a : allowed)
    if (v == a) return true;
  return false;
}

rtcc_status validate_config(const rtcc_model_config& c) {
  if (c.n_agents < 1 || c.n_agents > RTCC_MAX_AGENTS) return RTCC_E_ARG;
  if (c.grid_w < 1 || c.grid_h < 1 || c.grid_w > 4096 || c.grid_h > 4096) return RTCC_E_ARG;
  if (!(c.pillar > 0.f) || !(c.x_max > c.x_min) || !(c.y_max > c.y_min) || !(c.z_max > c.z_min))
    return RTCC_E_ARG;
  if (!grid_coords_ok(c.x_min, c.y_min, c.z_min, c.z_max, c.pillar, c.grid_w, c.grid_h))
    return RTCC_E_ARG;
  if (c.max_pillars < 1 || c.max_pts < 1 || c.max_pts > 32) return RTCC_E_ARG;
  if (!pow2_in(c.pfn_ch, {32, 64})) return RTCC_E_ARG;
  if (c.n_blocks < 1 || c.n_blocks > RTCC_MAX_BLOCKS) return RTCC_E_ARG;
  if (c.anchors != 2 || c.max_boxes < 1 || c.max_boxes > 512) return RTCC_E_ARG;
  if (!(c.nms_iou >= 0.f && c.nms_iou <= 1.f)) return RTCC_E_ARG;
  if (c.max_points < 0 || c.max_points > (1 << 24)) return RTCC_E_ARG;
  if (c.fusion != RTCC_FUSE_MAX && c.fusion != RTCC_FUSE_ATTN) return RTCC_E_ARG;
  if (c.dtype != RTCC_FP16 && c.dtype != RTCC_BF16) return RTCC_E_ARG;
  int w = c.grid_w, h = c.grid_h;
  bool neck = c.up_stride[0] != 0;
  for (int b = 0; b < c.n_blocks; ++b) {
    if (c.block_layers[b] < 1 || c.block_layers[b] > 16) return RTCC_E_ARG;
    if (!pow2_in(c.block_ch[b], {32, 64, 128, 256})) return RTCC_E_ARG;
    if (c.block_stride[b] != 1 && c.block_stride[b] != 2) return RTCC_E_ARG;
    if (c.block_stride[b] == 2) {
      if ((w & 1) || (h & 1)) return RTCC_E_ARG;
      w /= 2;
      h /= 2;
    }
    if ((c.up_stride[b] != 0) != neck) return RTCC_E_ARG;
  }
  if (!neck && c.n_blocks != 1) return RTCC_E_ARG;
  if ((c.flags & RTCC_FLAG_MULTISCALE) && !neck) return RTCC_E_ARG;
  if (neck) {
    if (c.up_ch != 128) return RTCC_E_ARG;
    // every deconv output must land on block 0's grid
    int w0 = c.grid_w / c.block_stride[0], h0 = c.grid_h / c.block_stride[0];
    int wb = c.grid_w, hb = c.grid_h;
    for (int b = 0; b < c.n_blocks; ++b) {
      wb /= c.block_stride[b];
      hb /= c.block_stride[b];
      if (!pow2_in(c.up_stride[b], {1, 2, 4})) return RTCC_E_ARG;
      if (wb * c.up_stride[b] != w0 || hb * c.up_stride[b] != h0) return RTCC_E_ARG;
    }
  }
  return RTCC_OK;
}

size_t expected_floats(const rtcc_model_config& c, int cf) {
  size_t n = (size_t)c.pfn_ch * 9 + c.pfn_ch;
  int cin = c.pfn_ch;
  for (int b = 0; b < c.n_blocks; ++b)
    for (int l = 0; l < c.block_layers[b]; ++l) {
      n += (size_t)c.block_ch[b] * cin * 9 + c.block_ch[b];
      cin = c.block_ch[b];
    }
  if (c.up_stride[0])
    for (int b = 0; b < c.n_blocks; ++b)
      n += (size_t)c.block_ch[b] * c.up_ch * c.up_stride[b] * c.up_stride[b] + c.up_ch;
  n += (size_t)16 * cf + 16;
  return n;
}

rtcc_status upload_f32(rtcc_ctx* c, const float* src, size_t n, float** dst) {
  RS(dalloc(c, dst, n * sizeof(float)));
  std::vector<float> v(src, src + n);
  for (auto& x : v) x = round_store(x, c->bf16);
  CK(cudaMemcpy(*dst, v.data(), n * sizeof(float), cudaMemcpyHostToDevice));
  return RTCC_OK;
}

// W [Co][Ci][3][3] -> [Co][tap][Ci] in the storage type
// W [Co][Ci][3][3] -> tap-major [tap][Co][Ci] (one TMA box carries several taps)
rtcc_status upload_conv(rtcc_ctx* c, const float* w, int co, int ci) {
  std::vector<uint16_t> p((size_t)co * 9 * ci);
  for (int o = 0; o < co; ++o)
    for (int i = 0; i < ci; ++i)
      for (int t = 0; t < 9; ++t)
        p[((size_t)t * co + o) * ci + i] = bits_store(w[((size_t)o * ci + i) * 9 + t], c->bf16);
  void* d = nullptr;
  RS(dalloc(c, &d, p.size() * 2));
  CK(cudaMemcpy(d, p.data(), p.size() * 2, cudaMemcpyHostToDevice));
  c->wbufs.push_back(d);
  return RTCC_OK;
}

// W [Ci][Co][s][s] -> [(sy*s+sx)*Co + co][Ci]
rtcc_status upload_deconv(rtcc_ctx* c, const float* w, int ci, int co, int s) {
  std::vector<uint16_t> p((size_t)s * s * co * ci);
  for (int i = 0; i < ci; ++i)
    for (int o = 0; o < co; ++o)
      for (int sy = 0; sy < s; ++sy)
        for (int sx = 0; sx < s; ++sx)
          p[((size_t)(sy * s + sx) * co + o) * ci + i] =
              bits_store(w[(((size_t)i * co + o) * s + sy) * s + sx], c->bf16);
  void* d = nullptr;
  RS(dalloc(c, &d, p.size() * 2));
  CK(cudaMemcpy(d, p.data(), p.size() * 2, cudaMemcpyHostToDevice));
  c->wbufs.push_back(d);
  return RTCC_OK;
}

rtcc_status upload_weights(rtcc_ctx* c, const float* w) {
  const rtcc_model_config& g = c->cfg;
  size_t o = 0;
  RS(upload_f32(c, w + o, (size_t)g.pfn_ch * 9, &c->pfn_w));
  o += (size_t)g.pfn_ch * 9;
  RS(upload_f32(c, w + o, g.pfn_ch, &c->pfn_b));
  o += g.pfn_ch;
  int cin = g.pfn_ch;
  for (int b = 0; b < g.n_blocks; ++b)
    for (int l = 0; l < g.block_layers[b]; ++l) {
      const int co = g.block_ch[b];
      RS(upload_conv(c, w + o, co, cin));
      o += (size_t)co * cin * 9;
      float* bias = nullptr;
      RS(upload_f32(c, w + o, co, &bias));
      c->bbufs.push_back(bias);
      o += co;
      cin = co;
    }
  if (g.up_stride[0])
    for (int b = 0; b < g.n_blocks; ++b) {
      const int s = g.up_stride[b], ci = g.block_ch[b], co = g.up_ch;
      RS(upload_deconv(c, w + o, ci, co, s));
      o += (size_t)ci * co * s * s;
      float* bias = nullptr;
      RS(upload_f32(c, w + o, co, &bias));
      c->bbufs.push_back(bias);
      o += co;
    }
  std::vector<float> hw(w + o, w + o + (size_t)16 * c->Cf);
  for (auto& x : hw) x = round_store(x, c->bf16);
  std::vector<float> hp((size_t)16 * c->Cf);
  permute_head_weights(hw.data(), c->Cf, hp.data());
  RS(dalloc(c, &c->head_wp, hp.size() * sizeof(float)));
  CK(cudaMemcpy(c->head_wp, hp.data(), hp.size() * sizeof(float), cudaMemcpyHostToDevice));
  std::vector<uint16_t> h16(hw.size());
  for (size_t i = 0; i < hw.size(); ++i) h16[i] = bits_store(hw[i], c->bf16);
  RS(dalloc(c, &c->head_w16, h16.size() * sizeof(uint16_t)));
  CK(cudaMemcpy(c->head_w16, h16.data(), h16.size() * sizeof(uint16_t), cudaMemcpyHostToDevice));
  o += (size_t)16 * c->Cf;
  RS(upload_f32(c, w + o, 16, &c->head_b));
  return RTCC_OK;
}

// N tile and split-K factor of a conv layer, from a cost model of the
// persistent backbone kernel: one tcgen05 MMA instruction costs about the same
// for every N <= 128, so a k-block costs the same for every N tile; a CTA
// holds one item at a time, so items beyond the grid take another round; a
// split of a 64-wide tile into kMaxSplits slices (one item per CTA) is reduced
// through distributed shared memory at about the cost of 7 k-blocks.  Measured
// on the 64x64x128 block, a 2-way split (9 k-blocks per slice) was slower than
// 32-wide tiles without split (18 k-blocks), so only 4-way splits are used.
// Ties go to the narrower tile (more CTAs).
void pick_tile(int m_tiles, int co, int total_kb, int grid, int* bn_out, int* sp_out) {
  double best = 1e30;
  int bb = std::min(co, 64), bs = 1;
  for (int bn : {32, 64, 128}) {
    if (bn > co || co % bn) continue;
    for (int sp : {1, kMaxSplits}) {
      const int items = m_tiles * (co / bn) * sp;
      if (sp > 1 && (bn != 64 || total_kb / sp < 4 || items > grid)) continue;
      const int rounds = (items + grid - 1) / grid;
      const double cost = rounds * (double)((total_kb + sp - 1) / sp) + (sp > 1 ? 7.0 : 0.0);
      if (cost < best - 1e-9) {
        best = cost;
        bb = bn;
        bs = sp;
      }
    }
  }
  *bn_out = bb;
  *sp_out = bs;
}

constexpr size_t kFrameZeroBytes = 8 * sizeof(int) + (kMaxLayers + 1) * sizeof(unsigned);

// Tile of a conv layer in a launch over `batch` agents, with its K slices
// fixed (they decide the fp32 summation order, so they are the same for every
// batch size and a branch's result does not depend on the launch that ran
// it; the N tile only decides which channels an item computes, and the tile
// shape which pixels).  Cost model: rounds of items over the grid times
// k-blocks per item times a k-block's MMA time at that N tile (measured:
// 45, 48 and 64 clocks per K = 16 MMA at N = 32, 64, 128); a tall tile
// (halo layers without split-K: two 128-row MMAs on every weight box) costs
// kTallCost short k-blocks per k-block -- more than one because it does
// twice the MMAs, less than two because it halves the weight boxes per FLOP,
// which bound a short k-block once every CTA has several items.  The tile
// may also be laid the other way round (a halo layer's tiles transposed, a
// tap-box layer's 16 x 8 instead of 8 x 16): the same work per item, but a
// different item count where the image's sides are not multiples of the
// tile's (352 x 100 in 8 x 16 tiles: 308 items, 3 rounds on 152 CTAs;
// transposed, 286).  Ties go to the short, then the narrower tile, then the
// first orientation.
constexpr double kTallCost = 1.6;
double kblock_cost(int bn) { return bn >= 128 ? 1.0 : bn >= 64 ? 0.75 : 0.70; }
void pick_tile_batch(const ConvLayer L0, int sp, int grid, int batch, bool need64, ConvLayer* out) {
  double best = 1e30;
  out->bn = std::min(L0.cout, 64);
  out->tall = out->tr = out->wide = 0;
  const int total_kb = 9 * (L0.cin / L0.bk);
  for (int tall = 0; tall <= 1; ++tall) {
    for (int bn : {32, 64, 128}) {
      if (bn > L0.cout || L0.cout % bn) continue;
      if (need64 && bn != 64) continue;
      for (int orient = 0; orient <= 1; ++orient) {
        ConvLayer L = L0;
        L.splits = sp;
        L.tall = tall;
        const bool halo = conv_uses_halo(L);
        L.tr = orient && halo;
        L.wide = orient && !halo;
        if (!conv_shape_ok(L)) continue;
        const int items = batch * conv_m_tiles(L) * (L.cout / bn) * sp;
        const int rounds = (items + grid - 1) / grid;
        const double cost =
            rounds * (double)((total_kb + sp - 1) / sp) * kblock_cost(bn) * (tall ? kTallCost : 1.0);
        if (cost < best - 1e-9) {
          best = cost;
          out->bn = bn;
          out->tall = L.tall;
          out->tr = L.tr;
          out->wide = L.wide;
        }
      }
    }
  }
}

// The K slices of conv layer L (its split-K factor, with its K chunk and a
// first N tile) from the one-agent model; they stay the same for every batch
// size.  L's kind, channels and output extent (gw x gh) must be set.
void choose_split(ConvLayer& L, int grid) {
  const int m_tiles = ((L.gw + conv_tile_w() - 1) / conv_tile_w()) * ((L.gh + conv_tile_h() - 1) / conv_tile_h());
  L.bk = (L.cin >= 64) ? 64 : 32;
  pick_tile(m_tiles, L.cout, 9 * (L.cin / L.bk), grid, &L.bn, &L.splits);
  L.n_tiles_n = L.cout / L.bn;
}

// The N tile and tile shape of conv layer L (K slices already chosen) in a
// launch over nb agents.  A split layer whose items fit the clustered grid
// keeps the DSMEM exchange (64-wide tiles); otherwise it reduces through
// global memory.
void choose_tiles(ConvLayer& L, int grid, int nb) {
  const int m_tiles = conv_m_tiles(L);
  const bool dsm_fit = L.splits > 1 && nb * m_tiles * (L.cout / 64) * L.splits <= grid;
  pick_tile_batch(L, L.splits, grid, nb, dsm_fit, &L);
  L.n_tiles_n = L.cout / L.bn;
}

// The backbone's layer list over the agent-major tensors of all K agents, and
// the launch parameters for every batch size.
rtcc_status build_backbone(rtcc_ctx* c) {
  const rtcc_model_config& g = c->cfg;
  const int K = c->K;
  // the tile choice uses the clustered grid with or without clusters, so the
  // K slices (and the results) do not depend on RTCC_FLAG_NO_CLUSTERS
  int grid = backbone_grid(kMaxSplits);
  if (grid < 1) grid = backbone_grid(1);
  if (grid < 1) return RTCC_E_CUDA;
  const size_t es = 2;   // 16-bit storage
  c->img_elems = (size_t)c->W * c->H * c->Cp;
  c->feat_elems = (size_t)c->Wf * c->Hf * c->Cf;
  RS(dalloc(c, &c->feat_all, (size_t)K * c->feat_elems * es));
  CK(cudaMemset(c->feat_all, 0, (size_t)K * c->feat_elems * es));
  const bool neck = g.up_stride[0] != 0;
  const bool keep = (g.flags & RTCC_FLAG_KEEP_LAYERS) != 0;
  int block_last[RTCC_MAX_BLOCKS] = {};
  const void* in = c->image_all;                  // the agents' pseudo-images, agent-major
  long long in_as = (long long)c->img_elems;
  int cin = c->Cp, w = c->W, h = c->H;
  int wi = 0;
  for (int bi = 0; bi < g.n_blocks; ++bi) {
    const int st = g.block_stride[bi];
    const int ow = w / st, oh = h / st;
    const int co = g.block_ch[bi];
    const size_t per = (size_t)ow * oh * co;
    if (!keep) {
      RS(dalloc(c, &c->block_all[bi][0], (size_t)K * per * es));
      RS(dalloc(c, &c->block_all[bi][1], (size_t)K * per * es));
    }
    for (int li = 0; li < g.block_layers[bi]; ++li) {
      ConvLayer L{};
      L.kind = (li == 0 && st == 2) ? CONV3_S2 : CONV3_S1;
      L.n_agents = K;
      L.cin = cin;
      L.cout = co;
      L.s = 1;
      L.in_w = (li == 0) ? w : ow;
      L.in_h = (li == 0) ? h : oh;
      L.out_w = ow;
      L.out_h = oh;
      L.gw = ow;
      L.gh = oh;
      L.ldc = co;
      L.choff = 0;
      choose_split(L, grid);
      L.in = in;
      L.in_astride = in_as;
      const bool last = (bi == g.n_blocks - 1) && (li == g.block_layers[bi] - 1);
      void* dst = nullptr;
      long long out_as = (long long)per;
      if (!neck && last) {
        dst = c->feat_all;
        out_as = (long long)c->feat_elems;
      } else if (keep) {
        RS(dalloc(c, &dst, (size_t)K * per * es));
      } else {
        dst = c->block_all[bi][li & 1];
      }
      L.out = dst;
      L.out_astride = out_as;
      c->layer_all.push_back(dst);
      c->layer_elems.push_back(per);
      L.wpacked = c->wbufs[wi];
      L.bias = c->bbufs[wi];
      L.wait_layers = (int)c->layers.size();          // reads the previous conv's output
      ++wi;
      c->layers.push_back(L);
      in = L.out;
      in_as = out_as;
      cin = co;
    }
    c->block_out[bi] = const_cast<void*>(in);
    block_last[bi] = (int)c->layers.size();          // layers [0, block_last) done
    c->block_w[bi] = ow;
    c->block_h[bi] = oh;
    w = ow;
    h = oh;
  }
  c->ms = (g.flags & RTCC_FLAG_MULTISCALE) != 0;
  if (neck && c->ms) {
    // the neck runs after the join, once, on the fused block maps
    for (int bi = 0; bi < g.n_blocks; ++bi)
      RS(dalloc(c, &c->fblk[bi], (size_t)c->block_w[bi] * c->block_h[bi] * g.block_ch[bi] * es));
    RS(dalloc(c, &c->neck_out, c->feat_elems * es));
    CK(cudaMemset(c->neck_out, 0, c->feat_elems * es));
    for (int bi = 0; bi < g.n_blocks; ++bi) {
      ConvLayer L{};
      L.kind = DECONV;
      L.n_agents = 1;
      L.s = g.up_stride[bi];
      L.cin = g.block_ch[bi];
      L.cout = g.up_ch;
      L.in_w = c->block_w[bi];
      L.in_h = c->block_h[bi];
      L.out_w = c->Wf;
      L.out_h = c->Hf;
      L.gw = L.in_w;
      L.gh = L.in_h;
      L.ldc = c->Cf;
      L.choff = bi * g.up_ch;
      L.bn = g.up_ch;
      L.bk = (L.cin >= 64) ? 64 : 32;
      L.n_tiles_n = L.s * L.s;
      L.splits = 1;
      L.in = c->fblk[bi];
      L.in_astride = (long long)c->block_w[bi] * c->block_h[bi] * g.block_ch[bi];
      L.out = c->neck_out;
      L.out_astride = (long long)c->feat_elems;
      L.wpacked = c->wbufs[wi];
      L.bias = c->bbufs[wi];
      L.wait_layers = 0;                              // the fused maps precede the launch
      ++wi;
      if (conv_make_maps(L, c->bf16) != cudaSuccess) return RTCC_E_CUDA;
      c->neck_layers.push_back(L);
    }
  } else if (neck) {
    for (int bi = 0; bi < g.n_blocks; ++bi) {
      ConvLayer L{};
      L.kind = DECONV;
      L.n_agents = K;
      L.s = g.up_stride[bi];
      L.cin = g.block_ch[bi];
      L.cout = g.up_ch;
      L.in_w = c->block_w[bi];
      L.in_h = c->block_h[bi];
      L.out_w = c->Wf;
      L.out_h = c->Hf;
      L.gw = L.in_w;
      L.gh = L.in_h;
      L.ldc = c->Cf;
      L.choff = bi * g.up_ch;
      L.bn = g.up_ch;
      L.bk = (L.cin >= 64) ? 64 : 32;
      L.n_tiles_n = L.s * L.s;
      L.in = c->block_out[bi];
      L.in_astride = (long long)c->block_w[bi] * c->block_h[bi] * g.block_ch[bi];
      L.out = c->feat_all;
      L.out_astride = (long long)c->feat_elems;
      L.wpacked = c->wbufs[wi];
      L.bias = c->bbufs[wi];
      L.wait_layers = block_last[bi];                 // only its block's output
      ++wi;
      c->layers.push_back(L);
    }
  }
  // fp32 workspace of the global-memory split-K reduction (used when a split
  // layer cannot reduce through DSMEM): one per branch for its own launches,
  // and one for the batched launches; deconvs never split
  size_t ws_floats = 0, max_tiles = 0;
  for (ConvLayer& L : c->layers) {
    const int m_tiles = ((L.gw + conv_tile_w() - 1) / conv_tile_w()) *
                        ((L.gh + conv_tile_h() - 1) / conv_tile_h());
    if (L.kind == DECONV || L.splits < 1) L.splits = 1;
    if (L.splits > 1) {
      // the widest tile any batch size may pick: co / 32 tiles of 32 ... 128 columns
      ws_floats = std::max(ws_floats, (size_t)L.splits * m_tiles * L.cout * conv_tile_m());
      max_tiles = std::max(max_tiles, (size_t)m_tiles * (L.cout / 32));
    }
  }
  c->splitk_cnt_bytes = max_tiles * sizeof(int);
  for (int k = 0; k < K; ++k) {
    Branch& b = c->br[k];
    if (ws_floats) {
      RS(dalloc(c, &b.splitk_ws, ws_floats * sizeof(float)));
      RS(dalloc(c, &b.splitk_cnt, max_tiles * sizeof(int)));
      CK(cudaMemset(b.splitk_cnt, 0, max_tiles * sizeof(int)));
    }
  }
  if (ws_floats) {
    RS(dalloc(c, &c->batch_ws, (size_t)K * ws_floats * sizeof(float)));
    RS(dalloc(c, &c->batch_cnt, (size_t)K * max_tiles * sizeof(int)));
    CK(cudaMemset(c->batch_cnt, 0, (size_t)K * max_tiles * sizeof(int)));
  }
  RS(dalloc(c, &c->batch_bar, (kMaxLayers + 1) * sizeof(unsigned)));
  CK(cudaMemset(c->batch_bar, 0, (kMaxLayers + 1) * sizeof(unsigned)));
  c->wait_budget = (g.flags & RTCC_FLAG_SHORT_WAITS) ? 20000000LL : 2000000000LL;
  // launch parameters per batch size: the same K slices, the N tile and tile
  // height chosen for the batch
  for (int nb = 1; nb <= K; ++nb) {
    std::vector<ConvLayer> Lb = c->layers;
    for (ConvLayer& L : Lb) {
      if (L.kind != DECONV) choose_tiles(L, grid, nb);
      L.ws = c->batch_ws;
      L.counters = c->batch_cnt;
      if (conv_make_maps(L, c->bf16) != cudaSuccess) return RTCC_E_CUDA;
    }
    if (nb == 1) c->layers = Lb;                      // the maps of the one-agent tiles
    c->bbt[nb] = new (std::nothrow) BackboneParams;
    if (!c->bbt[nb]) return RTCC_E_NOMEM;
    if (backbone_fill(Lb, nb, c->batch_bar, c->d_err, nullptr, (g.flags & RTCC_FLAG_NO_CLUSTERS) == 0,
                      c->wait_budget, c->bbt[nb]) != cudaSuccess)
      return RTCC_E_ARG;
  }
  c->launch_p = new (std::nothrow) BackboneParams;
  if (!c->launch_p) return RTCC_E_NOMEM;
  if (c->ms) {
    RS(dalloc(c, &c->neck_bar, (kMaxLayers + 1) * sizeof(unsigned)));
    CK(cudaMemset(c->neck_bar, 0, (kMaxLayers + 1) * sizeof(unsigned)));
    c->neck_p = new (std::nothrow) BackboneParams;
    if (!c->neck_p) return RTCC_E_NOMEM;
    if (backbone_fill(c->neck_layers, 1, c->neck_bar, c->d_err, nullptr, false, c->wait_budget, c->neck_p) !=
        cudaSuccess)
      return RTCC_E_ARG;
  }
  return RTCC_OK;
}

// Per-agent state of branch k: payload slot, pillar scratch, its own launch
// parameters (the one-agent template pointed at this agent and its counters).
rtcc_status build_branch(rtcc_ctx* c, int k) {
  Branch& b = c->br[k];
  const rtcc_model_config& g = c->cfg;
  const int cells = c->W * c->H;
  RS(halloc(c, &b.staging, kHdrBytes + (size_t)c->cap * 16));
  std::memset(b.staging, 0, kHdrBytes);
  RS(dalloc(c, &b.in_dev, kHdrBytes + (size_t)c->cap * 16));
  CK(cudaMemset(b.in_dev, 0, kHdrBytes));
  PillarBufs& p = b.pb;
  p.pts = reinterpret_cast<const float4*>(b.in_dev + kHdrBytes);
  p.n_hdr = reinterpret_cast<const int*>(b.in_dev);
  p.cap = c->cap;
  p.P = c->P;
  p.N = c->N;
  p.C = c->Cp;
  const size_t tiles = (size_t)scan_tiles(c->cap);
  RS(dalloc(c, &p.cell_of, scan_pad(c->cap) * 4));
  RS(dalloc(c, &p.slot_of, scan_pad(c->cap) * 4));
  RS(dalloc(c, &p.cnt_cell, (size_t)cells * 4));
  RS(dalloc(c, &p.first_cell, (size_t)cells * 4));
  RS(dalloc(c, &p.cell_loc, (size_t)cells * sizeof(int2)));
  RS(dalloc(c, &p.tile_agg, tiles * kAggStride * sizeof(unsigned long long)));
  RS(dalloc(c, &p.pillar_rec, (size_t)c->P * sizeof(int4)));
  RS(dalloc(c, &p.touched, (size_t)(c->cap > 0 ? c->cap : 1) * 4));
  RS(dalloc(c, &p.ntouched, 4));
  RS(dalloc(c, &p.list, (size_t)(c->cap > 0 ? c->cap : 1) * 4));
  RS(dalloc(c, &p.bucket, (size_t)c->P * c->N * sizeof(float4)));
  RS(dalloc(c, &p.np_prev, 4));
  CK(cudaMemset(p.np_prev, 0, 4));
  // valid cells and empty pillars from the start (read only after a wait ran out)
  CK(cudaMemset(p.pillar_rec, 0, (size_t)c->P * sizeof(int4)));
  CK(cudaMemset(p.touched, 0, (size_t)(c->cap > 0 ? c->cap : 1) * 4));
  CK(cudaMemset(p.cell_loc, 0x7F, (size_t)cells * sizeof(int2)));
  p.err = c->d_err;
  p.clear_all = 0;                              // image and cell2pillar start cleared below
  p.present_flag = c->d_present + k;
  if (g.flags & RTCC_FLAG_TIMELINE) {
    RS(dalloc(c, &p.pfn_span, 3 * sizeof(unsigned long long)));
    CK(cudaMemset(p.pfn_span, 0, 3 * sizeof(unsigned long long)));
  }
  RS(dalloc(c, &p.pillar_cell, (size_t)c->P * 4));
  CK(cudaMemset(p.pillar_cell, 0, (size_t)c->P * 4));
  RS(dalloc(c, &p.pcount, (size_t)c->P * 4));
  // words the first pillar kernel of every pass clears: the pillar stats [8]
  // and the backbone's per-layer arrival counters and exit count
  RS(dalloc(c, &b.frame_zero, kFrameZeroBytes));
  CK(cudaMemset(b.frame_zero, 0, kFrameZeroBytes));
  p.stats = reinterpret_cast<int*>(b.frame_zero);
  p.zero_words = p.stats;                       // cleared by the pass's first kernel
  p.n_zero = (int)(kFrameZeroBytes / sizeof(int));
  RS(dalloc(c, &p.cell2pillar, (size_t)cells * 4));
  CK(cudaMemset(p.cnt_cell, 0, (size_t)cells * 4));
  CK(cudaMemset(p.first_cell, 0x7F, (size_t)cells * 4));
  CK(cudaMemset(p.cell2pillar, 0xFF, (size_t)cells * 4));
  // the pseudo-image is agent k's part of the agent-major image tensor
  p.image = static_cast<uint8_t*>(c->image_all) + (size_t)k * c->img_elems * 2;
  b.grid_bar = reinterpret_cast<unsigned*>(static_cast<uint8_t*>(b.frame_zero) + 8 * sizeof(int));
  CK(cudaStreamCreateWithFlags(&b.st, cudaStreamNonBlocking));
  CK(cudaEventCreateWithFlags(&b.h2d_done, cudaEventDisableTiming));
  CK(cudaEventCreateWithFlags(&b.done, cudaEventDisableTiming));
  CK(cudaEventCreateWithFlags(&b.pill_done, cudaEventDisableTiming));
  CK(cudaEventCreate(&b.ev_start));
  CK(cudaEventCreate(&b.ev_bb0));
  CK(cudaEventCreate(&b.ev_bb1));
  CK(cudaEventCreate(&b.ev_end));
  return RTCC_OK;
}

// Branch k's own launch parameters (after build_backbone).
rtcc_status build_branch_params(rtcc_ctx* c, int k) {
  Branch& b = c->br[k];
  b.feat = static_cast<uint8_t*>(c->feat_all) + (size_t)k * c->feat_elems * 2;
  if (c->cfg.flags & RTCC_FLAG_LAYER_TIMES) {
    RS(dalloc(c, &b.stamps, 2 * c->layers.size() * sizeof(unsigned long long)));
    CK(cudaMemset(b.stamps, 0, 2 * c->layers.size() * sizeof(unsigned long long)));
  }
  b.bb = new (std::nothrow) BackboneParams;
  if (!b.bb) return RTCC_E_NOMEM;
  *b.bb = *c->bbt[1];
  b.bb->agents[0] = k;
  b.bb->grid_bar = b.grid_bar;
  b.bb->stamps = b.stamps;
  b.bb->done_word = c->done_words + k;
  b.bb->stall = c->stall;
  for (int l = 0; l < b.bb->n_layers; ++l) {
    b.bb->L[l].ws = b.splitk_ws;
    b.bb->L[l].counters = b.splitk_cnt;
  }
  return RTCC_OK;
}

// Timestamp node inside a captured graph (a plain record only adds a
// dependency during capture).
cudaError_t record_node(cudaEvent_t ev, cudaStream_t st) {
  return cudaEventRecordWithFlags(ev, st, cudaEventRecordExternal);
}

// Branch k's graph: the per-frame words, the pillar chain, and (with_bb) the
// backbone of this agent alone as a programmatic dependent of the PFN.
rtcc_status capture_branch_graph(rtcc_ctx* c, int k, const PillarBufs& pb, bool with_bb,
                                 cudaGraphExec_t* out) {
  Branch& b = c->br[k];
  const bool tl = with_bb && (c->cfg.flags & RTCC_FLAG_TIMELINE) != 0;
  (void)cudaGetLastError();   // no stale error may leak into the launch checks
  GridGeom gg{c->cfg.x_min, c->cfg.y_min, c->cfg.z_min, c->cfg.z_max, c->cfg.pillar, c->W, c->H};
  CK(cudaStreamBeginCapture(b.st, cudaStreamCaptureModeRelaxed));
  cudaError_t e = cudaSuccess;
  if (tl) e = record_node(b.ev_start, b.st);
  // kernels only (the first one clears the per-frame words), so that the
  // pillar chain and the backbone are programmatic dependent launches of each
  // other
  if (e == cudaSuccess) e = launch_pillarise(pb, gg, c->pfn_w, c->pfn_b, c->bf16, b.st);
  if (e == cudaSuccess && tl) e = record_node(b.ev_bb0, b.st);
  if (e == cudaSuccess && with_bb) e = launch_backbone(*b.bb, c->bf16, b.st);
  if (e == cudaSuccess && tl) e = record_node(b.ev_bb1, b.st);
  if (e == cudaSuccess && tl) e = record_node(b.ev_end, b.st);
  cudaGraph_t graph = nullptr;
  cudaError_t e2 = cudaStreamEndCapture(b.st, &graph);
  if (e != cudaSuccess || e2 != cudaSuccess) {
    if (graph) cudaGraphDestroy(graph);
    return RTCC_E_CUDA;
  }
  e = cudaGraphInstantiate(out, graph, 0);
  cudaGraphDestroy(graph);
  return e == cudaSuccess ? RTCC_OK : RTCC_E_CUDA;
}

// Four graphs per branch: with and without the backbone (a branch released
// alone runs its own; branches released together share one batched launch),
// each for a payload already in the device slot and for one whose first
// kernel reads the payload from the pinned staging buffer (over the host
// link) and copies it into the device slot as it goes, so a host payload
// needs no copy-engine transfer and no cross-stream event.
rtcc_status capture_branch(rtcc_ctx* c, int k) {
  Branch& b = c->br[k];
  PillarBufs ph = b.pb;
  ph.src_hdr = reinterpret_cast<const int*>(b.staging);
  ph.src_pts = reinterpret_cast<const float4*>(reinterpret_cast<const uint8_t*>(b.staging) + kHdrBytes);
  ph.dst_hdr = reinterpret_cast<int*>(b.in_dev);
  ph.dst_pts = reinterpret_cast<float4*>(b.in_dev + kHdrBytes);
  RS(capture_branch_graph(c, k, b.pb, true, &b.exec));
  RS(capture_branch_graph(c, k, ph, true, &b.exec_host));
  RS(capture_branch_graph(c, k, b.pb, false, &b.pill));
  return capture_branch_graph(c, k, ph, false, &b.pill_host);
}

rtcc_status capture_post(rtcc_ctx* c) {
  const bool tl = (c->cfg.flags & RTCC_FLAG_TIMELINE) != 0;
  // multi-scale placement: fuse each block's outputs, run the neck once on the
  // fused maps, then the head over that one map (the max "fusion" of a single
  // input is the identity, so the tensor-core head kernel serves as the head).
  // Single-scale attention takes the same two steps on the 384-channel slots:
  // the bandwidth-bound fusion writes the fused map, the tensor-core kernel
  // runs the head over it.
  const bool attn1 = !c->ms && c->cfg.fusion == RTCC_FUSE_ATTN && fuse_tc_chunk(c->Cf, 1) > 0 && c->fused;
  FuseBlocksArgs fb{};
  if (attn1) {
    fb.n = 1;
    fb.src[0] = c->feat_all;
    fb.cells[0] = c->Wf * c->Hf;
    fb.ch[0] = c->Cf;
    fb.astride[0] = (long long)c->feat_elems;
    fb.dst[0] = c->fused;
    fb.present = c->d_present;
    fb.K = c->K;
    fb.attention = 1;
    fb.span = c->fuse_span;
  } else if (c->ms) {
    fb.n = c->cfg.n_blocks;
    for (int bi = 0; bi < fb.n; ++bi) {
      fb.src[bi] = c->block_out[bi];
      fb.cells[bi] = c->block_w[bi] * c->block_h[bi];
      fb.ch[bi] = c->cfg.block_ch[bi];
      fb.astride[bi] = (long long)fb.cells[bi] * fb.ch[bi];
      fb.dst[bi] = c->fblk[bi];
    }
    fb.present = c->d_present;
    fb.K = c->K;
    fb.attention = c->cfg.fusion == RTCC_FUSE_ATTN;
    fb.span = c->fuse_span;
  }
  const bool two_step = c->ms || attn1;
  const int K_head = two_step ? 1 : c->K;
  FuseArgs fa{};
  fa.feats = c->d_feat_ptrs;
  fa.present = c->d_present;
  fa.K = c->K;
  fa.C = c->Cf;
  fa.cells = c->Wf * c->Hf;
  fa.attention = c->cfg.fusion == RTCC_FUSE_ATTN;
  fa.head_wp = c->head_wp;
  fa.head_b = c->head_b;
  fa.head_out = c->head_out;
  fa.fused = c->fused;
  fa.keys = c->keys;
  fa.hist0 = c->hist0;
  fa.cls_thresh = c->cfg.cls_thresh;
  fa.anchors = c->cfg.anchors;
  fa.span = c->fuse_span;
  // max fusion: tensor-core kernel (TMA-staged agent tiles, max in shared
  // memory, head as an N = 16 MMA); attention fusion: CUDA-core kernel
  const int bkc = fuse_tc_chunk(c->Cf, K_head);
  const bool use_tc = (two_step || !fa.attention) && bkc > 0;
  if (two_step && !use_tc) return RTCC_E_ARG;
  FuseTcParams tp{};
  if (use_tc) {
    const int swz = bkc * 2;                    // 128- or 64-byte rows
    for (int k = 0; k < K_head; ++k)
      CK(tmap_2d(&tp.feat[k], c->ms ? c->neck_out : (attn1 ? c->fused : c->br[k].feat), c->bf16,
                 (uint64_t)c->Cf,
                 (uint64_t)fa.cells, (uint32_t)bkc, 128u, swz));
    // the K slots are consecutive in feat_all (K_head = 1: the one fused map)
    CK(tmap_3d(&tp.feat_all, c->ms ? c->neck_out : (attn1 ? c->fused : c->feat_all), c->bf16,
               (uint64_t)c->Cf, (uint64_t)fa.cells, (uint64_t)K_head, (uint32_t)bkc, 128u,
               (uint32_t)K_head, swz));
    CK(tmap_2d(&tp.wmap, c->head_w16, c->bf16, (uint64_t)c->Cf, 16u, (uint32_t)bkc, 16u, swz));
    tp.present = two_step ? c->d_one : c->d_present;
    tp.K = K_head;
    tp.C = c->Cf;
    tp.cells = fa.cells;
    tp.bkc = bkc;
    tp.stages = fuse_tc_stages(c->Cf, K_head);
    tp.head_b = c->head_b;
    tp.head_out = c->head_out;
    tp.fused = two_step ? nullptr : c->fused;
    tp.keys = c->keys;
    tp.hist0 = c->hist0;
    tp.cls_thresh = c->cfg.cls_thresh;
    tp.anchors = c->cfg.anchors;
    tp.err = c->d_err;
    tp.span = two_step ? nullptr : c->fuse_span;
  }
  DecodeArgs da{};
  da.head = c->head_out;
  da.keys = c->keys;
  da.hist0 = c->hist0;
  da.feat_w = c->Wf;
  da.feat_h = c->Hf;
  da.anchors = c->cfg.anchors;
  da.x_min = c->cfg.x_min;
  da.y_min = c->cfg.y_min;
  da.x_max = c->cfg.x_max;
  da.y_max = c->cfg.y_max;
  da.max_boxes = c->cfg.max_boxes;
  da.err = c->d_err;
  da.out = c->det_host;                           // pinned host memory, addressable on the device
  da.present = c->d_present;
  da.K = c->K;
  da.done = c->h_done;
  da.dev_boxes = c->dec_boxes;                    // null without NMS
  da.dev_n = c->dec_n;
  NmsArgs na{};
  na.in = c->dec_boxes;
  na.n_in = c->dec_n;
  na.mask = c->nms_mask;
  na.ticket = c->nms_ticket;
  na.max_boxes = c->cfg.max_boxes;
  na.iou = c->cfg.nms_iou;
  na.err = c->d_err;
  na.out = c->det_host;
  na.done = c->h_done;
  (void)cudaGetLastError();
  CK(cudaStreamBeginCapture(c->post, cudaStreamCaptureModeRelaxed));
  cudaError_t e = cudaSuccess;
  if (tl) e = record_node(c->ev_post0, c->post);
  if (e == cudaSuccess && tl) e = record_node(c->ev_fuse0, c->post);
  if (two_step) {
    if (e == cudaSuccess) e = launch_fuse_blocks(fb, c->bf16, c->post);
    if (e == cudaSuccess && tl) e = record_node(c->ev_fuse1, c->post);
    if (e == cudaSuccess && c->ms) e = launch_backbone(*c->neck_p, c->bf16, c->post);
    if (e == cudaSuccess) e = launch_fuse_max_head(tp, c->bf16, c->post);
  } else {
    if (e == cudaSuccess) {
      if (use_tc)
        e = launch_fuse_max_head(tp, c->bf16, c->post);
      else
        e = launch_fuse_head(fa, c->bf16, c->post);
    }
    if (e == cudaSuccess && tl) e = record_node(c->ev_fuse1, c->post);
  }
  if (e == cudaSuccess) e = launch_decode(da, c->post);
  if (e == cudaSuccess && c->dec_boxes) e = launch_nms(na, c->post);
  if (e == cudaSuccess && tl) e = record_node(c->ev_post1, c->post);
  // fusion(s) and head, decode, NMS
  c->post_kernels = (two_step ? (c->ms ? 3 : 2) : 1) + 1 + (c->dec_boxes ? 1 : 0);
  cudaGraph_t graph = nullptr;
  cudaError_t e2 = cudaStreamEndCapture(c->post, &graph);
  if (e != cudaSuccess || e2 != cudaSuccess) {
    if (graph) cudaGraphDestroy(graph);
    return RTCC_E_CUDA;
  }
  e = cudaGraphInstantiate(&c->post_exec, graph, 0);
  cudaGraphDestroy(graph);
  return e == cudaSuccess ? RTCC_OK : RTCC_E_CUDA;
}

void free_all(rtcc_ctx* c) {
  if (c->disp.joinable()) {
    {
      std::lock_guard<std::mutex> lk(c->mu);
      c->stop = true;
    }
    c->cv.notify_all();
    c->disp.join();
  }
  for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
    Branch& b = c->br[k];
    if (b.st) cudaStreamSynchronize(b.st);
    for (cudaGraphExec_t g : {b.exec, b.exec_host, b.pill, b.pill_host})
      if (g) cudaGraphExecDestroy(g);
    for (cudaEvent_t ev : {b.h2d_done, b.done, b.pill_done, b.ev_start, b.ev_bb0, b.ev_bb1, b.ev_end})
      if (ev) cudaEventDestroy(ev);
    delete b.bb;
    b.bb = nullptr;
    if (b.st) cudaStreamDestroy(b.st);
  }
  if (c->bbst) cudaStreamSynchronize(c->bbst);
  if (c->post) cudaStreamSynchronize(c->post);
  if (c->xfer) cudaStreamSynchronize(c->xfer);
  if (c->post_exec) cudaGraphExecDestroy(c->post_exec);
  for (cudaEvent_t ev : {c->det_ready, c->ev_post0, c->ev_fuse0, c->ev_fuse1, c->ev_post1})
    if (ev) cudaEventDestroy(ev);
  for (int j = 0; j < RTCC_MAX_AGENTS; ++j)
    for (cudaEvent_t ev : {c->batch_ev[j], c->batch_t0[j], c->batch_t1[j]})
      if (ev) cudaEventDestroy(ev);
  for (int n = 0; n <= RTCC_MAX_AGENTS; ++n) {
    delete c->bbt[n];
    c->bbt[n] = nullptr;
  }
  delete c->launch_p;
  delete c->neck_p;
  c->launch_p = nullptr;
  if (c->bbst) cudaStreamDestroy(c->bbst);
  if (c->post) cudaStreamDestroy(c->post);
  if (c->xfer) cudaStreamDestroy(c->xfer);
  for (void* p : c->allocs) cudaFree(p);
  for (void* p : c->host_allocs) cudaFreeHost(p);
  c->allocs.clear();
  c->host_allocs.clear();
}

void dispatcher_main(rtcc_ctx* c);

rtcc_status init_impl(rtcc_ctx* c, const float* weights) {
  const rtcc_model_config& g = c->cfg;
  RS(upload_weights(c, weights));
  RS(dalloc(c, &c->d_err, 16));
  if (g.flags & RTCC_FLAG_TIMELINE) {
    RS(dalloc(c, &c->fuse_span, 3 * sizeof(unsigned long long)));
    CK(cudaMemset(c->fuse_span, 0, 3 * sizeof(unsigned long long)));
  }
  CK(cudaMemset(c->d_err, 0, 16));
  RS(dalloc(c, &c->d_present, RTCC_MAX_AGENTS * 4));
  CK(cudaMemset(c->d_present, 0, RTCC_MAX_AGENTS * 4));
  {
    int* d = nullptr;
    RS(halloc(c, &d, 2 * RTCC_MAX_AGENTS * sizeof(int)));
    for (int i = 0; i < 2 * RTCC_MAX_AGENTS; ++i) d[i] = 1;
    c->done_words = d;
    if (g.flags & RTCC_FLAG_SHORT_WAITS) {
      int* s = nullptr;
      RS(halloc(c, &s, sizeof(int)));
      *s = 0;
      c->stall = s;
    }
  }
  const size_t img = (size_t)c->W * c->H * c->Cp;
  RS(dalloc(c, &c->image_all, (size_t)c->K * img * 2));
  CK(cudaMemset(c->image_all, 0, (size_t)c->K * img * 2));
  c->img_elems = img;
  for (int k = 0; k < c->K; ++k) RS(build_branch(c, k));
  RS(build_backbone(c));
  for (int k = 0; k < c->K; ++k) RS(build_branch_params(c, k));
  const int cells_f = c->Wf * c->Hf;
  RS(dalloc(c, &c->d_feat_ptrs, RTCC_MAX_AGENTS * sizeof(void*)));
  void* fp[RTCC_MAX_AGENTS] = {};
  for (int k = 0; k < c->K; ++k) fp[k] = c->br[k].feat;
  CK(cudaMemcpy(c->d_feat_ptrs, fp, sizeof(fp), cudaMemcpyHostToDevice));
  RS(dalloc(c, &c->head_out, (size_t)cells_f * 16 * sizeof(float)));
  // attention fusion writes the fused map (the head then reads it), so it always
  // has one; max fusion keeps it only for parity read-backs
  if ((g.flags & RTCC_FLAG_KEEP_FUSED) || (g.fusion == RTCC_FUSE_ATTN && !c->ms))
    RS(dalloc(c, &c->fused, (size_t)cells_f * c->Cf * 2));
  {
    int one[RTCC_MAX_AGENTS] = {1};
    RS(dalloc(c, &c->d_one, sizeof(one)));
    CK(cudaMemcpy(c->d_one, one, sizeof(one), cudaMemcpyHostToDevice));
  }
  const size_t nkeys = decode_key_capacity(cells_f * g.anchors);
  RS(dalloc(c, &c->keys, nkeys * sizeof(uint32_t)));
  CK(cudaMemset(c->keys, 0xFF, nkeys * sizeof(uint32_t)));   // padding stays invalid
  RS(dalloc(c, &c->hist0, kDecodeHistBins * sizeof(uint32_t)));
  CK(cudaMemset(c->hist0, 0, kDecodeHistBins * sizeof(uint32_t)));
  if (g.nms_iou > 0.f) {
    RS(dalloc(c, &c->dec_boxes, (size_t)g.max_boxes * sizeof(rtcc_box)));
    RS(dalloc(c, &c->dec_n, sizeof(int)));
    CK(cudaMemset(c->dec_n, 0, sizeof(int)));
    RS(dalloc(c, &c->nms_mask, nms_mask_words(g.max_boxes) * sizeof(uint32_t)));
    // all ones: a word the kernel read without writing it this frame would
    // suppress boxes (and show in the parity tests) instead of passing as 0
    CK(cudaMemset(c->nms_mask, 0xFF, nms_mask_words(g.max_boxes) * sizeof(uint32_t)));
    RS(dalloc(c, &c->nms_ticket, sizeof(unsigned)));
    CK(cudaMemset(c->nms_ticket, 0, sizeof(unsigned)));
  }
  c->det_bytes = sizeof(DetResultHeader) + (size_t)g.max_boxes * sizeof(rtcc_box);
  RS(halloc(c, &c->det_host, c->det_bytes));
  std::memset(c->det_host, 0, c->det_bytes);
  {
    int* d = nullptr;
    RS(halloc(c, &d, sizeof(int)));
    *d = 0;
    c->h_done = d;
  }
  CK(cudaStreamCreateWithFlags(&c->xfer, cudaStreamNonBlocking));
  CK(cudaStreamCreateWithFlags(&c->post, cudaStreamNonBlocking));
  CK(cudaStreamCreateWithFlags(&c->bbst, cudaStreamNonBlocking));
  CK(cudaEventCreateWithFlags(&c->det_ready, cudaEventDisableTiming));
  CK(cudaEventCreate(&c->ev_post0));
  CK(cudaEventCreate(&c->ev_fuse0));
  CK(cudaEventCreate(&c->ev_fuse1));
  CK(cudaEventCreate(&c->ev_post1));
  for (int j = 0; j < RTCC_MAX_AGENTS; ++j) {
    CK(cudaEventCreateWithFlags(&c->batch_ev[j], cudaEventDisableTiming));
    CK(cudaEventCreate(&c->batch_t0[j]));
    CK(cudaEventCreate(&c->batch_t1[j]));
  }
  for (int k = 0; k < c->K; ++k) RS(capture_branch(c, k));
  RS(capture_post(c));
  // warm-up: every graph once on empty payloads (pays first-launch costs),
  // and one batched launch of every batch size
  for (int k = 0; k < c->K; ++k) CK(cudaGraphLaunch(c->br[k].exec, c->br[k].st));
  for (int k = 0; k < c->K; ++k) CK(cudaGraphLaunch(c->br[k].exec_host, c->br[k].st));
  for (int k = 0; k < c->K; ++k) CK(cudaGraphLaunch(c->br[k].pill, c->br[k].st));
  for (int k = 0; k < c->K; ++k) CK(cudaStreamSynchronize(c->br[k].st));
  for (int n = 2; n <= c->K; ++n) {
    *c->launch_p = *c->bbt[n];
    c->launch_p->stall = nullptr;
    CK(launch_backbone(*c->launch_p, c->bf16, c->bbst));
  }
  CK(cudaStreamSynchronize(c->bbst));
  CK(cudaGraphLaunch(c->post_exec, c->post));
  CK(cudaStreamSynchronize(c->post));
  int herr = 0;
  CK(cudaMemcpy(&herr, c->d_err, 4, cudaMemcpyDeviceToHost));
  if (herr) return RTCC_E_DEVICE;
  if (!(g.flags & RTCC_FLAG_NO_BATCH)) {
    c->disp = std::thread(dispatcher_main, c);
  }
  return RTCC_OK;
}

// Make agent k's payload available to its first kernel.  Returns whether the
// branch graphs that read the pinned staging buffer (zero-copy) are to be
// used; with RTCC_FLAG_H2D_COPY the payload is instead copied to the device
// slot by the copy engine on the transfer stream, and the branch stream waits
// for that copy's event (the release path of Sec. IV-F as written).
rtcc_status stage_payload(rtcc_ctx* c, int k, bool* host_variant) {
  Branch& b = c->br[k];
  *host_variant = false;
  if (b.pend_resident) return RTCC_OK;
  const int n = b.pend_n;
  float* pts = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(b.staging) + kHdrBytes);
  if (n > 0 && b.pend_ptr != pts) std::memcpy(pts, b.pend_ptr, (size_t)n * 16);
  *reinterpret_cast<volatile int*>(b.staging) = n;
  std::atomic_thread_fence(std::memory_order_seq_cst);
  if (c->cfg.flags & RTCC_FLAG_H2D_COPY) {
    CK(cudaMemcpyAsync(b.in_dev, b.staging, kHdrBytes + (size_t)n * 16, cudaMemcpyHostToDevice, c->xfer));
    CK(cudaEventRecord(b.h2d_done, c->xfer));
    CK(cudaStreamWaitEvent(b.st, b.h2d_done, 0));
    return RTCC_OK;
  }
  *host_variant = true;
  return RTCC_OK;
}

void note_dispatch(rtcc_ctx* c, int k) {
  Branch& b = c->br[k];
  b.launched = true;
  c->ctrl.mark(k, RTCC_RUNNING);
  c->present_dirty = true;
  c->info.t_release_ms[k] = now_ms();
  if (c->info.n_dispatched < RTCC_MAX_AGENTS) c->info.dispatch_order[c->info.n_dispatched++] = k;
}

void note_launch(rtcc_ctx* c, int word, int size) {
  if (c->n_launches < RTCC_MAX_AGENTS) {
    c->launch_size[c->n_launches] = size;
    c->launch_word[c->n_launches] = word;
  }
  ++c->n_launches;
  c->inflight = word;
}

// Branch k released alone: pillar chain and its own backbone (one graph).
// Called with the context mutex held, as are the launches below.
rtcc_status launch_full(rtcc_ctx* c, int k) {
  Branch& b = c->br[k];
  bool hv = false;
  RS(stage_payload(c, k, &hv));
  c->done_words[k] = 0;
  CK(cudaGraphLaunch(hv ? b.exec_host : b.exec, b.st));
  CK(cudaEventRecord(b.done, b.st));
  b.feat_ev = b.done;
  b.stamp_src = k;
  b.launch_idx = c->n_launches;
  b.full_graph = true;
  note_launch(c, k, 1);
  note_dispatch(c, k);
  return RTCC_OK;
}

// Branch k's pillar chain alone; its backbone joins a batch.
rtcc_status launch_pill(rtcc_ctx* c, int k) {
  Branch& b = c->br[k];
  bool hv = false;
  RS(stage_payload(c, k, &hv));
  CK(cudaGraphLaunch(hv ? b.pill_host : b.pill, b.st));
  CK(cudaEventRecord(b.pill_done, b.st));
  c->pending.push_back(k);
  note_dispatch(c, k);
  return RTCC_OK;
}

// One backbone launch for every pending agent (their pillar chains are
// already enqueued).  One agent: its own launch parameters, on its own stream
// behind its pillar chain.  Several: the batch template for that count, on
// the batch stream after every chain's event; each agent still writes its
// own slot, and its result does not depend on the batch (see pick_tile_batch).
rtcc_status launch_batch(rtcc_ctx* c) {
  std::vector<int> ag = c->pending;
  c->pending.clear();
  if (ag.empty()) return RTCC_OK;
  std::sort(ag.begin(), ag.end());
  const bool tl = (c->cfg.flags & RTCC_FLAG_TIMELINE) != 0;
  const int n = (int)ag.size();
  if (n == 1) {
    Branch& b = c->br[ag[0]];
    c->done_words[ag[0]] = 0;
    if (tl) CK(cudaEventRecord(b.ev_bb0, b.st));
    CK(launch_backbone(*b.bb, c->bf16, b.st));
    if (tl) CK(cudaEventRecord(b.ev_bb1, b.st));
    CK(cudaEventRecord(b.done, b.st));
    b.feat_ev = b.done;
    b.stamp_src = ag[0];
    b.launch_idx = c->n_launches;
    note_launch(c, ag[0], 1);
    return RTCC_OK;
  }
  const int j = std::min(c->n_launches, RTCC_MAX_AGENTS - 1);
  const int word = RTCC_MAX_AGENTS + j;
  BackboneParams& P = *c->launch_p;
  P = *c->bbt[n];
  for (int i = 0; i < n; ++i) P.agents[i] = ag[i];
  P.stamps = c->br[ag[0]].stamps;
  P.done_word = c->done_words + word;
  P.stall = c->stall;
  for (int k : ag) CK(cudaStreamWaitEvent(c->bbst, c->br[k].pill_done, 0));
  c->done_words[word] = 0;
  if (tl) CK(cudaEventRecord(c->batch_t0[j], c->bbst));
  CK(launch_backbone(P, c->bf16, c->bbst));
  if (tl) CK(cudaEventRecord(c->batch_t1[j], c->bbst));
  CK(cudaEventRecord(c->batch_ev[j], c->bbst));
  for (int k : ag) {
    c->br[k].feat_ev = c->batch_ev[j];
    c->br[k].stamp_src = ag[0];
    c->br[k].launch_idx = c->n_launches;
  }
  note_launch(c, word, n);
  return RTCC_OK;
}

bool backbone_busy(const rtcc_ctx* c) { return c->inflight >= 0 && c->done_words[c->inflight] == 0; }

rtcc_status launch_post(rtcc_ctx* c) {
  // the presence flags are set on the device by the branches that ran (their
  // first kernel) and cleared by the decode kernel
  for (int k = 0; k < c->K; ++k)
    if (c->ctrl.present(k)) CK(cudaStreamWaitEvent(c->post, c->br[k].feat_ev, 0));
  *c->h_done = 0;                                 // the decode kernel sets it when the boxes are written
  std::atomic_thread_fence(std::memory_order_seq_cst);
  CK(cudaGraphLaunch(c->post_exec, c->post));
  CK(cudaEventRecord(c->det_ready, c->post));
  c->post_launched = true;
  return RTCC_OK;
}

// Dispatch what an event made ready; launch the post-join once every branch
// is resolved.  `t_entry` is the host time the event call began.
//
// Batching (unless RTCC_FLAG_NO_BATCH): a release that does not resolve the
// last branch enqueues only its pillar chain and waits in `pending`; the
// dispatcher thread launches one backbone over every pending agent once the
// backbone in flight (if any) has ended and no release has come for kHoldMs.
// Completions reported close together (several agents completing at one
// instant, reported by one call each) so share one launch, and a lone branch
// loses only the hold beyond its pillar chain, which the backbone waits for
// anyway.  Agents released by one event (Barrier's release of all branches at
// A) form one batch.  The release that resolves the last branch launches at
// once: with nothing pending and the GPU free, as its own branch graph;
// otherwise with whatever is pending, queued behind the running backbone;
// the post-join follows.
rtcc_status after_event(rtcc_ctx* c, const std::vector<int>& released, double t_entry) {
  const bool batching = (c->cfg.flags & RTCC_FLAG_NO_BATCH) == 0;
  const bool last = c->ctrl.join_ready();
  if (!batching) {
    for (int k : released) RS(launch_full(c, k));
  } else if (released.size() == 1 && last && c->pending.empty() && !backbone_busy(c)) {
    RS(launch_full(c, released[0]));
  } else if (!released.empty()) {
    for (int k : released) RS(launch_pill(c, k));
    if (released.size() > 1 || last) {
      RS(launch_batch(c));
    } else {
      // the hold starts after the wake-up call, which can take microseconds;
      // the dispatcher reads it only once this call has released the mutex
      c->cv.notify_all();
      c->t_hold.store(now_ms(), std::memory_order_relaxed);
    }
  }
  if (last && !c->post_launched) {
    if (!c->pending.empty()) RS(launch_batch(c));
    c->t_last_event = t_entry;
    RS(launch_post(c));
  }
  return RTCC_OK;
}

// Gathering window of a batch: a release leaves its batch open this long for
// the next one.  It covers the host's gap between completions reported back
// to back, and stays near the pillar chain's own length (about 20 us), which
// the backbone waits for in any case.
constexpr double kHoldMs = 0.04;

// Launches the pending batch once the backbone in flight has ended and the
// hold has run out (see after_event).  Waits for the end on the launch's done
// word in pinned host memory, without the context mutex.
void dispatcher_main(rtcc_ctx* c) {
  cudaSetDevice(c->dev);
  std::unique_lock<std::mutex> lk(c->mu);
  while (true) {
    c->cv.wait(lk, [c] { return c->stop || !c->pending.empty(); });
    if (c->stop) break;
    const int w = c->inflight;
    lk.unlock();
    const double t0 = now_ms();
    for (uint32_t it = 1; w >= 0 && c->done_words[w] == 0; ++it) {
      // a launch that never reports its end (it failed) stops holding the batch back
      if ((it & 1023u) == 0 && now_ms() - t0 > 2000.0) break;
    }
    while (now_ms() - c->t_hold.load(std::memory_order_relaxed) < kHoldMs) {
    }
    lk.lock();
    if (c->stop) break;
    // a release that came in meanwhile reopens the hold (the loop comes back)
    if (!c->pending.empty() && c->inflight == w &&
        now_ms() - c->t_hold.load(std::memory_order_relaxed) >= kHoldMs) {
      if (launch_batch(c) != RTCC_OK) c->disp_err = true;
    }
  }
}

}  // namespace

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------

extern "C" {

rtcc_status rtcc_init(const rtcc_model_config* cfg, const float* weights, size_t n_floats,
                      rtcc_ctx** out) {
  if (!cfg || !weights || !out) return RTCC_E_ARG;
  *out = nullptr;
  RS(validate_config(*cfg));
  const bool neck = cfg->up_stride[0] != 0;
  const int cf = neck ? cfg->up_ch * cfg->n_blocks : cfg->block_ch[0];
  if (n_floats != expected_floats(*cfg, cf)) return RTCC_E_ARG;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return RTCC_E_CUDA;
  rtcc_ctx* c = new (std::nothrow) rtcc_ctx(cfg->n_agents, cfg->max_points,
                                            cfg->fusion == RTCC_FUSE_ATTN);
  if (!c) return RTCC_E_NOMEM;
  c->cfg = *cfg;
  c->dev = dev;
  c->bf16 = cfg->dtype == RTCC_BF16;
  c->K = cfg->n_agents;
  c->W = cfg->grid_w;
  c->H = cfg->grid_h;
  c->Cp = cfg->pfn_ch;
  c->P = cfg->max_pillars;
  c->N = cfg->max_pts;
  c->cap = std::max(cfg->max_points, 1);
  c->Wf = cfg->grid_w / cfg->block_stride[0];
  c->Hf = cfg->grid_h / cfg->block_stride[0];
  c->Cf = cf;
  for (int b = 0; b < cfg->n_blocks; ++b) c->n_conv += cfg->block_layers[b];
  c->n_deconv = neck ? cfg->n_blocks : 0;
  rtcc_status s = init_impl(c, weights);
  if (s != RTCC_OK) {
    free_all(c);
    delete c;
    return s;
  }
  *out = c;
  return RTCC_OK;
}

void rtcc_destroy(rtcc_ctx* c) {
  if (!c) return;
  free_all(c);
  delete c;
}

rtcc_status rtcc_set_mode(rtcc_ctx* c, rtcc_mode mode) {
  if (!c) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  return c->ctrl.set_mode(mode);
}

rtcc_status rtcc_staging_buffer(rtcc_ctx* c, int32_t agent, float** host_points,
                                int32_t* cap_points) {
  if (!c) return RTCC_E_ARG;
  if (agent < 0 || agent >= c->K) return RTCC_E_AGENT;
  if (host_points)
    *host_points = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(c->br[agent].staging) +
                                            kHdrBytes);
  if (cap_points) *cap_points = c->cfg.max_points;
  return RTCC_OK;
}

rtcc_status rtcc_stage_resident(rtcc_ctx* c, int32_t agent, const float* host_points,
                                int32_t n_points) {
  if (!c) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  if (agent < 0 || agent >= c->K) return RTCC_E_AGENT;
  if (c->ctrl.frame_open()) return RTCC_E_STATE;
  if (n_points < 0 || n_points > c->cfg.max_points || (!host_points && n_points > 0))
    return RTCC_E_MALFORMED;
  Branch& b = c->br[agent];
  CK(cudaStreamSynchronize(b.st));
  CK(cudaStreamSynchronize(c->xfer));
  float* pts = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(b.staging) + kHdrBytes);
  if (n_points > 0 && host_points != pts) std::memcpy(pts, host_points, (size_t)n_points * 16);
  *reinterpret_cast<int*>(b.staging) = n_points;
  CK(cudaMemcpy(b.in_dev, b.staging, kHdrBytes + (size_t)n_points * 16, cudaMemcpyHostToDevice));
  b.resident_ok = true;
  return RTCC_OK;
}

rtcc_status rtcc_frame_begin(rtcc_ctx* c, uint64_t frame_id, double t0_ms) {
  if (!c) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  RS(c->ctrl.begin(frame_id, t0_ms));
  if (c->present_dirty) {
    // a previous frame launched branches but ran no post-join to clear their
    // presence flags
    for (int k = 0; k < c->K; ++k) CK(cudaStreamSynchronize(c->br[k].st));
    CK(cudaStreamSynchronize(c->bbst));
    CK(cudaMemset(c->d_present, 0, RTCC_MAX_AGENTS * 4));
    c->present_dirty = false;
  }
  c->post_launched = false;
  c->n_launches = 0;
  c->pending.clear();
  c->t_last_event = 0.0;
  std::memset(&c->info, 0, sizeof(c->info));
  for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
    c->info.dispatch_order[k] = -1;
    c->info.gpu_backbone_ms[k] = -1.f;
    c->info.gpu_branch_ms[k] = -1.f;
    c->info.t_release_ms[k] = NAN;
    c->br[k].launched = false;
    c->br[k].feat_ev = nullptr;
    c->br[k].stamp_src = -1;
    c->br[k].launch_idx = -1;
    c->br[k].full_graph = false;
  }
  c->info.gpu_fusion_ms = -1.f;
  c->info.gpu_post_ms = -1.f;
  c->info.gpu_fusion_kernel_ms = -1.f;
  for (int k = 0; k < RTCC_MAX_AGENTS; ++k) c->info.gpu_pfn_kernel_ms[k] = -1.f;
  return RTCC_OK;
}

static rtcc_status complete_impl(rtcc_ctx* c, int32_t agent, const float* host_points,
                                 int32_t n_points, double t_ms, bool resident) {
  if (!c) return RTCC_E_ARG;
  const double t_entry = now_ms();
  std::lock_guard<std::mutex> lk(c->mu);
  if (resident && agent >= 0 && agent < c->K && !c->br[agent].resident_ok) return RTCC_E_STATE;
  std::vector<int> rel;
  const void* payload = resident ? static_cast<const void*>(c) : host_points;
  const int n = resident ? 0 : n_points;
  RS(c->ctrl.complete(agent, payload, n, t_ms, &rel));
  Branch& b = c->br[agent];
  b.pend_ptr = host_points;
  b.pend_n = n_points;
  b.pend_resident = resident;
  return after_event(c, rel, t_entry);
}

rtcc_status rtcc_payload_complete(rtcc_ctx* c, int32_t agent, const float* host_points,
                                  int32_t n_points, double t_ms) {
  return complete_impl(c, agent, host_points, n_points, t_ms, false);
}

rtcc_status rtcc_payload_resident(rtcc_ctx* c, int32_t agent, double t_ms) {
  return complete_impl(c, agent, nullptr, 0, t_ms, true);
}

rtcc_status rtcc_payload_absent(rtcc_ctx* c, int32_t agent, double t_ms) {
  if (!c) return RTCC_E_ARG;
  const double t_entry = now_ms();
  std::lock_guard<std::mutex> lk(c->mu);
  std::vector<int> rel;
  RS(c->ctrl.absent(agent, t_ms, &rel));
  return after_event(c, rel, t_entry);
}

rtcc_status rtcc_frame_abort(rtcc_ctx* c) {
  if (!c) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  if (c->post_launched) return RTCC_E_STATE;   // complete already: wait for it instead
  return c->ctrl.abort();
}

rtcc_status rtcc_wait_detection(rtcc_ctx* c, int32_t timeout_ms, rtcc_box* out, int32_t cap,
                                int32_t* n_out, double* t_ready_ms) {
  if (!c) return RTCC_E_ARG;
  cudaEvent_t ev;
  {
    std::lock_guard<std::mutex> lk(c->mu);
    if (!c->ctrl.frame_open()) return RTCC_E_STATE;
    if (c->ctrl.aborted()) {
      // branches already released finish; a batch still held back is
      // launched now so that its pillar chains' work is not left half done
      const rtcc_status ls = launch_batch(c);
      for (int k = 0; k < c->K; ++k)
        if (c->br[k].launched) cudaStreamSynchronize(c->br[k].st);
      cudaStreamSynchronize(c->bbst);
      if (ls != RTCC_OK) return ls;
      // no decode ran to clear the presence flags of the branches that did
      if (cudaMemset(c->d_present, 0, RTCC_MAX_AGENTS * 4) != cudaSuccess) return RTCC_E_CUDA;
      c->present_dirty = false;
      c->ctrl.end();
      return RTCC_E_INFEASIBLE;
    }
    if (!c->post_launched) return RTCC_E_STATE;
    ev = c->det_ready;
  }
  // The decode kernel writes the result block into pinned host memory and then
  // sets h_done; spinning on that word sees the result without a driver call.
  // Every 4096 polls the post stream's event is queried for errors (and to
  // notice a post-join that completed without setting the word).
  const double t0 = now_ms();
  for (uint32_t it = 1;; ++it) {
    if (*c->h_done) break;
    if ((it & 4095u) == 0) {
      const cudaError_t q = cudaEventQuery(ev);
      if (q != cudaSuccess && q != cudaErrorNotReady) return RTCC_E_CUDA;
      if (q == cudaSuccess && !*c->h_done) return RTCC_E_CUDA;
      if (timeout_ms >= 0 && now_ms() - t0 > (double)timeout_ms) return RTCC_E_TIMEOUT;
    }
  }
  const double t_ready = now_ms();
  std::atomic_thread_fence(std::memory_order_acquire);   // the block was written before the flag
  c->present_dirty = false;                              // the decode cleared the presence flags
  if (c->cfg.flags & RTCC_FLAG_TIMELINE) {
    // the event nodes' times are read below: wait for the graph's end
    if (cudaEventSynchronize(ev) != cudaSuccess) return RTCC_E_CUDA;
  }
  std::lock_guard<std::mutex> lk(c->mu);
  const DetResultHeader* hdr = reinterpret_cast<const DetResultHeader*>(c->det_host);
  const rtcc_box* boxes = reinterpret_cast<const rtcc_box*>(hdr + 1);
  const int n = std::min(hdr->n_boxes, c->cfg.max_boxes);
  if (out && cap > 0) std::memcpy(out, boxes, sizeof(rtcc_box) * (size_t)std::min(n, (int)cap));
  if (n_out) *n_out = n;
  if (t_ready_ms) *t_ready_ms = t_ready;
  c->info.t_ready_ms = t_ready;
  c->info.t_last_event_ms = c->t_last_event;
  c->info.n_backbone_launches = c->n_launches;
  for (int j = 0; j < RTCC_MAX_AGENTS; ++j) {
    c->info.backbone_batch[j] = j < c->n_launches ? c->launch_size[j] : 0;
    c->info.gpu_launch_ms[j] = -1.f;
  }
  if (c->cfg.flags & RTCC_FLAG_TIMELINE) {
    for (int j = 0; j < c->n_launches && j < RTCC_MAX_AGENTS; ++j) {
      float ms = -1.f;
      const int w = c->launch_word[j];
      if (w >= RTCC_MAX_AGENTS) {
        if (cudaEventElapsedTime(&ms, c->batch_t0[w - RTCC_MAX_AGENTS], c->batch_t1[w - RTCC_MAX_AGENTS]) ==
            cudaSuccess)
          c->info.gpu_launch_ms[j] = ms;
      } else if (cudaEventElapsedTime(&ms, c->br[w].ev_bb0, c->br[w].ev_bb1) == cudaSuccess) {
        c->info.gpu_launch_ms[j] = ms;
      }
    }
    for (int k = 0; k < c->K; ++k) {
      Branch& b = c->br[k];
      if (!b.launched) continue;
      float ms = -1.f;
      if (b.launch_idx >= 0 && b.launch_idx < RTCC_MAX_AGENTS)
        c->info.gpu_backbone_ms[k] = c->info.gpu_launch_ms[b.launch_idx];
      if (b.full_graph && cudaEventElapsedTime(&ms, b.ev_start, b.ev_end) == cudaSuccess)
        c->info.gpu_branch_ms[k] = ms;
      unsigned long long ps[2] = {0ull, 0ull};
      if (b.pb.pfn_span && cudaMemcpy(ps, b.pb.pfn_span, sizeof(ps), cudaMemcpyDeviceToHost) == cudaSuccess &&
          ps[1] > ps[0])
        c->info.gpu_pfn_kernel_ms[k] = (float)((double)(ps[1] - ps[0]) * 1e-6);
    }
    float ms = -1.f;
    if (cudaEventElapsedTime(&ms, c->ev_fuse0, c->ev_fuse1) == cudaSuccess) c->info.gpu_fusion_ms = ms;
    if (cudaEventElapsedTime(&ms, c->ev_post0, c->ev_post1) == cudaSuccess) c->info.gpu_post_ms = ms;
    unsigned long long sp[2] = {0ull, 0ull};
    if (c->fuse_span && cudaMemcpy(sp, c->fuse_span, sizeof(sp), cudaMemcpyDeviceToHost) == cudaSuccess &&
        sp[1] > sp[0])
      c->info.gpu_fusion_kernel_ms = (float)((double)(sp[1] - sp[0]) * 1e-6);
    (void)cudaGetLastError();
  }
  c->ctrl.end();
  if (c->stall) *c->stall = 0;                 // the test hook lasts one frame
  if (c->disp_err) {
    c->disp_err = false;
    return RTCC_E_CUDA;
  }
  if (hdr->err) {
    // A bounded device wait ran out.  The frame's kernels have all ended (the
    // post-join waited for them); clear the error word and the split-K tile
    // counters a kernel that wound down may have left, so the next frame
    // starts clean.
    for (int k = 0; k < c->K; ++k) cudaStreamSynchronize(c->br[k].st);
    cudaStreamSynchronize(c->bbst);
    cudaStreamSynchronize(c->post);
    CK(cudaMemset(c->d_err, 0, 16));
    for (int k = 0; k < c->K; ++k)
      if (c->br[k].splitk_cnt) CK(cudaMemset(c->br[k].splitk_cnt, 0, c->splitk_cnt_bytes));
    if (c->batch_cnt) CK(cudaMemset(c->batch_cnt, 0, (size_t)c->K * c->splitk_cnt_bytes));
    CK(cudaMemset(c->batch_bar, 0, (kMaxLayers + 1) * sizeof(unsigned)));
    // the pillar passes' per-cell state and their image cells, as at allocation
    const size_t cells = (size_t)c->W * c->H;
    for (int k = 0; k < c->K; ++k) {
      const PillarBufs& p = c->br[k].pb;
      CK(cudaMemset(p.cnt_cell, 0, cells * 4));
      CK(cudaMemset(p.first_cell, 0x7F, cells * 4));
      CK(cudaMemset(p.cell2pillar, 0xFF, cells * 4));
      CK(cudaMemset(p.np_prev, 0, 4));
      CK(cudaMemset(p.image, 0, (size_t)c->img_elems * 2));
    }
    return RTCC_E_DEVICE;
  }
  return RTCC_OK;
}

rtcc_status rtcc_get_frame_info(rtcc_ctx* c, rtcc_frame_info* info) {
  if (!c || !info) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  *info = c->info;
  return RTCC_OK;
}

rtcc_status rtcc_plan_conv(int32_t kind, int32_t cin, int32_t cout, int32_t out_w, int32_t out_h,
                           int32_t grid, int32_t n_batch, rtcc_conv_plan* out) {
  if (!out || (kind != 0 && kind != 1) || cin < 32 || cin > 256 || cout < 32 || cout > 256 ||
      cin % 32 || cout % 32 || (cin & (cin - 1)) || out_w < 1 || out_h < 1 || grid < 1 ||
      n_batch < 1 || n_batch > RTCC_MAX_AGENTS)
    return RTCC_E_ARG;
  ConvLayer L{};
  L.kind = kind == 1 ? CONV3_S2 : CONV3_S1;
  L.cin = cin;
  L.cout = cout;
  L.gw = out_w;
  L.gh = out_h;
  choose_split(L, grid);
  choose_tiles(L, grid, n_batch);
  out->splits = L.splits;
  out->bn = L.bn;
  out->tall = L.tall;
  out->transposed = L.tr;
  out->wide = L.wide;
  out->m_tiles = conv_m_tiles(L);
  out->items = n_batch * out->m_tiles * (cout / L.bn) * L.splits;
  return RTCC_OK;
}

rtcc_status rtcc_get_layer_spans(rtcc_ctx* c, int32_t agent, float* start_ms, float* end_ms,
                                 int32_t cap, int32_t* n_out) {
  if (!c) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  if (agent < 0 || agent >= c->K) return RTCC_E_AGENT;
  if (!c->br[agent].stamps) return RTCC_E_STATE;
  const int n = (int)c->layers.size();
  if (n_out) *n_out = n;
  if (!start_ms && !end_ms) return RTCC_OK;
  // the stamps of the launch that ran this agent (alone or in a batch)
  Branch& b = c->br[c->br[agent].stamp_src >= 0 ? c->br[agent].stamp_src : agent];
  CK(cudaStreamSynchronize(b.st));
  CK(cudaStreamSynchronize(c->bbst));
  std::vector<unsigned long long> t(2 * n);
  CK(cudaMemcpy(t.data(), b.stamps, 2 * n * sizeof(unsigned long long), cudaMemcpyDeviceToHost));
  unsigned long long t0 = 0;
  for (int i = 0; i < 2 * n; ++i)
    if (t[i] > 0 && (t0 == 0 || t[i] < t0)) t0 = t[i];
  for (int i = 0; i < n && i < cap; ++i) {
    const bool ok = t0 > 0 && t[i] > 0 && t[n + i] >= t[i];
    if (start_ms) start_ms[i] = ok ? (float)((t[i] - t0) * 1e-6) : -1.f;
    if (end_ms) end_ms[i] = ok ? (float)((t[n + i] - t0) * 1e-6) : -1.f;
  }
  return RTCC_OK;
}

rtcc_status rtcc_get_layer_times(rtcc_ctx* c, int32_t agent, float* host_ms, int32_t cap,
                                 int32_t* n_out) {
  if (!host_ms || cap <= 0) return rtcc_get_layer_spans(c, agent, nullptr, nullptr, 0, n_out);
  std::vector<float> a(cap), e(cap);
  int32_t n = 0;
  const rtcc_status r = rtcc_get_layer_spans(c, agent, a.data(), e.data(), cap, &n);
  if (r != RTCC_OK) return r;
  if (n_out) *n_out = n;
  for (int i = 0; i < n && i < cap; ++i) host_ms[i] = (a[i] >= 0.f && e[i] >= 0.f) ? e[i] - a[i] : -1.f;
  return RTCC_OK;
}

rtcc_status rtcc_get_branch_state(rtcc_ctx* c, int32_t agent, int32_t* state, double* release_ms) {
  if (!c) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  if (agent >= 0 && agent < c->K && state && release_ms) {
    // observe FINISHED lazily through the branch's completion event
    int st = 0;
    c->ctrl.state(agent, &st, nullptr);
    const cudaEvent_t fe = c->br[agent].feat_ev;
    if (st == RTCC_RUNNING && fe && cudaEventQuery(fe) == cudaSuccess) c->ctrl.mark(agent, RTCC_FINISHED);
  }
  int32_t st = 0;
  rtcc_status s = c->ctrl.state(agent, &st, release_ms);
  if (state) *state = st;
  return s;
}

rtcc_status rtcc_get_head(rtcc_ctx* c, float* host_out, size_t cap) {
  if (!c || !host_out) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  const size_t n = (size_t)c->Wf * c->Hf * 16;
  if (cap < n) return RTCC_E_ARG;
  CK(cudaStreamSynchronize(c->post));
  CK(cudaMemcpy(host_out, c->head_out, n * sizeof(float), cudaMemcpyDeviceToHost));
  return RTCC_OK;
}

rtcc_status rtcc_get_decoded(rtcc_ctx* c, rtcc_box* host_out, int32_t cap, int32_t* n_out) {
  if (!c || (!host_out && cap > 0) || cap < 0) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  CK(cudaStreamSynchronize(c->post));
  int n = 0;
  if (c->dec_boxes) {
    CK(cudaMemcpy(&n, c->dec_n, sizeof(int), cudaMemcpyDeviceToHost));
    n = std::max(0, std::min(n, c->cfg.max_boxes));
    if (cap > 0 && n > 0)
      CK(cudaMemcpy(host_out, c->dec_boxes, sizeof(rtcc_box) * (size_t)std::min(n, cap),
                    cudaMemcpyDeviceToHost));
  } else {
    // without NMS the decode's boxes are the result block's
    const DetResultHeader* hdr = reinterpret_cast<const DetResultHeader*>(c->det_host);
    n = std::max(0, std::min(hdr->n_boxes, c->cfg.max_boxes));
    if (cap > 0 && n > 0)
      std::memcpy(host_out, hdr + 1, sizeof(rtcc_box) * (size_t)std::min(n, cap));
  }
  if (n_out) *n_out = n;
  return RTCC_OK;
}

rtcc_status rtcc_get_pillars(rtcc_ctx* c, int32_t agent, int32_t* host_cell2pillar,
                             int32_t* host_pillar_cell, int32_t* host_count, int32_t* host_stats) {
  if (!c) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  if (agent < 0 || agent >= c->K) return RTCC_E_AGENT;
  Branch& b = c->br[agent];
  CK(cudaStreamSynchronize(b.st));
  int st[8];
  CK(cudaMemcpy(st, b.pb.stats, sizeof(st), cudaMemcpyDeviceToHost));
  const int np = st[2];
  if (host_cell2pillar)
    CK(cudaMemcpy(host_cell2pillar, b.pb.cell2pillar, (size_t)c->W * c->H * 4,
                  cudaMemcpyDeviceToHost));
  if (host_pillar_cell) {
    for (int p = 0; p < c->P; ++p) host_pillar_cell[p] = -1;
    if (np > 0) CK(cudaMemcpy(host_pillar_cell, b.pb.pillar_cell, (size_t)np * 4, cudaMemcpyDeviceToHost));
  }
  if (host_count) {
    for (int p = 0; p < c->P; ++p) host_count[p] = 0;
    if (np > 0) CK(cudaMemcpy(host_count, b.pb.pcount, (size_t)np * 4, cudaMemcpyDeviceToHost));
  }
  if (host_stats) {
    host_stats[0] = st[0];
    host_stats[1] = st[1];
    host_stats[2] = st[2];
    host_stats[3] = st[3];
    host_stats[4] = st[0] - st[1];      // out of range
    host_stats[5] = st[1] - st[7];      // dropped by the pillar cap
    host_stats[6] = st[6];              // dropped by the per-pillar point cap
    host_stats[7] = st[7];
  }
  return RTCC_OK;
}

rtcc_status rtcc_get_tensor(rtcc_ctx* c, int32_t agent, int32_t which, uint16_t* host_out,
                            size_t cap, size_t* n_elems) {
  if (!c) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  const void* src = nullptr;
  size_t n = 0;
  if (which == 9) {
    const void* f = c->ms ? c->neck_out : c->fused;
    if (!f) return RTCC_E_STATE;
    CK(cudaStreamSynchronize(c->post));
    src = f;
    n = (size_t)c->Wf * c->Hf * c->Cf;
  } else if (which >= 10 && which < 10 + c->cfg.n_blocks) {
    if (!c->ms) return RTCC_E_STATE;
    CK(cudaStreamSynchronize(c->post));
    const int bi = which - 10;
    src = c->fblk[bi];
    n = (size_t)c->block_w[bi] * c->block_h[bi] * c->cfg.block_ch[bi];
  } else {
    if (agent < 0 || agent >= c->K) return RTCC_E_AGENT;
    Branch& b = c->br[agent];
    CK(cudaStreamSynchronize(b.st));
    CK(cudaStreamSynchronize(c->bbst));
    if (which == 0) {
      src = b.pb.image;
      n = (size_t)c->W * c->H * c->Cp;
    } else if (which >= 1 && which <= c->cfg.n_blocks) {
      n = (size_t)c->block_w[which - 1] * c->block_h[which - 1] * c->cfg.block_ch[which - 1];
      src = static_cast<const uint8_t*>(c->block_out[which - 1]) + (size_t)agent * n * 2;
    } else if (which == 8) {
      src = b.feat;
      n = (size_t)c->Wf * c->Hf * c->Cf;
    } else if (which >= 16 && which - 16 < (int)c->layer_all.size() &&
               (c->cfg.flags & RTCC_FLAG_KEEP_LAYERS)) {
      n = c->layer_elems[which - 16];
      src = static_cast<const uint8_t*>(c->layer_all[which - 16]) + (size_t)agent * n * 2;
    } else {
      return RTCC_E_ARG;
    }
  }
  if (n_elems) *n_elems = n;
  if (!host_out) return RTCC_OK;
  if (cap < n) return RTCC_E_ARG;
  CK(cudaMemcpy(host_out, src, n * 2, cudaMemcpyDeviceToHost));
  return RTCC_OK;
}

const char* rtcc_status_str(rtcc_status s) {
  switch (s) {
    case RTCC_OK: return "ok";
    case RTCC_E_ARG: return "invalid argument or unsupported config";
    case RTCC_E_AGENT: return "agent index out of range";
    case RTCC_E_DUPLICATE: return "duplicate completion event";
    case RTCC_E_PREMATURE: return "premature event (no open frame or t < t0)";
    case RTCC_E_MALFORMED: return "malformed payload";
    case RTCC_E_STATE: return "call not allowed in this state";
    case RTCC_E_TIMEOUT: return "timed out";
    case RTCC_E_INFEASIBLE: return "frame infeasible (undelivered branches)";
    case RTCC_E_CUDA: return "CUDA error";
    case RTCC_E_NOMEM: return "out of memory";
    case RTCC_E_DEVICE: return "device-side bounded wait expired";
  }
  return "unknown status";
}

double rtcc_now_ms(void) { return now_ms(); }

int32_t rtcc_kernels_per_frame(rtcc_ctx* c, int32_t n_present) {
  if (!c) return 0;
  std::lock_guard<std::mutex> lk(c->mu);
  // pillar chain per branch; the backbone launches of the last frame (one per
  // branch when none was batched); fusion, decode (and NMS)
  const int bb = c->n_launches > 0 ? c->n_launches : n_present;
  return n_present * 5 + bb + c->post_kernels;
}

rtcc_status rtcc_test_unreachable_wait(rtcc_ctx* c) {
  if (!c) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  if (!c->stall) return RTCC_E_STATE;
  if (c->ctrl.frame_open()) return RTCC_E_STATE;
  *c->stall = 1;
  return RTCC_OK;
}

rtcc_status rtcc_nms(const rtcc_box* host_in, int32_t n, float iou, rtcc_box* host_out,
                     int32_t* n_out) {
  if (n < 0 || n > kDecodeKeep || (n > 0 && (!host_in || !host_out)) || !n_out ||
      !(iou >= 0.f && iou <= 1.f))
    return RTCC_E_ARG;
  const int mb = n > 0 ? n : 1;
  // one scratch block: boxes in, count, ticket, error word, done word,
  // result block (header + boxes), bitmask
  const size_t in_b = (size_t)mb * sizeof(rtcc_box), res_b = sizeof(DetResultHeader) + in_b;
  const size_t off_n = (in_b + 15) / 16 * 16, off_res = off_n + 64,
               off_mask = off_res + (res_b + 15) / 16 * 16;
  const size_t total = off_mask + nms_mask_words(mb) * sizeof(uint32_t);
  uint8_t* d = nullptr;
  if (cudaMalloc(&d, total) != cudaSuccess) return RTCC_E_NOMEM;
  cudaStream_t st = nullptr;
  rtcc_status r = RTCC_E_CUDA;
  int* ints = reinterpret_cast<int*>(d + off_n);       // [0] n, [1] ticket, [2] err, [3] done
  do {
    if (cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking) != cudaSuccess) break;
    if (cudaMemsetAsync(d + off_n, 0, 64, st) != cudaSuccess) break;
    // bitmask scratch all ones (see the context's allocation)
    if (cudaMemsetAsync(d + off_mask, 0xFF, nms_mask_words(mb) * sizeof(uint32_t), st) != cudaSuccess) break;
    if (n > 0 && cudaMemcpyAsync(d, host_in, in_b, cudaMemcpyHostToDevice, st) != cudaSuccess) break;
    if (cudaMemcpyAsync(ints, &n, sizeof(int), cudaMemcpyHostToDevice, st) != cudaSuccess) break;
    NmsArgs a{};
    a.in = reinterpret_cast<const rtcc_box*>(d);
    a.n_in = ints;
    a.ticket = reinterpret_cast<unsigned*>(ints + 1);
    a.err = ints + 2;
    a.done = ints + 3;
    a.mask = reinterpret_cast<uint32_t*>(d + off_mask);
    a.max_boxes = mb;
    a.iou = iou;
    a.out = d + off_res;
    if (launch_nms(a, st) != cudaSuccess) break;
    DetResultHeader h{};
    if (cudaMemcpyAsync(&h, d + off_res, sizeof(h), cudaMemcpyDeviceToHost, st) != cudaSuccess) break;
    if (cudaStreamSynchronize(st) != cudaSuccess) break;
    const int k = std::max(0, std::min(h.n_boxes, n));
    if (k > 0 && cudaMemcpy(host_out, d + off_res + sizeof(DetResultHeader), (size_t)k * sizeof(rtcc_box),
                            cudaMemcpyDeviceToHost) != cudaSuccess)
      break;
    *n_out = k;
    r = RTCC_OK;
  } while (false);
  if (st) cudaStreamDestroy(st);
  cudaFree(d);
  return r;
}

}  // extern "C"

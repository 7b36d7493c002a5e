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
#include <cstring>
#include <mutex>
#include <new>
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
  void* block_buf[RTCC_MAX_BLOCKS][2] = {};
  std::vector<void*> layer_out;    // every conv layer's output (RTCC_FLAG_KEEP_LAYERS)
  std::vector<size_t> layer_elems;
  void* block_out[RTCC_MAX_BLOCKS] = {};
  int block_w[RTCC_MAX_BLOCKS] = {}, block_h[RTCC_MAX_BLOCKS] = {};
  void* feat = nullptr;            // agent-indexed feature slot [H'][W'][C_feat]
  std::vector<ConvLayer> layers;
  float* splitk_ws = nullptr;      // split-K partials, shared by the branch's layers
  int* splitk_cnt = nullptr;       // split-K per-tile arrival counters
  unsigned* grid_bar = nullptr;      // inside frame_zero
  void* frame_zero = nullptr;         // [kFrameZeroBytes] cleared at the start of every branch graph    // backbone per-layer arrival counters
  unsigned long long* stamps = nullptr;   // RTCC_FLAG_LAYER_TIMES: layer starts, then ends
  BackboneParams* bb = nullptr;    // backbone kernel parameters (host copy)
  cudaStream_t st = nullptr;
  cudaGraphExec_t exec = nullptr;       // payload already in the device slot
  cudaGraphExec_t exec_host = nullptr;  // payload in the pinned staging buffer (zero-copy)
  cudaEvent_t h2d_done = nullptr, done = nullptr;
  cudaEvent_t ev_start = nullptr, ev_bb0 = nullptr, ev_bb1 = nullptr, ev_end = nullptr;
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
rtcc_status upload_conv(rtcc_ctx* c, const float* w, int co, int ci) {
  std::vector<uint16_t> p((size_t)co * 9 * ci);
  for (int o = 0; o < co; ++o)
    for (int i = 0; i < ci; ++i)
      for (int t = 0; t < 9; ++t)
        p[((size_t)o * 9 + t) * ci + i] = bits_store(w[((size_t)o * ci + i) * 9 + t], c->bf16);
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

constexpr size_t kFrameZeroBytes = 8 * sizeof(int) + kMaxLayers * sizeof(unsigned);

rtcc_status build_branch(rtcc_ctx* c, int k) {
  Branch& b = c->br[k];
  const rtcc_model_config& g = c->cfg;
  // CTAs of a backbone launch in clusters (split-K slices share a cluster)
  int grid = backbone_grid(kMaxSplits);
  if (grid < 1) grid = backbone_grid(1);
  if (grid < 1) return RTCC_E_CUDA;
  const size_t es = 2;   // 16-bit storage
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
  RS(dalloc(c, &p.cell_of, (size_t)c->cap * 4));
  RS(dalloc(c, &p.cnt_cell, (size_t)cells * 4));
  RS(dalloc(c, &p.first_cell, (size_t)cells * 4));
  RS(dalloc(c, &p.c2p, (size_t)cells * 4));
  RS(dalloc(c, &p.blocksum, (size_t)scan_blocks(c->cap) * sizeof(int2)));
  RS(dalloc(c, &p.items, (size_t)scan_blocks(c->cap) * kScanTile * sizeof(int2)));
  RS(dalloc(c, &p.pcnt_raw, (size_t)c->P * 4));
  RS(dalloc(c, &p.poff, (size_t)c->P * 4));
  RS(dalloc(c, &p.cursor, (size_t)c->P * 4));
  RS(dalloc(c, &p.list, (size_t)c->cap * 4));
  RS(dalloc(c, &p.np_prev, 4));
  CK(cudaMemset(p.np_prev, 0, 4));
  p.clear_all = 0;                              // image and cell2pillar start cleared below
  p.present_flag = c->d_present + k;
  if (g.flags & RTCC_FLAG_TIMELINE) {
    RS(dalloc(c, &p.pfn_span, 3 * sizeof(unsigned long long)));
    CK(cudaMemset(p.pfn_span, 0, 3 * sizeof(unsigned long long)));
  }
  RS(dalloc(c, &p.pillar_cell, (size_t)c->P * 4));
  RS(dalloc(c, &p.pcount, (size_t)c->P * 4));
  // words cleared at the start of every branch graph (one memset): the pillar
  // stats [8] and the backbone's per-layer arrival counters [kMaxLayers]
  RS(dalloc(c, &b.frame_zero, kFrameZeroBytes));
  CK(cudaMemset(b.frame_zero, 0, kFrameZeroBytes));
  p.stats = reinterpret_cast<int*>(b.frame_zero);
  RS(dalloc(c, &p.cell2pillar, (size_t)cells * 4));
  RS(dalloc(c, &p.image, (size_t)cells * c->Cp * es));
  CK(cudaMemset(p.cnt_cell, 0, (size_t)cells * 4));
  CK(cudaMemset(p.first_cell, 0x7F, (size_t)cells * 4));
  CK(cudaMemset(p.image, 0, (size_t)cells * c->Cp * es));
  CK(cudaMemset(p.cell2pillar, 0xFF, (size_t)cells * 4));
  RS(dalloc(c, &b.feat, (size_t)c->Wf * c->Hf * c->Cf * es));
  CK(cudaMemset(b.feat, 0, (size_t)c->Wf * c->Hf * c->Cf * es));

  // backbone layers
  const bool neck = g.up_stride[0] != 0;
  int block_last[RTCC_MAX_BLOCKS] = {};
  const void* in = p.image;
  int cin = c->Cp, w = c->W, h = c->H;
  int wi = 0;
  for (int bi = 0; bi < g.n_blocks; ++bi) {
    const int st = g.block_stride[bi];
    const int ow = w / st, oh = h / st;
    const int co = g.block_ch[bi];
    const bool keep = (g.flags & RTCC_FLAG_KEEP_LAYERS) != 0;
    if (!keep) {
      RS(dalloc(c, &b.block_buf[bi][0], (size_t)ow * oh * co * es));
      RS(dalloc(c, &b.block_buf[bi][1], (size_t)ow * oh * co * es));
    }
    for (int li = 0; li < g.block_layers[bi]; ++li) {
      ConvLayer L{};
      L.kind = (li == 0 && st == 2) ? CONV3_S2 : CONV3_S1;
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
      const int m_tiles = ((ow + conv_tile_w() - 1) / conv_tile_w()) *
                          ((oh + conv_tile_h() - 1) / conv_tile_h());
      L.bk = (cin >= 64) ? 64 : 32;
      pick_tile(m_tiles, co, 9 * (cin / L.bk), grid, &L.bn, &L.splits);
      L.n_tiles_n = co / L.bn;
      L.in = in;
      const bool last = (bi == g.n_blocks - 1) && (li == g.block_layers[bi] - 1);
      void* dst = nullptr;
      if (!neck && last) {
        dst = b.feat;
      } else if (keep) {
        RS(dalloc(c, &dst, (size_t)ow * oh * co * es));
      } else {
        dst = b.block_buf[bi][li & 1];
      }
      L.out = dst;
      b.layer_out.push_back(dst);
      b.layer_elems.push_back((size_t)ow * oh * co);
      L.wpacked = c->wbufs[wi];
      L.bias = c->bbufs[wi];
      L.wait_layers = (int)b.layers.size();          // reads the previous conv's output
      ++wi;
      if (conv_make_maps(L, c->bf16) != cudaSuccess) return RTCC_E_CUDA;
      b.layers.push_back(L);
      in = L.out;
      cin = co;
    }
    b.block_out[bi] = const_cast<void*>(in);
    block_last[bi] = (int)b.layers.size();          // layers [0, block_last) done

    b.block_w[bi] = ow;
    b.block_h[bi] = oh;
    w = ow;
    h = oh;
  }
  if (neck) {
    for (int bi = 0; bi < g.n_blocks; ++bi) {
      ConvLayer L{};
      L.kind = DECONV;
      L.s = g.up_stride[bi];
      L.cin = g.block_ch[bi];
      L.cout = g.up_ch;
      L.in_w = b.block_w[bi];
      L.in_h = b.block_h[bi];
      L.out_w = c->Wf;
      L.out_h = c->Hf;
      L.gw = L.in_w;
      L.gh = L.in_h;
      L.ldc = c->Cf;
      L.choff = bi * g.up_ch;
      L.bn = g.up_ch;
      L.bk = (L.cin >= 64) ? 64 : 32;
      L.n_tiles_n = L.s * L.s;
      L.in = b.block_out[bi];
      L.out = b.feat;
      L.wpacked = c->wbufs[wi];
      L.bias = c->bbufs[wi];
      L.wait_layers = block_last[bi];                 // only its block's output
      ++wi;
      if (conv_make_maps(L, c->bf16) != cudaSuccess) return RTCC_E_CUDA;
      b.layers.push_back(L);
    }
  }
  // fp32 workspace of the global-memory split-K reduction (used when a split
  // layer cannot reduce through DSMEM); deconvs do not wait on their
  // predecessor, so they may not share it: they never split
  size_t ws_floats = 0, max_tiles = 0;
  for (ConvLayer& L : b.layers) {
    const int m_tiles = ((L.gw + conv_tile_w() - 1) / conv_tile_w()) *
                        ((L.gh + conv_tile_h() - 1) / conv_tile_h());
    const int base = m_tiles * L.n_tiles_n;
    if (L.kind == DECONV || L.splits < 1) L.splits = 1;
    const int sp = L.splits;
    if (sp > 1) {
      ws_floats = std::max(ws_floats, (size_t)sp * base * conv_tile_m() * L.bn);
      max_tiles = std::max(max_tiles, (size_t)base);
    }
  }
  if (ws_floats) {
    RS(dalloc(c, &b.splitk_ws, ws_floats * sizeof(float)));
    RS(dalloc(c, &b.splitk_cnt, max_tiles * sizeof(int)));
    CK(cudaMemset(b.splitk_cnt, 0, max_tiles * sizeof(int)));
  }
  for (ConvLayer& L : b.layers) {
    L.ws = b.splitk_ws;
    L.counters = b.splitk_cnt;
  }
  b.grid_bar = reinterpret_cast<unsigned*>(static_cast<uint8_t*>(b.frame_zero) + 8 * sizeof(int));
  if (g.flags & RTCC_FLAG_LAYER_TIMES) {
    RS(dalloc(c, &b.stamps, 2 * b.layers.size() * sizeof(unsigned long long)));
    CK(cudaMemset(b.stamps, 0, 2 * b.layers.size() * sizeof(unsigned long long)));
  }
  b.bb = new (std::nothrow) BackboneParams;
  if (!b.bb) return RTCC_E_NOMEM;
  if (backbone_fill(b.layers, b.grid_bar, c->d_err, b.stamps,
                    (g.flags & RTCC_FLAG_NO_CLUSTERS) == 0, b.bb) != cudaSuccess)
    return RTCC_E_ARG;
  CK(cudaStreamCreateWithFlags(&b.st, cudaStreamNonBlocking));
  CK(cudaEventCreateWithFlags(&b.h2d_done, cudaEventDisableTiming));
  CK(cudaEventCreateWithFlags(&b.done, cudaEventDisableTiming));
  CK(cudaEventCreate(&b.ev_start));
  CK(cudaEventCreate(&b.ev_bb0));
  CK(cudaEventCreate(&b.ev_bb1));
  CK(cudaEventCreate(&b.ev_end));
  return RTCC_OK;
}

// Timestamp node inside a captured graph (a plain record only adds a
// dependency during capture).
cudaError_t record_node(cudaEvent_t ev, cudaStream_t st) {
  return cudaEventRecordWithFlags(ev, st, cudaEventRecordExternal);
}

rtcc_status capture_branch_graph(rtcc_ctx* c, int k, const PillarBufs& pb, cudaGraphExec_t* out) {
  Branch& b = c->br[k];
  const bool tl = (c->cfg.flags & RTCC_FLAG_TIMELINE) != 0;
  (void)cudaGetLastError();   // no stale error may leak into the launch checks
  GridGeom gg{c->cfg.x_min, c->cfg.y_min, c->cfg.z_min, c->cfg.z_max, c->cfg.pillar, c->W, c->H};
  CK(cudaStreamBeginCapture(b.st, cudaStreamCaptureModeRelaxed));
  cudaError_t e = cudaSuccess;
  if (tl) e = record_node(b.ev_start, b.st);
  // one memset of the per-frame words, then kernels only, so that the pillar
  // chain and the backbone are programmatic dependent launches of each other
  if (e == cudaSuccess) e = cudaMemsetAsync(b.frame_zero, 0, kFrameZeroBytes, b.st);
  if (e == cudaSuccess) e = launch_pillarise(pb, gg, c->pfn_w, c->pfn_b, c->bf16, c->d_err, b.st);
  if (e == cudaSuccess && tl) e = record_node(b.ev_bb0, b.st);
  if (e == cudaSuccess) e = launch_backbone(*b.bb, c->bf16, b.st);
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

// Two graphs per branch: one for payloads already in the device slot, and
// one whose first kernel reads the payload from the pinned staging buffer
// (over the host link) and copies it into the device slot as it goes, so a
// host payload needs no copy-engine transfer and no cross-stream event.
rtcc_status capture_branch(rtcc_ctx* c, int k) {
  Branch& b = c->br[k];
  RS(capture_branch_graph(c, k, b.pb, &b.exec));
  PillarBufs ph = b.pb;
  ph.src_hdr = reinterpret_cast<const int*>(b.staging);
  ph.src_pts = reinterpret_cast<const float4*>(reinterpret_cast<const uint8_t*>(b.staging) + kHdrBytes);
  ph.dst_hdr = reinterpret_cast<int*>(b.in_dev);
  ph.dst_pts = reinterpret_cast<float4*>(b.in_dev + kHdrBytes);
  return capture_branch_graph(c, k, ph, &b.exec_host);
}

rtcc_status capture_post(rtcc_ctx* c) {
  const bool tl = (c->cfg.flags & RTCC_FLAG_TIMELINE) != 0;
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
  const int bkc = fuse_tc_chunk(c->Cf, c->K);
  const bool use_tc = !fa.attention && bkc > 0;
  FuseTcParams tp{};
  if (use_tc) {
    const int swz = bkc * 2;                    // 128- or 64-byte rows
    for (int k = 0; k < c->K; ++k)
      CK(tmap_2d(&tp.feat[k], c->br[k].feat, c->bf16, (uint64_t)c->Cf, (uint64_t)fa.cells,
                 (uint32_t)bkc, 128u, swz));
    CK(tmap_2d(&tp.wmap, c->head_w16, c->bf16, (uint64_t)c->Cf, 16u, (uint32_t)bkc, 16u, swz));
    tp.present = c->d_present;
    tp.K = c->K;
    tp.C = c->Cf;
    tp.cells = fa.cells;
    tp.bkc = bkc;
    tp.stages = fuse_tc_stages(c->Cf, c->K);
    tp.head_b = c->head_b;
    tp.head_out = c->head_out;
    tp.fused = c->fused;
    tp.keys = c->keys;
    tp.hist0 = c->hist0;
    tp.cls_thresh = c->cfg.cls_thresh;
    tp.anchors = c->cfg.anchors;
    tp.err = c->d_err;
    tp.span = c->fuse_span;
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
  if (e == cudaSuccess) {
    if (use_tc)
      e = launch_fuse_max_head(tp, c->bf16, c->post);
    else
      e = launch_fuse_head(fa, c->bf16, c->post);
  }
  if (e == cudaSuccess && tl) e = record_node(c->ev_fuse1, c->post);
  if (e == cudaSuccess) e = launch_decode(da, c->post);
  if (e == cudaSuccess && c->dec_boxes) e = launch_nms(na, c->post);
  if (e == cudaSuccess && tl) e = record_node(c->ev_post1, c->post);
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
  for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
    Branch& b = c->br[k];
    if (b.st) cudaStreamSynchronize(b.st);
    if (b.exec) cudaGraphExecDestroy(b.exec);
    if (b.exec_host) cudaGraphExecDestroy(b.exec_host);
    for (cudaEvent_t ev : {b.h2d_done, b.done, b.ev_start, b.ev_bb0, b.ev_bb1, b.ev_end})
      if (ev) cudaEventDestroy(ev);
    delete b.bb;
    b.bb = nullptr;
    if (b.st) cudaStreamDestroy(b.st);
  }
  if (c->post) cudaStreamSynchronize(c->post);
  if (c->xfer) cudaStreamSynchronize(c->xfer);
  if (c->post_exec) cudaGraphExecDestroy(c->post_exec);
  for (cudaEvent_t ev : {c->det_ready, c->ev_post0, c->ev_fuse0, c->ev_fuse1, c->ev_post1})
    if (ev) cudaEventDestroy(ev);
  if (c->post) cudaStreamDestroy(c->post);
  if (c->xfer) cudaStreamDestroy(c->xfer);
  for (void* p : c->allocs) cudaFree(p);
  for (void* p : c->host_allocs) cudaFreeHost(p);
  c->allocs.clear();
  c->host_allocs.clear();
}

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
  for (int k = 0; k < c->K; ++k) RS(build_branch(c, k));
  const int cells_f = c->Wf * c->Hf;
  RS(dalloc(c, &c->d_feat_ptrs, RTCC_MAX_AGENTS * sizeof(void*)));
  void* fp[RTCC_MAX_AGENTS] = {};
  for (int k = 0; k < c->K; ++k) fp[k] = c->br[k].feat;
  CK(cudaMemcpy(c->d_feat_ptrs, fp, sizeof(fp), cudaMemcpyHostToDevice));
  RS(dalloc(c, &c->head_out, (size_t)cells_f * 16 * sizeof(float)));
  if (g.flags & RTCC_FLAG_KEEP_FUSED) RS(dalloc(c, &c->fused, (size_t)cells_f * c->Cf * 2));
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
  CK(cudaEventCreateWithFlags(&c->det_ready, cudaEventDisableTiming));
  CK(cudaEventCreate(&c->ev_post0));
  CK(cudaEventCreate(&c->ev_fuse0));
  CK(cudaEventCreate(&c->ev_fuse1));
  CK(cudaEventCreate(&c->ev_post1));
  for (int k = 0; k < c->K; ++k) RS(capture_branch(c, k));
  RS(capture_post(c));
  // warm-up: every graph once on empty payloads (pays first-launch costs)
  for (int k = 0; k < c->K; ++k) CK(cudaGraphLaunch(c->br[k].exec, c->br[k].st));
  for (int k = 0; k < c->K; ++k) CK(cudaGraphLaunch(c->br[k].exec_host, c->br[k].st));
  for (int k = 0; k < c->K; ++k) CK(cudaStreamSynchronize(c->br[k].st));
  CK(cudaGraphLaunch(c->post_exec, c->post));
  CK(cudaStreamSynchronize(c->post));
  int herr = 0;
  CK(cudaMemcpy(&herr, c->d_err, 4, cudaMemcpyDeviceToHost));
  return herr ? RTCC_E_DEVICE : RTCC_OK;
}

// Launch branch k: H2D of its payload on the transfer stream (unless the input
// is resident), an event gating the branch stream, the branch graph, and the
// branch's completion event.  Called with the context mutex held.
rtcc_status launch_branch(rtcc_ctx* c, int k) {
  Branch& b = c->br[k];
  if (!b.pend_resident) {
    // the branch's first kernel reads the payload from the pinned staging
    // buffer and copies it to the device slot (no copy engine, no event)
    const int n = b.pend_n;
    float* pts = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(b.staging) + kHdrBytes);
    if (n > 0 && b.pend_ptr != pts) std::memcpy(pts, b.pend_ptr, (size_t)n * 16);
    *reinterpret_cast<volatile int*>(b.staging) = n;
    std::atomic_thread_fence(std::memory_order_seq_cst);
    CK(cudaGraphLaunch(b.exec_host, b.st));
  } else {
    CK(cudaGraphLaunch(b.exec, b.st));
  }
  CK(cudaEventRecord(b.done, b.st));
  b.launched = true;
  c->ctrl.mark(k, RTCC_RUNNING);
  c->present_dirty = true;
  c->info.t_release_ms[k] = now_ms();
  if (c->info.n_dispatched < RTCC_MAX_AGENTS) c->info.dispatch_order[c->info.n_dispatched++] = k;
  return RTCC_OK;
}

rtcc_status launch_post(rtcc_ctx* c) {
  // the presence flags are set on the device by the branches that ran (their
  // first kernel) and cleared by the decode kernel
  for (int k = 0; k < c->K; ++k)
    if (c->ctrl.present(k)) CK(cudaStreamWaitEvent(c->post, c->br[k].done, 0));
  *c->h_done = 0;                                 // the decode kernel sets it when the boxes are written
  std::atomic_thread_fence(std::memory_order_seq_cst);
  CK(cudaGraphLaunch(c->post_exec, c->post));
  CK(cudaEventRecord(c->det_ready, c->post));
  c->post_launched = true;
  return RTCC_OK;
}

// Dispatch what an event made ready; launch the post-join once every branch
// is resolved.  `t_entry` is the host time the event call began.
rtcc_status after_event(rtcc_ctx* c, const std::vector<int>& released, double t_entry) {
  for (int k : released) RS(launch_branch(c, k));
  if (c->ctrl.join_ready() && !c->post_launched) {
    c->t_last_event = t_entry;
    RS(launch_post(c));
  }
  return RTCC_OK;
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
    CK(cudaMemset(c->d_present, 0, RTCC_MAX_AGENTS * 4));
    c->present_dirty = false;
  }
  c->post_launched = false;
  c->t_last_event = 0.0;
  std::memset(&c->info, 0, sizeof(c->info));
  for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
    c->info.dispatch_order[k] = -1;
    c->info.gpu_backbone_ms[k] = -1.f;
    c->info.gpu_branch_ms[k] = -1.f;
    c->info.t_release_ms[k] = NAN;
    c->br[k].launched = false;
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
      for (int k = 0; k < c->K; ++k)
        if (c->br[k].launched) cudaStreamSynchronize(c->br[k].st);
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
  if (c->cfg.flags & RTCC_FLAG_TIMELINE) {
    for (int k = 0; k < c->K; ++k) {
      Branch& b = c->br[k];
      if (!b.launched) continue;
      float ms = -1.f;
      if (cudaEventElapsedTime(&ms, b.ev_bb0, b.ev_bb1) == cudaSuccess) c->info.gpu_backbone_ms[k] = ms;
      if (cudaEventElapsedTime(&ms, b.ev_start, b.ev_end) == cudaSuccess) c->info.gpu_branch_ms[k] = ms;
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
  return hdr->err ? RTCC_E_DEVICE : RTCC_OK;
}

rtcc_status rtcc_get_frame_info(rtcc_ctx* c, rtcc_frame_info* info) {
  if (!c || !info) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  *info = c->info;
  return RTCC_OK;
}

rtcc_status rtcc_get_layer_spans(rtcc_ctx* c, int32_t agent, float* start_ms, float* end_ms,
                                 int32_t cap, int32_t* n_out) {
  if (!c) return RTCC_E_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  if (agent < 0 || agent >= c->K) return RTCC_E_AGENT;
  Branch& b = c->br[agent];
  if (!b.stamps) return RTCC_E_STATE;
  const int n = (int)b.layers.size();
  if (n_out) *n_out = n;
  if (!start_ms && !end_ms) return RTCC_OK;
  CK(cudaStreamSynchronize(b.st));
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
    if (st == RTCC_RUNNING && cudaEventQuery(c->br[agent].done) == cudaSuccess)
      c->ctrl.mark(agent, RTCC_FINISHED);
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
    if (!c->fused) return RTCC_E_STATE;
    CK(cudaStreamSynchronize(c->post));
    src = c->fused;
    n = (size_t)c->Wf * c->Hf * c->Cf;
  } else {
    if (agent < 0 || agent >= c->K) return RTCC_E_AGENT;
    Branch& b = c->br[agent];
    CK(cudaStreamSynchronize(b.st));
    if (which == 0) {
      src = b.pb.image;
      n = (size_t)c->W * c->H * c->Cp;
    } else if (which >= 1 && which <= c->cfg.n_blocks) {
      src = b.block_out[which - 1];
      n = (size_t)b.block_w[which - 1] * b.block_h[which - 1] * c->cfg.block_ch[which - 1];
    } else if (which == 8) {
      src = b.feat;
      n = (size_t)c->Wf * c->Hf * c->Cf;
    } else if (which >= 16 && which - 16 < (int)b.layer_out.size() &&
               (c->cfg.flags & RTCC_FLAG_KEEP_LAYERS)) {
      src = b.layer_out[which - 16];
      n = b.layer_elems[which - 16];
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
  // pillar chain + backbone per branch; fusion, decode (and NMS)
  return n_present * (5 + 1) + 2 + (c->dec_boxes ? 1 : 0);
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

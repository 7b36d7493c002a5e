/*
 * rtcc.h -- C ABI of the release-triggered communication-computation coupling
 * (RTCC) runtime for multi-agent cooperative perception on one GB300 GPU.
 *
 * The runtime owns a fork-join intermediate-fusion detector: K per-agent
 * encoder branches E_k (pillarise -> pillar feature net -> BEV scatter -> 3x3
 * conv backbone -> deconv neck) and one shared post-join subgraph (cross-agent
 * fusion -> 1x1 head -> anchor decode).  Sec. III-B of the paper defines this
 * DAG; Sec. IV-C..F define the release path implemented here:
 *
 *   rtcc_payload_complete(k)  -- the completion event e_k = Complete(k, a_k)
 *                                (Eq. 17).  It is validated (Sec. IV-C), the
 *                                branch moves WAITING -> RELEASED (Eq. 18) with
 *                                release time r_k = a_k, its input is copied
 *                                host -> device on a transfer stream, a CUDA
 *                                event gates the branch's compute stream, and
 *                                the branch's CUDA graph is launched into the
 *                                agent-indexed feature slot k (Sec. IV-F).
 *   last branch resolved      -- the post-join graph waits on every branch's
 *                                event and runs fusion, head and decode.
 *   RTCC_MODE_BARRIER         -- the baseline of Sec. V: every branch is
 *                                released only at the last arrival
 *                                A = max_k a_k, in agent-index order.
 *
 * Both modes run the same kernels on the same inputs into the same slots, so
 * their outputs are bit-identical (Sec. III-C, last paragraph; Sec. V-F).
 *
 * Conventions (all entry points):
 *  - Errors are returned as rtcc_status; no entry point aborts the process or
 *    traps the GPU.  rtcc_status_str() names a code.
 *  - Pointers named host_* are host memory owned by the caller; the library
 *    never keeps them past the call except where stated.  Pointers named d_*
 *    are device memory owned by the caller.
 *  - A context is opaque and owned by the library.  Calls on one context are
 *    serialised by an internal mutex, so different host threads may report
 *    completions of different agents.  rtcc_wait_detection releases the mutex
 *    while it waits.
 *  - Times passed in (t_ms, t0_ms) are the caller's frame timebase in ms; they
 *    decide validation and release order.  Times returned (t_ready_ms and
 *    rtcc_frame_info) are the library's steady host clock, rtcc_now_ms().
 *  - Layouts: points are float32 [n][4] = (x, y, z, intensity); BEV tensors
 *    are row-major [rows][cols][channels] (NHWC, N = 1); the head output is
 *    float32 [H'][W'][8A].
 */
#ifndef RTCC_H
#define RTCC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define RTCC_MAX_AGENTS 8
#define RTCC_MAX_BLOCKS 3

typedef struct rtcc_ctx rtcc_ctx;

typedef enum {
  RTCC_OK = 0,
  RTCC_E_ARG = 1,         /* null pointer, bad size or unsupported config      */
  RTCC_E_AGENT = 2,       /* agent index outside [0, n_agents)                 */
  RTCC_E_DUPLICATE = 3,   /* a second event for an agent within one frame      */
  RTCC_E_PREMATURE = 4,   /* no frame begun, or event time before the frame t0 */
  RTCC_E_MALFORMED = 5,   /* payload pointer/size inconsistent (n < 0, n > cap,
                             null pointer with n > 0)                          */
  RTCC_E_STATE = 6,       /* call not allowed in the current frame state       */
  RTCC_E_TIMEOUT = 7,     /* host-side wait limit passed; the GPU is untouched */
  RTCC_E_INFEASIBLE = 8,  /* frame aborted with undelivered branches: no output
                             (Sec. IV-C, last sentence)                        */
  RTCC_E_CUDA = 9,        /* a CUDA runtime call failed                        */
  RTCC_E_NOMEM = 10,      /* device or pinned allocation failed                */
  RTCC_E_DEVICE = 11      /* a kernel gave up a bounded wait and flagged it    */
} rtcc_status;

typedef enum { RTCC_MODE_RTCC = 0, RTCC_MODE_BARRIER = 1 } rtcc_mode;
typedef enum { RTCC_FUSE_MAX = 0, RTCC_FUSE_ATTN = 1 } rtcc_fusion;
typedef enum { RTCC_FP16 = 0, RTCC_BF16 = 1 } rtcc_dtype;

/* Branch lifecycle, Eq. 18 (ABSENT: declared missing, masked from fusion). */
typedef enum {
  RTCC_WAITING = 0, RTCC_RELEASED = 1, RTCC_RUNNING = 2, RTCC_FINISHED = 3,
  RTCC_ABSENT = 4
} rtcc_branch_state;

/* config.flags */
#define RTCC_FLAG_TIMELINE    1  /* record CUDA events around the backbone and
                                    the fusion kernel of every frame           */
#define RTCC_FLAG_KEEP_FUSED  2  /* also store the fused BEV map (parity)      */
#define RTCC_FLAG_KEEP_LAYERS 4  /* give every conv layer its own output buffer
                                    so each can be read back (parity)         */
#define RTCC_FLAG_LAYER_TIMES 8  /* record the GPU times at which the backbone
                                    kernel starts and ends each conv/deconv
                                    layer                                     */
#define RTCC_FLAG_NO_CLUSTERS 16 /* launch the backbone without thread-block
                                    clusters: split-K slices then reduce
                                    through global memory instead of
                                    distributed shared memory (same results)  */
#define RTCC_FLAG_SHORT_WAITS 32 /* bounded device waits give up after about
                                    10 ms instead of about 1 s, and
                                    rtcc_test_unreachable_wait is enabled
                                    (tests of the wait limit)                  */
#define RTCC_FLAG_NO_BATCH    64 /* every branch runs its own backbone launch,
                                    also when branches are released together
                                    (same results; for comparisons)           */
#define RTCC_FLAG_H2D_COPY   128 /* host payloads reach the device slot by a
                                    copy-engine transfer on a transfer stream
                                    whose event gates the branch stream, instead
                                    of the branch's first kernel reading the
                                    pinned staging buffer (same results)       */
#define RTCC_FLAG_MULTISCALE 256 /* the fusion placement of Sec. IV-A (needs a
                                    neck): each branch ends at its backbone
                                    blocks; after the join, every block's map
                                    is fused across the present agents (the
                                    configured max or ego-query attention, at
                                    the block's channel count), the neck
                                    (deconvs + concatenation) runs once on the
                                    fused maps, then the head.  Without it the
                                    branches run the neck and the 384-channel
                                    maps are fused                            */

/*
 * Network and workload description.  Supported: 1 <= n_agents <= 8;
 * grid_w, grid_h >= 1; max_pts in [1, 32]; pfn_ch in {32, 64}; n_blocks in
 * [1, 3]; block_ch in {32, 64, 128, 256}; block_stride in {1, 2} (inputs of a
 * stride-2 block must have even sizes); up_stride[b] in {1, 2, 4} for every
 * block, or all 0 for "no neck" (then n_blocks == 1 and the features are the
 * block's output); up_ch == 128 when a neck exists; anchors == 2;
 * 1 <= max_boxes <= 512; 0 <= nms_iou <= 1.
 */
typedef struct {
  int32_t n_agents;
  int32_t grid_w, grid_h;           /* pillars along x and y                 */
  float x_min, y_min, z_min;        /* metres; half-open box [min, max)      */
  float x_max, y_max, z_max;
  float pillar;                     /* pillar edge length v                  */
  int32_t max_pillars;              /* P_max                                 */
  int32_t max_pts;                  /* N_max, points kept per pillar         */
  int32_t pfn_ch;                   /* C_p                                   */
  int32_t n_blocks;
  int32_t block_layers[RTCC_MAX_BLOCKS];
  int32_t block_ch[RTCC_MAX_BLOCKS];
  int32_t block_stride[RTCC_MAX_BLOCKS];
  int32_t up_stride[RTCC_MAX_BLOCKS];
  int32_t up_ch;
  int32_t fusion;                   /* rtcc_fusion                           */
  int32_t anchors;                  /* A                                     */
  int32_t dtype;                    /* rtcc_dtype: storage of weights and
                                       activations; accumulation is fp32     */
  int32_t max_points;               /* payload capacity, points per agent    */
  int32_t max_boxes;                /* top-K after thresholding              */
  float cls_thresh;                 /* keep anchors whose class logit is
                                       >= cls_thresh                         */
  float nms_iou;                    /* rotated BEV NMS after the top-K: a box
                                       is dropped when its IoU with a kept
                                       higher-ranked box exceeds nms_iou;
                                       0 = no NMS; 0 <= nms_iou <= 1         */
  int32_t flags;                    /* RTCC_FLAG_*                           */
} rtcc_model_config;

/* One detection: centre, size, heading, score = sigmoid(logit), and the anchor
 * index (iy * W' + ix) * A + a it was decoded from. */
typedef struct {
  float x, y, z, l, w, h, yaw, score;
  int32_t anchor;
} rtcc_box;

/* Host timestamps (rtcc_now_ms) and GPU spans of the most recent frame. */
typedef struct {
  double t_last_event_ms;           /* entry of the call that resolved the
                                       last branch (start of the tail)        */
  double t_ready_ms;                /* wait_detection saw the output ready    */
  double t_release_ms[RTCC_MAX_AGENTS];   /* host time each branch launched   */
  float gpu_backbone_ms[RTCC_MAX_AGENTS]; /* conv/deconv span per branch; -1
                                             without RTCC_FLAG_TIMELINE        */
  float gpu_branch_ms[RTCC_MAX_AGENTS];   /* whole branch incl. pillarise     */
  float gpu_fusion_ms;              /* fusion+head kernel                     */
  float gpu_post_ms;                /* whole post-join graph                  */
  int32_t dispatch_order[RTCC_MAX_AGENTS];  /* agents in launch order, -1 pad */
  int32_t n_dispatched;
  float gpu_fusion_kernel_ms;       /* the fusion+head kernel's own span on the
                                       GPU global timer (block 0 past its
                                       dependency wait to the last block's
                                       end); -1 without RTCC_FLAG_TIMELINE    */
  float gpu_pfn_kernel_ms[RTCC_MAX_AGENTS];  /* each branch's PFN kernel span, the
                                                same way; -1 without the flag  */
  int32_t n_backbone_launches;      /* backbone launches of the frame: agents
                                       released together share one            */
  int32_t backbone_batch[RTCC_MAX_AGENTS];  /* agents in each launch, in launch
                                               order; 0 pad                    */
  float gpu_launch_ms[RTCC_MAX_AGENTS];     /* each launch's backbone span (CUDA
                                               events); -1 without
                                               RTCC_FLAG_TIMELINE              */
} rtcc_frame_info;

/* ------------------------------------------------------------------------ */
/* Context lifecycle (offline stage, Sec. IV-A)                             */
/* ------------------------------------------------------------------------ */

/*
 * Build a context on the current CUDA device.  `weights` is the fp32 master
 * blob (little-endian), `n_floats` its length; order: PFN W [C_p][9], b;
 * every conv of every block W [Co][Ci][3][3], b; every deconv W [Ci][Co][s][s],
 * b; head W [8A][C_feat], b.  The library rounds each tensor once to the
 * storage dtype and repacks it for its kernels; the caller's blob is not kept.
 * Allocates all device memory, pinned staging buffers, streams, events and
 * the K branch graphs plus the post-join graph, and (unless
 * RTCC_FLAG_NO_BATCH) starts one host thread, the dispatcher of batched
 * backbone launches (see rtcc_payload_complete), which rtcc_destroy joins.
 * RTCC_E_ARG for an unsupported config or a blob of the wrong length.  A
 * grid whose x or y bounds (x_min, x_min + grid_w * pillar, and the same in
 * y) lie more than 2^20 pillar edges from 0, or whose z bounds lie more than
 * 2^20 times (z_max - z_min) from 0, is unsupported: the PFN forms the means
 * as fixed-point sums of the points' offsets from their pillar, which needs
 * float32 to place each point within one edge of its pillar's centre.
 */
rtcc_status rtcc_init(const rtcc_model_config* cfg, const float* weights,
                      size_t n_floats, struct rtcc_ctx** out);

/* Free everything the context owns; waits for its GPU work.  NULL is a no-op. */
void rtcc_destroy(struct rtcc_ctx* ctx);

/* Select RTCC or Barrier release; only between frames (else RTCC_E_STATE). */
rtcc_status rtcc_set_mode(struct rtcc_ctx* ctx, rtcc_mode mode);

/*
 * Library-owned pinned staging buffer of `agent` (capacity *cap_points
 * points).  A payload written here and passed to rtcc_payload_complete is
 * copied to the device without an extra host copy.  Valid until destroy.
 */
rtcc_status rtcc_staging_buffer(struct rtcc_ctx* ctx, int32_t agent,
                                float** host_points, int32_t* cap_points);

/*
 * Copy a payload into agent's device input slot now (blocking), for the
 * resident-input mode: a later rtcc_payload_resident releases the branch with
 * no host->device copy on the release path.  Only between frames.
 */
rtcc_status rtcc_stage_resident(struct rtcc_ctx* ctx, int32_t agent,
                                const float* host_points, int32_t n_points);

/* ------------------------------------------------------------------------ */
/* Online stage (Sec. IV-B..F, Algorithm 1)                                 */
/* ------------------------------------------------------------------------ */

/* Start a frame whose timebase begins at t0_ms; every branch is WAITING.
 * RTCC_E_STATE while a previous frame is still open (not yet waited on). */
rtcc_status rtcc_frame_begin(struct rtcc_ctx* ctx, uint64_t frame_id, double t0_ms);

/*
 * Completion event of agent's uplink payload at time t_ms (Eq. 17).
 * Validation (Sec. IV-C): RTCC_E_PREMATURE without an open frame or with
 * t_ms < t0; RTCC_E_AGENT for a bad index; RTCC_E_DUPLICATE if the branch is
 * no longer WAITING; RTCC_E_MALFORMED for n_points < 0, n_points > capacity
 * or host_points == NULL with n_points > 0.  n_points == 0 is a valid empty
 * payload.  On success in RTCC mode the branch is launched before return; in
 * Barrier mode it is held until every branch is resolved.  host_points must
 * stay unchanged until rtcc_wait_detection returns for this frame; when it is
 * the staging buffer no host copy is made.
 *
 * Launches (Sec. III-B's single encoder stream, kept busy): a released branch
 * starts its pillar chain before return.  Unless it resolves the last branch,
 * its backbone is held: the dispatcher thread launches one backbone over every
 * held branch once the backbone in flight (if any) has ended and no release
 * has come for 40 us, so completions reported close together share a launch.
 * Branches released by one event (Barrier at A) share one launch.  The event
 * that resolves the last branch launches at once: alone onto a free GPU as
 * the branch's own graph (pillar chain and backbone), else together with
 * whatever is held.  Every branch writes its own slot and its result does not
 * depend on the launch that ran it, so RTCC and Barrier outputs stay
 * byte-identical.
 */
rtcc_status rtcc_payload_complete(struct rtcc_ctx* ctx, int32_t agent,
                                  const float* host_points, int32_t n_points,
                                  double t_ms);

/* Same as rtcc_payload_complete for the payload placed by
 * rtcc_stage_resident (no host->device copy on the release path). */
rtcc_status rtcc_payload_resident(struct rtcc_ctx* ctx, int32_t agent, double t_ms);

/*
 * Declare agent absent for this frame: its branch never runs and fusion masks
 * it out.  Same validation as rtcc_payload_complete.  RTCC_E_ARG for the ego
 * (agent 0) under attention fusion, or when it would leave no agent present.
 */
rtcc_status rtcc_payload_absent(struct rtcc_ctx* ctx, int32_t agent, double t_ms);

/*
 * The communication horizon expired with branches still WAITING: the frame is
 * infeasible, the post-join subgraph is withheld (Sec. IV-C, last sentence)
 * and the next rtcc_wait_detection returns RTCC_E_INFEASIBLE.  Branches
 * already launched still finish on the GPU.
 */
rtcc_status rtcc_frame_abort(struct rtcc_ctx* ctx);

/*
 * Wait (host-side, up to timeout_ms; < 0 = no limit) until the frame's
 * detections are ready -- decoded, thresholded, cut to max_boxes and, with
 * nms_iou > 0, passed through rotated BEV NMS: the endpoint of T^det
 * (Sec. V-A-3) -- then copy up to `cap` boxes (score-descending) to
 * out, their number to *n_out and the ready time to *t_ready_ms (any of the
 * three may be NULL).  Closes the frame.  RTCC_E_TIMEOUT leaves the frame
 * open (call again); RTCC_E_INFEASIBLE after rtcc_frame_abort;
 * RTCC_E_STATE if the frame is still missing branches; RTCC_E_DEVICE if a
 * kernel flagged an expired bounded wait.
 */
rtcc_status rtcc_wait_detection(struct rtcc_ctx* ctx, int32_t timeout_ms,
                                rtcc_box* out, int32_t cap, int32_t* n_out,
                                double* t_ready_ms);

/* Timestamps and GPU spans of the last closed frame. */
rtcc_status rtcc_get_frame_info(struct rtcc_ctx* ctx, rtcc_frame_info* info);

/* Per-layer GPU times (ms) of `agent`'s conv and deconv layers in the last
 * closed frame, in order (13 convs then 3 deconvs for the PointPillars
 * backbone): for each layer, from the moment the backbone kernel's CTA that
 * holds its first item has seen every input item stored, to the moment its
 * last output item is counted.  Layers may overlap (the neck deconvs of the
 * first two blocks run beside the deeper blocks), so the times do not add up
 * to the backbone's time.  Needs RTCC_FLAG_LAYER_TIMES.  *n_out receives the
 * layer count; entries beyond it are not written; -1 where a stamp is
 * missing.  RTCC_E_STATE without the flag. */
rtcc_status rtcc_get_layer_times(struct rtcc_ctx* ctx, int32_t agent, float* host_ms,
                                 int32_t cap, int32_t* n_out);

/* The same stamps as start and end offsets (ms) from the earliest layer start
 * of the backbone launch, so that overlapping layers can be laid out on one
 * time axis.  Either array may be NULL. */
rtcc_status rtcc_get_layer_spans(struct rtcc_ctx* ctx, int32_t agent, float* start_ms,
                                 float* end_ms, int32_t cap, int32_t* n_out);

/* State z_k of a branch in the open (or last) frame, and its release time
 * r_k in the caller's timebase (NaN while WAITING). */
rtcc_status rtcc_get_branch_state(struct rtcc_ctx* ctx, int32_t agent,
                              int32_t* state, double* release_ms);

/* ------------------------------------------------------------------------ */
/* Read-back of the last closed frame (parity and bit-identity checks)      */
/* All copy device -> host and block; `cap` counts elements of the output.  */
/* ------------------------------------------------------------------------ */

/* Head output float32 [H'][W'][8A]. */
rtcc_status rtcc_get_head(struct rtcc_ctx* ctx, float* host_out, size_t cap);

/* The decode's top-K boxes before NMS (rank order: score descending, anchor
 * index ascending), up to `cap` of them; *n_out = their count.  Without NMS
 * (nms_iou == 0) these are the frame's result boxes. */
rtcc_status rtcc_get_decoded(struct rtcc_ctx* ctx, rtcc_box* host_out, int32_t cap,
                             int32_t* n_out);

/* Pillarisation of `agent`: cell2pillar int32 [H*W] (-1 = empty),
 * pillar_cell int32 [P_max] (-1 pad), count int32 [P_max] (kept points), and
 * stats int32 [8] = {n_points, n_in_range, n_pillars, n_kept, drop_range,
 * drop_pcap, drop_ncap, 0}.  Any output pointer may be NULL. */
rtcc_status rtcc_get_pillars(struct rtcc_ctx* ctx, int32_t agent,
                             int32_t* host_cell2pillar, int32_t* host_pillar_cell,
                             int32_t* host_count, int32_t* host_stats);

/* Raw 16-bit (fp16 or bf16 per config) tensors of `agent`:
 *   which = 0: BEV pseudo-image [H][W][C_p]
 *   which = 1..n_blocks: output of block which-1 [H_b][W_b][C_b]
 *   which = 8: feature slot [H'][W'][C_feat]
 *   which = 9: fused map [H'][W'][C_feat] (agent ignored; needs
 *              RTCC_FLAG_KEEP_FUSED, or with RTCC_FLAG_MULTISCALE the neck's
 *              output on the fused blocks)
 *   which = 10..9+n_blocks: RTCC_FLAG_MULTISCALE: fused map of block
 *              which-10 [H_b][W_b][C_b] (agent ignored)
 *   which = 16 + i: output of the i-th 3x3 conv of the branch, counting
 *              through all blocks (needs RTCC_FLAG_KEEP_LAYERS)
 * *n_elems receives the tensor's element count. */
rtcc_status rtcc_get_tensor(struct rtcc_ctx* ctx, int32_t agent, int32_t which,
                            uint16_t* host_out, size_t cap, size_t* n_elems);

/* ------------------------------------------------------------------------ */
/* Allocation-free pillarisation (no counterpart in the paper)              */
/* ------------------------------------------------------------------------ */

/*
 * The pillarise -> PFN -> scatter pass of one branch, for callers that cannot
 * allocate device memory where they need it: code running while a stream is
 * being captured into a CUDA graph (cudaMalloc cannot be captured), plugin
 * hosts that own all device memory and offer no allocator, and latency-bound
 * loops that must not risk the device synchronisation an allocation can
 * trigger.  This call allocates nothing: its scratch is one fixed array in
 * device memory that the library reserves on every GPU that loads it (about
 * 11.8 MB, kept until the process exits).  The array bounds the sizes:
 * grid_w * grid_h <= 65536 cells, n_points <= 131072, max_pillars <= 16384,
 * pfn_ch in {32, 64}, max_pts <= 32; larger requests, and grid bounds that
 * rtcc_init rejects, return RTCC_E_ARG.
 *
 * Uses from cfg: grid_w/h, x_min, y_min, z_min, z_max, pillar, max_pillars,
 * max_pts, pfn_ch, dtype.  Inputs (device, caller-owned): d_points float32
 * [n_points][4]; d_pfn_w float32 [pfn_ch][9] and d_pfn_b float32 [pfn_ch]
 * with the values the kernels should use (rtcc_init rounds them to the storage
 * type first).  Outputs (device, caller-owned): d_cell2pillar int32 [H*W],
 * d_pillar_cell and d_count int32 [max_pillars] (entries >= n_pillars are left
 * untouched), d_stats int32 [8] = {n, n_in_range, n_pillars, n_kept, 0, 0,
 * dropped by the per-pillar cap, points of kept pillars before that cap},
 * d_image 16-bit [H][W][pfn_ch].  d_points and d_image must be 16-byte
 * aligned and the other pointers 4-byte aligned, else RTCC_E_ARG.  Work is
 * enqueued on `stream` (a cudaStream_t; NULL = the default stream) and the
 * call returns without waiting.  RTCC_E_CUDA reports a failed launch of this
 * call's own kernels; an error left by the caller's earlier work is neither
 * reported nor cleared.
 *
 * The first call on a device looks up the array's device address; make that
 * first call outside any stream capture.  Every call shares the array and
 * clears what must start at zero before use, so calls that overlap on the GPU
 * race with each other: serialise them (one stream, or events).
 */
rtcc_status rtcc_pillarise_noalloc(const rtcc_model_config* cfg, const float* d_points,
                                   int32_t n_points, const float* d_pfn_w,
                                   const float* d_pfn_b, int32_t* d_cell2pillar,
                                   int32_t* d_pillar_cell, int32_t* d_count,
                                   int32_t* d_stats, void* d_image, void* stream);

/* ------------------------------------------------------------------------ */
/* Release controller alone (host only; no GPU needed)                      */
/* ------------------------------------------------------------------------ */

/*
 * The validation, state machine (Eq. 18) and ready queue ordered by
 * (r_k, k) (Sec. IV-C/D) that rtcc_payload_complete runs, exposed without an
 * executor.  Each event call returns, in *released / *n_released, the agents
 * that become dispatchable by that event, in dispatch order: under RTCC the
 * completing agent; under Barrier nothing until the last branch resolves,
 * then every present agent in index order.  `released` must hold
 * RTCC_MAX_AGENTS entries.
 */
typedef struct rtcc_controller rtcc_controller;
rtcc_status rtcc_ctrl_create(int32_t n_agents, int32_t cap_points, int32_t attn_ego,
                             rtcc_controller** out);
void rtcc_ctrl_destroy(rtcc_controller* c);
rtcc_status rtcc_ctrl_set_mode(rtcc_controller* c, rtcc_mode mode);
rtcc_status rtcc_ctrl_begin(rtcc_controller* c, uint64_t frame_id, double t0_ms);
rtcc_status rtcc_ctrl_complete(rtcc_controller* c, int32_t agent, const void* payload,
                               int32_t n_points, double t_ms,
                               int32_t* released, int32_t* n_released);
rtcc_status rtcc_ctrl_absent(rtcc_controller* c, int32_t agent, double t_ms,
                             int32_t* released, int32_t* n_released);
/* Executor feedback: RELEASED -> RUNNING -> FINISHED. */
rtcc_status rtcc_ctrl_mark(rtcc_controller* c, int32_t agent, int32_t state);
rtcc_status rtcc_ctrl_abort(rtcc_controller* c);
/* 1 when every branch is resolved and at least one is present (the post-join
 * may be launched), else 0. */
int32_t rtcc_ctrl_join_ready(const rtcc_controller* c);
rtcc_status rtcc_ctrl_state(const rtcc_controller* c, int32_t agent,
                            int32_t* state, double* release_ms);
/* Close the frame (after its output was consumed or it was aborted). */
rtcc_status rtcc_ctrl_end(rtcc_controller* c);

/* ------------------------------------------------------------------------ */
/* Slot-level uplink (host only; the source of completion events)           */
/* ------------------------------------------------------------------------ */

typedef enum {
  RTCC_SCHED_MAXRATE = 0,     /* RB to the eligible agent of highest rate      */
  RTCC_SCHED_ROUNDROBIN = 1,  /* RB to the first eligible agent after the one
                                 served last, in cyclic index order           */
  RTCC_SCHED_MAXWEIGHT = 2,   /* highest queue x rate                          */
  RTCC_SCHED_EARLIEST = 3,    /* least time to empty the queue at this rate    */
  RTCC_SCHED_WEIGHTED = 4     /* highest weight_k x rate (DAG rank, task weight) */
} rtcc_sched;

/*
 * Completion slots of one frame's uploads over a slot-level OFDMA uplink
 * (Sec. III-A, Eqs. 1-5).  Each slot t = 1..t_max: agents with bits left and
 * t >= first_slot[k] are eligible; each of the n_rb resource blocks goes to
 * one eligible agent by `policy` (ties to the smaller index); agent k then
 * sends slot_s x rate bits on each of its RBs; completion_slot[k] is the slot
 * in which its queue reached zero (0 if not within t_max).  Inputs (host,
 * caller-owned): payload_bits[n_agents], first_slot[n_agents] (1-based),
 * rates float64 [t_max][n_agents][n_rb] in bit/s, weight[n_agents] for
 * RTCC_SCHED_WEIGHTED (else unused, may be NULL).  *n_slots_used (optional)
 * receives the last slot simulated.  RTCC_E_ARG for bad sizes or pointers.
 * Deterministic: the same rates give the same slots.
 */
rtcc_status rtcc_uplink_simulate(int32_t n_agents, int32_t n_rb, int32_t t_max,
                                 const double* payload_bits, const int32_t* first_slot,
                                 const double* rates, double slot_s, int32_t policy,
                                 const double* weight, int32_t* completion_slot,
                                 int32_t* n_slots_used);

/* ------------------------------------------------------------------------ */
/* Backbone tile plan (host only; no counterpart in the paper)              */
/* ------------------------------------------------------------------------ */

/* How one 3x3 conv layer of the backbone is cut into work items. */
typedef struct {
  int32_t splits;       /* K slices per tile (split-K); fixed for every batch
                           size, since they decide the fp32 summation order  */
  int32_t bn;           /* output channels per item (32, 64 or 128)          */
  int32_t tall;         /* 1: tiles of 8 x 32 pixels (two 128-row MMAs per
                           weight box), else 8 x 16 (or 16 x 8 when wide)   */
  int32_t transposed;   /* 1: the tiles' 8-pixel side runs along the image's
                           rows (H) instead of W                            */
  int32_t wide;         /* 1: tiles of 16 x 8 pixels (stride-2 and other
                           layers that load one box per tap)                */
  int32_t m_tiles;      /* pixel tiles covering one agent's output          */
  int32_t items;        /* work items of the launch:
                           n_batch x m_tiles x (cout / bn) x splits         */
} rtcc_conv_plan;

/*
 * The tile choice rtcc_init makes for one 3x3 conv layer (pad 1) of a
 * backbone launch over n_batch agents on `grid` CTAs: kind 0 = stride 1,
 * 1 = stride 2; cin, cout its channels; out_w x out_h its output.  The K
 * slices come from the one-agent cost model, the N tile and tile shape from
 * the cost model at n_batch (rounds of items over the grid x k-blocks per
 * item x the k-block's MMA time).  Pure host arithmetic: no device, no
 * context.  RTCC_E_ARG unless kind is 0 or 1, cin is a power of two in
 * 32..256, cout is a multiple of 32 in 32..256, the extents and grid are
 * positive and 1 <= n_batch <= RTCC_MAX_AGENTS; `out` is caller-owned.
 */
rtcc_status rtcc_plan_conv(int32_t kind, int32_t cin, int32_t cout, int32_t out_w, int32_t out_h,
                           int32_t grid, int32_t n_batch, rtcc_conv_plan* out);

/* ------------------------------------------------------------------------ */
/* Misc                                                                     */
/* ------------------------------------------------------------------------ */

const char* rtcc_status_str(rtcc_status s);
/* Library steady clock in milliseconds. */
double rtcc_now_ms(void);
/* Number of kernel launches of the most recent frame (pillar chains, backbone
 * launches, post-join) for the given number of present agents; before any
 * frame, with one backbone launch per branch. */
int32_t rtcc_kernels_per_frame(struct rtcc_ctx* ctx, int32_t n_present);

/*
 * Test hook for the device-side wait limit (no counterpart in the paper): each
 * backbone launch of the next frame waits, in its first layer that depends on
 * another, for one more finished work item than that layer has.  The wait runs
 * out after the context's limit (use RTCC_FLAG_SHORT_WAITS: about 10 ms), the
 * kernel sets its error word and winds down without trapping, and
 * rtcc_wait_detection returns RTCC_E_DEVICE; it then clears the error state so
 * the next frame runs normally.  Only between frames; RTCC_E_STATE on a
 * context without RTCC_FLAG_SHORT_WAITS.
 */
rtcc_status rtcc_test_unreachable_wait(struct rtcc_ctx* ctx);

/*
 * Rotated BEV NMS of n <= 512 boxes already in rank order (the frame's own
 * post-join step, run on the caller's boxes on the current device): a box is
 * dropped when its IoU with a kept earlier box exceeds iou (0 <= iou <= 1).
 * Writes the kept boxes in order to host_out (room for n) and their number to
 * *n_out.  Boxes are rectangles in x-y: centre (x, y), length l along
 * (cos yaw, sin yaw), width w across it; z, h and score are carried along.
 * Synchronous; allocates and frees its own device scratch.
 */
rtcc_status rtcc_nms(const rtcc_box* host_in, int32_t n, float iou, rtcc_box* host_out,
                     int32_t* n_out);

#ifdef __cplusplus
}
#endif

#endif /* RTCC_H */

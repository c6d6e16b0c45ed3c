/*
 * mafat.h -- C ABI of a GB300 (sm_103a) implementation of fused-tile execution
 * of CNN layer groups, after MAFAT: Memory-Aware Fusing and Tiling of Neural
 * Networks for Accelerated Edge Inference (Farley & Gerstlauer, arXiv
 * 2107.06960).
 *
 * The method (Sec. 3-4): a stack of n convolution / max-pool layers is cut into
 * at most two layer groups (group 1 = layers 0..cut-1, group 2 = cut..n-1).
 * The last-layer output of each group is split into an even N x M grid of
 * tiles; every tile's input region (with the overlap, or halo, its receptive
 * field needs) is found by walking the layers of the group backwards, and the
 * tile runs all layers of its group as one fused unit.  The group-1 tiles are
 * merged into the full cut tensor, which group 2 re-tiles.  Sec. 4.1-4.2 add a
 * memory predictor (Algorithm 1) and a configuration search (Algorithm 2).
 *
 * Conventions shared by every call:
 *  - Every call returns a mafat_status; nothing aborts, exits or throws.  On
 *    failure mafat_last_error() returns a message for the calling thread.
 *  - Handles are created and destroyed only by this library.
 *  - Layers are numbered from 0.  A "cut" is the index of the first layer of
 *    group 2 (the paper's cut); cut <= 0 or cut >= n means a single group.
 *  - Rectangles are int32_t[4] = {y0, y1, x0, x1}, half-open, in the
 *    coordinates of the feature map they live on.
 *  - A grid N x M has N tiles along rows (height) and M along columns.
 *  - Streams are passed as void* holding a cudaStream_t (NULL = legacy default).
 *  - Device pointers must be 16-byte aligned and must not alias each other.
 *
 * Supported layers: 3x3 / stride 1 / pad 1 and 1x1 / stride 1 / pad 0
 * convolutions with folded batch-norm (per-channel scale and bias) followed by
 * leaky ReLU with slope 0.1, and 2x2 / stride 2 max-pool layers that directly
 * follow a convolution of the same group (they are fused into it).  Output
 * channel counts must be multiples of 8; input channel counts above 8 must be
 * multiples of 16; a 1x1 convolution needs at least 9 input channels.
 */
#ifndef MAFAT_H
#define MAFAT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    MAFAT_OK = 0,
    MAFAT_EINVAL = 1,        /* bad argument (null pointer, bad size, misaligned pointer) */
    MAFAT_EUNSUPPORTED = 2,  /* valid request this library does not implement */
    MAFAT_ENOMEM = 3,        /* host or device allocation failed */
    MAFAT_ECUDA = 4,         /* a CUDA runtime call failed */
    MAFAT_ETIMEOUT = 5,      /* a bounded device-side wait on another tile ran out */
    MAFAT_ENOFIT = 6,        /* a plan's per-tile working set cannot be scheduled */
    MAFAT_EDEVICE = 7        /* a bounded device-side pipeline wait ran out (internal error) */
} mafat_status;

typedef enum { MAFAT_CONV = 0, MAFAT_MAXPOOL = 1 } mafat_layer_type;

/* Most layer groups a plan may have (the paper uses one or two). */
#define MAFAT_MAX_GROUPS 4

/* Arithmetic of a plan.  BF16: bf16 activations and weights, fp32 accumulation
 * on the tensor cores (tcgen05), every layer output rounded to bf16.  FP32: the
 * same fused tiling computed in fp32 on the CUDA cores (a check mode). */
typedef enum { MAFAT_BF16 = 0, MAFAT_FP32 = 1 } mafat_dtype;

/* One layer of the network description (the W, H, F, S vectors of Sec. 4.1 and
 * Algorithm 2: filter size k = F_l, stride = S_l; W_l, H_l and channel counts
 * are inferred).  `filters` is the output channel count of a convolution and is
 * ignored for a max-pool. */
typedef struct {
    int32_t type;     /* mafat_layer_type */
    int32_t k;
    int32_t stride;
    int32_t pad;
    int32_t filters;
} mafat_layer_desc;

typedef struct mafat_net_s mafat_net_t;
typedef struct mafat_plan_s mafat_plan_t;

/* Optional knobs of mafat_plan_ex.  Zero-initialise and set struct_size. */
typedef struct {
    int32_t struct_size;        /* sizeof(mafat_plan_options) */
    int32_t ring_slots;         /* tiles whose intermediate buffers may be live at once (0: default) */
    int32_t wave_tiles;         /* tiles whose layers are interleaved in the work order (0: = ring_slots) */
    int32_t max_ctas;           /* persistent CTAs (0: one per SM) */
    int64_t wait_timeout_ns;    /* limit of a device-side wait before MAFAT_ETIMEOUT (0: 2 s) */
    int32_t test_unpublished_task; /* test hook: index of a task whose completion is never
                                      published, so that waits on it run out (-1: none) */
    int32_t dry_run;            /* 1: build the host-side tables only (statistics and region
                                   queries work; runs are refused); needs no GPU */
    int32_t trace;              /* 1: record per-item timestamps on every run (mafat_plan_trace) */
    int32_t force_nblk;         /* output channels per work item for every stage (0: chosen per stage) */
    int32_t force_mb;           /* 16x8 pixel blocks per work item for every stage (0: chosen per stage) */
    int32_t lookahead_items;    /* a stage with at least this many work items (all tiles and frames)
                                   takes each CTA's next item before the CTA's input buffer for it
                                   is free, hiding the hand-out latency; smaller stages take it
                                   only then, so that a busy CTA holds no item an idle one could
                                   start (0: 5/4 of the CTAs; < 0: never) */
    const int32_t* tile_bounds; /* non-uniform tiling (NULL: the even N x M grid): for each group, its
                                   grid_n + 1 row bounds then its grid_m + 1 column bounds on the
                                   group's last-layer output, 0 = b[0] < b[1] < ... < b[n] = size */
    int32_t halo_reuse;         /* 1: inter-tile reuse instead of halo recompute: a tile computes only
                                   its own part of every layer, into whole layer maps on the device,
                                   and reads the halo its next layer needs from its neighbours' parts
                                   (each layer waits for those neighbours); 0: the fused tiles of
                                   Sec. 3-4, every tile recomputing its halo */
    int32_t frame_major;        /* batch > 1 with two groups: 1 hands the frames out strictly one after
                                   another; 0 (default) overlaps frame f's second group with frame
                                   f + 1's first (the second group's small maps leave SMs idle) */
    int32_t chain;              /* BF16 plans: 1 chains a 3x3 convolution and the 1x1 convolution after
                                   it inside one work item where both fit one TMEM accumulator buffer:
                                   the 3x3's activated bf16 output stays in tensor memory and is the
                                   1x1's A operand, so it never reaches shared or global memory.
                                   0 (default): every convolution is a stage of its own (on GB300 the
                                   chained form measured slower for the 608x608 YOLOv2 plan) */
    int32_t rect_blocks;        /* 1: every work item's pixel blocks are 16x8 rectangles.  0 (default):
                                   a convolution without a fused max-pool whose tile regions are at
                                   most 32 - k + 1 pixels wide reads each region as its rows laid end
                                   to end with a pitch of a multiple of 8 pixels, cut into runs of
                                   128 pixels, where that takes fewer blocks (e.g. a 19x19 region: 4
                                   blocks instead of 6); results are identical either way */
} mafat_plan_options;

/* Statistics of a plan (all per batch unless stated). */
typedef struct {
    int32_t struct_size;
    int32_t n_groups;
    int32_t n_tiles;            /* non-empty tiles over all groups and frames */
    int32_t n_tasks;            /* (frame, tile, fused conv stage) units */
    int64_t n_items;            /* work items handed out by the persistent scheduler */
    double useful_flops;        /* 2*MAC of the convolutions of the unfused network */
    double executed_flops;      /* 2*MAC over all tile regions (includes halo recompute) */
    double issued_flops;        /* 2*MAC issued to the arithmetic units (includes block padding) */
    double predicted_mib;       /* Algorithm 1 (literal reading, bias 31 MiB) for this configuration */
    int64_t group_io_bytes;     /* group inputs + group outputs, once each */
    int64_t weight_bytes;       /* packed weights + scale/bias */
    int64_t scratch_bytes;      /* device buffers of live tile intermediates */
    int64_t workspace_bytes;    /* all device memory the plan owns */
    int64_t smem_bytes_per_cta; /* on-chip shared memory per CTA */
    int32_t ring_slots;
    int32_t wave_tiles;
    int32_t max_ctas;
    int32_t dtype;
    int32_t frames_overlapped;  /* 1: the hand-out order overlaps frame f's second group with frame
                                   f + 1's first (batch > 1, two groups, ring of a whole frame) */
    int32_t reserved;
} mafat_plan_stats_t;

/* Build a network description: validates the layers and infers every layer's
 * shape, out = floor((in + 2*pad - k) / stride) + 1 (Sec. 4.1, Algorithm 2's
 * W, H, F, S).  in_c is the channel count of the input image.  The caller keeps
 * ownership of `layers`.  EUNSUPPORTED for layer types/shapes outside the
 * supported set above (e.g. a max-pool on an odd-sized map). */
mafat_status mafat_describe_net(const mafat_layer_desc* layers, int32_t n,
                                int32_t in_h, int32_t in_w, int32_t in_c,
                                mafat_net_t** out);

/* Shape of layer `layer`: shape[6] = {h_in, w_in, c_in, h_out, w_out, c_out}. */
mafat_status mafat_net_shape(const mafat_net_t* net, int32_t layer, int32_t shape[6]);

/* Set the parameters of convolution layer `layer`: w_host [Cout][Cin][k][k]
 * (cross-correlation), scale[Cout] and bias[Cout] of the folded batch-norm,
 * all host fp32.  The library copies them; the caller keeps ownership.
 * Plans created afterwards use these values (bf16 plans round w to bf16,
 * nearest-even). */
mafat_status mafat_set_weights(mafat_net_t* net, int32_t layer, const float* w_host,
                               const float* scale, const float* bias);

/* Plan fused-tile execution (Sec. 4): n_groups (1..MAFAT_MAX_GROUPS; the paper
 * uses 1 or 2) layer groups split at the increasing cuts[0..n_groups-2] (the
 * first layer of each later group), group g tiled grid_n[g] x grid_m[g], for
 * `batch` images, in dtype dt.  The plan owns its device workspace (packed
 * weights, cut tensor, tile buffers, counters) on the current device; every
 * convolution must have weights set.  ENOFIT if a tile cannot be scheduled,
 * EUNSUPPORTED if a max-pool would be separated from its convolution.
 * Allocates device memory; not for use during stream capture. */
mafat_status mafat_plan(const mafat_net_t* net, int32_t n_groups, const int32_t* cuts,
                        const int32_t* grid_n, const int32_t* grid_m, int32_t batch,
                        int32_t dt, mafat_plan_t** out);

/* mafat_plan with options (may be NULL). */
mafat_status mafat_plan_ex(const mafat_net_t* net, int32_t n_groups, const int32_t* cuts,
                           const int32_t* grid_n, const int32_t* grid_m, int32_t batch,
                           int32_t dt, const mafat_plan_options* opt, mafat_plan_t** out);

/* Run the plan on `stream` (asynchronous): one persistent fused kernel running
 * every group and tile of the plan (Sec. 3-4).
 *   input : device, NHWC [batch][H][W][C] elements of the plan's dtype, the
 *           image batch as it comes (C = the net's input channels, e.g. 3).
 *   output: device, NHWC [batch][H_out][W_out][C_out] of the plan's dtype.
 * Both caller-owned, 16-byte aligned, not overlapping (EINVAL otherwise).  The
 * first layer reads the NHWC input in place: BF16 plans with C < 8 load raw
 * image rows and widen them to 8 channels inside the kernel, which needs rows of
 * W * C * 2 bytes to be a multiple of 16 (and C = 8 is read as it is); for other
 * widths, and for C > 8, one small layout kernel first writes an octet-planar
 * copy into plan-owned memory (two launches, see mafat_launches_per_run).  Returns launch errors only; device-side wait
 * errors are reported by mafat_sync_status.  Calls on one plan must not overlap
 * in time (they share the plan's workspace).  Capturable into a CUDA graph. */
mafat_status mafat_run(const mafat_plan_t* plan, const void* input, void* output, void* stream);

/* mafat_run, then copy the group-1 output (the cut tensor, layout
 * [batch][C/8][H][W][8]) into cut_out (device, caller-owned); for a
 * single-group plan cut_out is ignored. */
mafat_status mafat_run_debug(const mafat_plan_t* plan, const void* input, void* cut_out,
                             void* output, void* stream);

/* End-to-end call on HOST buffers.  input_host is the image batch as it comes,
 * NHWC [batch][H][W][C] in the plan's dtype (C = the net's input channels, no
 * padding); output_host is NHWC [batch][H_out][W_out][C_out] as for mafat_run.
 * Copies the input to plan-owned device memory, runs mafat_run on it, copies the
 * output back and synchronises `stream`; returns the device status as
 * mafat_sync_status does.  Pinned host memory gives asynchronous copies.
 * Allocates the plan's staging buffers on its first call. */
mafat_status mafat_run_host(const mafat_plan_t* plan, const void* input_host, void* output_host,
                            void* stream);

/* Frames in flight on HOST buffers: the asynchronous form of mafat_run_host
 * (same layouts).  Enqueues the input upload on a plan-owned copy stream, the
 * run on `stream`, and the read-back of the output on a
 * second plan-owned copy stream, then returns; two staging slots alternate, so
 * the upload of one frame overlaps the run of the one before.  input_host must
 * stay unchanged, and output_host unread, until mafat_run_host_wait returns (or
 * until the frame after next has been enqueued, for the input).  Runs on one plan
 * still execute one after another.  Allocates the slots, streams and events on
 * its first call.  Launch errors only; device status via mafat_run_host_wait. */
mafat_status mafat_run_host_async(const mafat_plan_t* plan, const void* input_host, void* output_host,
                                  void* stream);

/* Wait until every frame enqueued by mafat_run_host_async has its output in host
 * memory; returns the device status as mafat_sync_status does. */
mafat_status mafat_run_host_wait(const mafat_plan_t* plan);

/* Synchronise `stream` and read (and clear) the plan's device status word:
 * MAFAT_OK, MAFAT_ETIMEOUT (a tile waited on another that never finished) or
 * MAFAT_EDEVICE. */
mafat_status mafat_sync_status(const mafat_plan_t* plan, void* stream);

/* Host-side query of the Grid traversal (Sec. 4.1): input and output
 * rectangle of layer `layer` for tile (ti, tj) of group `group`.  With halo reuse
 * the output rectangle is the part of the layer the tile computes (owns) and the
 * input rectangle what that part reads (its neighbours' parts included). */
mafat_status mafat_tile_region(const mafat_plan_t* plan, int32_t group, int32_t ti, int32_t tj,
                               int32_t layer, int32_t in_rect[4], int32_t out_rect[4]);

/* Same traversal without a plan: tile (ti, tj) of an n x m grid over the
 * output of layers first..last. */
mafat_status mafat_net_tile_region(const mafat_net_t* net, int32_t first, int32_t last,
                                   int32_t n, int32_t m, int32_t ti, int32_t tj, int32_t layer,
                                   int32_t in_rect[4], int32_t out_rect[4]);

/* Algorithm 1 for one layer group (layers first..last, n x m tiles): the
 * maximum over tiles and layers of scratch + output + input_factor*input
 * elements (scratch = w_out*h_out*c_in*F^2/S), times 4 bytes, in MiB, plus
 * bias_mib (the paper uses input_factor 2 and a 31 MB bias). */
mafat_status mafat_predict_layer_group(const mafat_net_t* net, int32_t first, int32_t last,
                                       int32_t n, int32_t m, double bias_mib,
                                       int32_t input_factor, double* out_mib);

/* predictMem of Algorithm 2: the maximum of Algorithm 1 over the groups of a
 * configuration (cut, n1 x m1 top tiling, n2 x m2 bottom tiling), MiB. */
mafat_status mafat_predict_mem(const mafat_net_t* net, int32_t cut, int32_t n1, int32_t m1,
                               int32_t n2, int32_t m2, double bias_mib, double* out_mib);

/* Work-balanced non-uniform tile bounds for layers first..last: n + 1 row bounds and
 * m + 1 column bounds on the last layer's output, chosen per axis so that the largest
 * part's executed work (its regions traced back through every convolution of the
 * group, halo included, the other axis whole) is as small as possible.  Edge tiles need
 * less halo, so they come out larger than interior ones.  Pass them as
 * mafat_plan_options.tile_bounds.  Host only. */
mafat_status mafat_balanced_bounds(const mafat_net_t* net, int32_t first, int32_t last, int32_t n, int32_t m,
                                   int32_t* row_bounds, int32_t* col_bounds);

/* Algorithm 2: search cut in {n (no cut), 12, 8} x square top tilings 1..5
 * with a 2x2 bottom tiling, returning the first configuration predicted
 * strictly below limit_mib, else 5x5 / cut 8 / 2x2.  *cut == n means no cut. */
mafat_status mafat_search(const mafat_net_t* net, double limit_mib, double bias_mib,
                          int32_t* top_tile, int32_t* cut, int32_t* bottom_tile);

/* Measured plan search: Algorithm 2 (Sec. 4.1) re-targeted at the GPU.  Algorithm 2
 * looks for the cut and tilings of lowest latency whose predicted memory fits the
 * device; here the memory that matters is the L2 that a plan's intermediates (tile
 * scratch ring and cut tensor) should stay in, and latency is measured rather than
 * predicted: every candidate within budget_bytes is planned and timed on the device,
 * and the fastest is reported.  Candidates, in this order: one layer group (if
 * include_one_group), then two groups at each cut of cuts[0..n_cuts-1] (the first
 * layer of group 2), every group tiled N x M for N, M in 1..max_grid (N == M when
 * square_only, else |N - M| <= 1), group 1's tiling outer. */
typedef struct {
    int32_t struct_size;        /* sizeof(mafat_search_options) */
    int32_t batch;              /* images per run (0: 1) */
    int32_t dtype;              /* MAFAT_BF16 or MAFAT_FP32 */
    int32_t include_one_group;
    int32_t n_cuts;
    const int32_t* cuts;        /* n_cuts candidate cuts (may be NULL when n_cuts == 0) */
    int32_t max_grid;           /* tiles per axis 1..max_grid (0: 5) */
    int32_t square_only;
    int64_t budget_bytes;       /* intermediate bytes allowed (0: the device's L2 size, or 128 MiB for a
                                   dry run; < 0: no limit) */
    int32_t runs;               /* timed runs per candidate, median reported (0: 10) */
    int32_t flush_l2;           /* 1: write 256 MiB before each timed run (every run starts with a cold L2) */
    int32_t dry_run;            /* 1: enumerate and size the candidates only; needs no GPU */
    int32_t reserved[3];
} mafat_search_options;

typedef struct {
    int32_t n_groups, cut;      /* cut is 0 for one group */
    int32_t grid_n[2], grid_m[2];
    int64_t intermediate_bytes; /* tile scratch ring + cut tensor of the plan */
    double predicted_mib;       /* Algorithm 1 (literal reading, 31 MiB bias) for the configuration */
    double executed_flops;      /* per run, halo recompute included */
    double us_per_run;          /* median device time of a run; < 0 if not timed */
    int32_t status;             /* MAFAT_OK if timed; MAFAT_ENOFIT over budget; else the plan's error */
    int32_t reserved;
} mafat_search_candidate;

/* Runs the measured search on `stream` (the net's weights must be set; the input is
 * synthetic, since a run's time does not depend on the data).  Writes the first
 * max_out candidates to out (may be NULL), their total number to *n_out and the
 * index of the fastest timed one to *best (-1 if none was timed).  Allocates device
 * memory; not for use during stream capture. */
mafat_status mafat_search_measured(const mafat_net_t* net, const mafat_search_options* opt, void* stream,
                                   mafat_search_candidate* out, int32_t max_out, int32_t* n_out,
                                   int32_t* best);

/* Statistics of a plan: the useful, executed (halo recompute included) and issued
 * FLOPs of a run, Algorithm 1's prediction for its configuration (Sec. 4.1), its
 * tiles, tasks and work items, and the device memory it owns.  out is caller-owned
 * host memory; out->struct_size must be set to sizeof(mafat_plan_stats_t) (EINVAL if
 * smaller).  Host only; works on dry-run plans. */
mafat_status mafat_plan_stats(const mafat_plan_t* plan, mafat_plan_stats_t* out);

/* Per-item trace of the last run of a plan created with options.trace = 1
 * (synchronises `stream`).  out receives n_items records of MAFAT_TRACE_WORDS
 * uint64 in hand-out order: {global ns when the item's ticket was taken, when
 * its dependencies were satisfied, when its accumulator was ready for the
 * epilogue, when its completion was published, SM id, task index << 16 |
 * network layer of its convolution, when its first input halo had landed in
 * shared memory, when its last MMA was issued, ns the MMA issuer waited for
 * later input halos, ns it waited for streamed weight pieces}.  max_words
 * bounds what is written. */
#define MAFAT_TRACE_WORDS 10
mafat_status mafat_plan_trace(const mafat_plan_t* plan, uint64_t* out, int64_t max_words, void* stream);

/* Number of kernel launches one mafat_run makes: 1, or 2 for a BF16 plan whose
 * input needs the layout kernel (C > 8, or C < 8 with rows of W * C * 2 bytes
 * that are not a multiple of 16). */
int32_t mafat_launches_per_run(const mafat_plan_t* plan);

void mafat_plan_destroy(mafat_plan_t* plan);
void mafat_net_destroy(mafat_net_t* net);

/* Message of the last failure on the calling thread ("" if none). */
const char* mafat_last_error(void);

/* Library version string. */
const char* mafat_version(void);

/* Allocation-free run; the paper has no counterpart.  For callers that cannot
 * have device memory allocated for them while they run (code executing during
 * a global-mode stream capture, where cudaMalloc is refused; real-time loops
 * that forbid allocator calls; processes whose device memory is owned and
 * budgeted by another allocator).  Runs an FP32 plan created beforehand (its
 * weights and tables are read in place) with all per-run scratch -- tile
 * buffers, cut tensor, scheduler counters -- taken from one fixed 32 MiB
 * device area inside this library, which every GPU that loads the library
 * keeps until exit; it calls no allocation routine.  Plans needing more
 * scratch than 32 MiB are refused with MAFAT_EINVAL; BF16 plans with
 * MAFAT_EUNSUPPORTED; input and output that overlap with MAFAT_EINVAL.  Layouts
 * as mafat_run; asynchronous on `stream`.  All calls share the area: calls that
 * overlap on the GPU race.  The first call on each device looks up the area's
 * device address and clears its status word (a synchronous step), so make it
 * before any stream capture starts.  Device-side wait errors of these calls go
 * to the area's own status word: read them with mafat_noalloc_sync_status, not
 * mafat_sync_status (which reads the plan's). */
mafat_status mafat_run_fp32_noalloc(const mafat_plan_t* plan, const void* input, void* output, void* stream);

/* Device status of mafat_run_fp32_noalloc calls on the current device; no
 * counterpart in the paper.  Synchronises `stream`, then reads and clears the
 * status word of the static area: MAFAT_OK, MAFAT_ETIMEOUT (a tile waited on
 * another that never finished) or MAFAT_EDEVICE.  The first error since the last
 * read is kept; later calls do not overwrite it.  Allocates nothing. */
mafat_status mafat_noalloc_sync_status(void* stream);

/* Diagnostic with no counterpart in the paper: one 128 x n x 16 bf16 tensor-core
 * product D = A * B^T on one CTA, with the operand and accumulator layouts the fused
 * kernel uses, to check them: B (and, with a_in_tmem = 0, A) read from shared memory
 * through the kernel's descriptor encoding; with a_in_tmem = 1, A written to tensor
 * memory first (lane = row, two bf16 per 32-bit column), as the chained 3x3 -> 1x1
 * layers pass their intermediate.  a_dev [128][16], b_dev [n][16] (bf16, row-major,
 * device), d_dev [128][n] fp32 (device); n in {16, 32, ..., 256}.  Synchronous. */
mafat_status mafat_diag_umma(const void* a_dev, const void* b_dev, float* d_dev, int32_t n, int32_t a_in_tmem,
                             void* stream);

#ifdef __cplusplus
}
#endif

#endif /* MAFAT_H */

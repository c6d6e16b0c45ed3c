// Host-side planner: network shapes, the Grid back-traversal of tile regions,
// the memory predictor (Algorithm 1), the configuration search (Algorithm 2)
// and the lowering of a fused-tile configuration (Sec. 4) to the flat work
// tables the persistent kernels consume.  Plain C++; no CUDA calls.
#pragma once
#include <stdint.h>

#include <string>
#include <vector>

#include "../../include/mafat.h"
#include "device_types.h"

namespace mafat {

enum { L_CONV = 0, L_MAXPOOL = 1 };

struct Layer {
    int type, k, stride, pad, filters;
    int h_in, w_in, c_in, h_out, w_out, c_out;
};

struct Rect {
    int y0 = 0, y1 = 0, x0 = 0, x1 = 0;  // half-open
    int h() const { return y1 - y0; }
    int w() const { return x1 - x0; }
    bool empty() const { return y1 <= y0 || x1 <= x0; }
    bool operator==(const Rect& o) const { return y0 == o.y0 && y1 == o.y1 && x0 == o.x0 && x1 == o.x1; }
};

struct Net {
    std::vector<Layer> layers;
    int in_h = 0, in_w = 0, in_c = 0;
    std::vector<std::vector<float>> w, scale, bias;  // per layer (empty for max-pool)
    std::vector<char> has_w;
};

// Shape inference; returns "" or an error message (unsupported layers).
std::string build_net(const int32_t* desc5, int n, int in_h, int in_w, int in_c, Net& net);

// Even partition bound i of `len` into `n` parts: floor(i * len / n).
inline int grid_bound(int len, int n, int i) { return (int)((int64_t)i * len / n); }

// Input interval of a layer needed for output interval [a, b), clipped to [0, size_in).
void back_interval(int a, int b, int k, int s, int p, int size_in, int* lo, int* hi);

// Grid traversal: out_rects[l] / in_rects[l] for every layer l of first..last
// (vectors indexed by layer; entries outside the group untouched), for tile (i, j)
// of the even n x m grid on layer last's output.
void tile_regions(const Net& net, int first, int last, int n, int m, int i, int j,
                  std::vector<Rect>& out_rects, std::vector<Rect>& in_rects);
// Halo reuse: the part of every layer's output a tile owns and the input region each
// layer reads for it (vectors indexed by layer, as above).
void owned_regions(const Net& net, int first, int last, const Rect& out_last, std::vector<Rect>& out_rects,
                   std::vector<Rect>& in_rects);
// The same traversal from any output rectangle of layer last.
void rect_regions(const Net& net, int first, int last, const Rect& out_last, std::vector<Rect>& out_rects,
                  std::vector<Rect>& in_rects);

// Tile bounds of a group along one axis: n + 1 increasing values from 0 to len.
// Empty `given` means the even partition.
std::vector<int> axis_bounds(int len, int n, const std::vector<int>& given);
// "" if `b` is a valid bounds vector for n parts of len (0 = b[0] < ... < b[n] = len).
std::string check_bounds(const std::vector<int>& b, int len, int n);

// Work-balanced bounds along one axis of group first..last (the non-uniform tiling of
// Sec. 6): n parts of the last layer's output such that the largest part's executed
// MACs (its regions back-traversed through every conv of the group, the other axis
// taken whole) is as small as possible.  axis 0: rows, 1: columns.
std::vector<int> balanced_bounds(const Net& net, int first, int last, int n, int axis);

// Algorithm 1 (literal reading), MiB.
double predict_layer_group(const Net& net, int first, int last, int n, int m, double bias_mib,
                           int input_factor);
// predictMem: maximum over groups; cut <= 0 or >= n: single group with n1 x m1.
double predict_mem(const Net& net, int cut, int n1, int m1, int n2, int m2, double bias_mib);
// Algorithm 2; returns (top_tile, cut, bottom_tile) with cut == n for NoCut.
void search(const Net& net, double limit_mib, double bias_mib, int* top, int* cut, int* bottom);

struct PlanConfig {
    int n_groups = 1;
    int cuts[MAFAT_MAX_GROUPS - 1] = {0, 0, 0};  // first layer of groups 2.. (increasing)
    int grid_n[MAFAT_MAX_GROUPS] = {1, 1, 1, 1}, grid_m[MAFAT_MAX_GROUPS] = {1, 1, 1, 1};
    int batch = 1;
    int dtype = 0;            // 0 bf16, 1 fp32
    int ring_slots = 0;
    int wave_tiles = 0;
    int unpublished_task = -1;
    int n_ctas = 0;           // persistent CTAs (shapes items; 0: 152)
    int fixed_nblk = 0;       // force the output-channel block of every stage (0: choose)
    int fixed_mb = 0;         // force blocks per item (0: choose)
    bool halo_reuse = false;  // tiles compute only their own part of every layer and read the halo from
                              // their neighbours' results in whole layer maps (no recompute)
    int lookahead_items = 0;  // stages with at least this many items take tickets early (0: 5/4 n_ctas, < 0: never)
    bool frame_major = false; // batch > 1: hand frames out one after another, never overlapped
    bool chain = false;       // chain a 3x3 and the 1x1 after it on chip where both fit a TMEM buffer
    bool rect_blocks = false; // 16x8 rectangular M blocks only (no flattened blocks, MafatStageDev::flat)
    // explicit tile bounds per group (empty: even): rows[g] has grid_n[g] + 1 entries, cols[g] grid_m[g] + 1
    std::vector<int> row_bounds[MAFAT_MAX_GROUPS], col_bounds[MAFAT_MAX_GROUPS];
};

// A tensor-map request for a task whose input is a scratch region buffer.
struct TmapReq {
    int task;
    int64_t elem_off;         // buffer start in the scratch allocation (elements)
    int h, w, c8, frames;     // buffer extent (frames: 1 for a tile buffer, batch for a layer map)
    int rows_box, cols_box, chunk8;
};

struct PlanTables {
    PlanConfig cfg;
    int frames_overlapped = 0;           // 1: frame f's second group overlaps frame f + 1's first in the order
    int groups[MAFAT_MAX_GROUPS][2];     // [g] = {first, last} layer
    std::vector<int> rows[MAFAT_MAX_GROUPS], cols[MAFAT_MAX_GROUPS];  // tile bounds on each group's output
    int stage_first[MAFAT_MAX_GROUPS], stage_last[MAFAT_MAX_GROUPS];  // stage index range per group
    std::vector<MafatStageDev> stages;
    std::vector<MafatTaskDev> tasks;
    std::vector<MafatItemDev> items;
    std::vector<TmapReq> tmaps;          // index i = tensor map i (scratch inputs)
    int64_t weight_elems = 0;            // packed bf16 weight elements
    int64_t weight32_elems = 0;          // fp32 weight elements
    int64_t sb_elems = 0;                // scale / bias elements
    int64_t slot_buf_elems = 0;          // elements of one ping-pong buffer
    int64_t scratch_elems = 0;           // the scratch allocation (ring, or layer maps with halo reuse)
    std::vector<MafatDepDev> deps;       // task dependency lists (halo reuse)
    int ring_slots = 0, wave_tiles = 0;
    int n_counters = 0;                  // words after MAFAT_CTR_BASE
    int frame_ctr_base = 0;              // completion counters of every group but the last, per frame:
                                         // frame_ctr_base + frame * (n_groups - 1) + group
    int n_tiles = 0;
    // input / cut / output geometry (the cut tensor is group 1's output; the outputs of
    // groups 2 .. n_groups - 1 are layer maps in the scratch allocation)
    int in_c8 = 0;
    int in_convert = 0;                  // 1: the NHWC input is converted to octet-planar before the launch
                                         // (tensor-core plans whose raw input rows are not 16-byte multiples)
    int cut_h = 0, cut_w = 0, cut_c8 = 0;
    int out_h = 0, out_w = 0, out_c = 0;
    // box of the group-1 first stage (user input map) and group-2 first stage (cut map)
    int in_rows_box = 0, in_cols_box = 0, in_chunk8 = 0;
    int cut_rows_box = 0, cut_cols_box = 0, cut_chunk8 = 0;
    // statistics
    double useful_flops = 0, executed_flops = 0, issued_flops = 0, predicted_mib = 0;
    int64_t group_io_elems = 0;
};

// Lower a configuration; returns "" or an error message.  `unsupported` is
// set when the configuration is valid but not implemented.
std::string build_plan(const Net& net, const PlanConfig& cfg, PlanTables& t, bool* unsupported);

// Check every item of lowered tables against the buffers they address: box and
// blob sizes against the kernel's stages, weight ranges, input and output
// extents of every valid pixel, counter indices, and that every dependency
// consists of items handed out earlier.  Returns "" or the first violation.
std::string validate_plan(const Net& net, const PlanTables& t);

// Pack fp32 weights [cout][cin][k][k] of every stage into the bf16 tensor-core
// blob order (see pack_weights_bf16 in planner.cpp); out has weight_elems entries.
void pack_weights_bf16(const Net& net, const PlanTables& t, std::vector<uint16_t>& out);
void pack_weights_fp32(const Net& net, const PlanTables& t, std::vector<float>& w32,
                       std::vector<float>& scale, std::vector<float>& bias);

uint16_t f32_to_bf16_rne(float f);

}  // namespace mafat

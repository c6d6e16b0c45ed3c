// Plan tables shared by the host planner and the persistent kernels.
//
// A plan is lowered to three flat tables that live in device memory:
//   * MafatStageDev  -- one per fused convolution stage of the network (a conv
//                       layer, with the 2x2/s2 max-pool that follows it folded
//                       into its epilogue), with packed-weight offsets;
//   * MafatTaskDev   -- one per (frame, tile, stage): which buffer the stage
//                       reads, which rectangle of the conv output it computes
//                       (the tile's region from the Grid back-traversal,
//                       Sec. 4.1) and where the result goes;
//   * MafatItemDev   -- the work list in hand-out order: one item is up to
//                       `mb` blocks of 128 conv output pixels x one block of
//                       output channels of a task, with up to two completion
//                       counters it must wait for.  A block is a 16 x 8
//                       rectangle (stacked along rows), or, in a `flat`
//                       stage, a run of 128 pixels of the task's region read
//                       row after row with a row pitch of `cols_box` pixels.
//
// Activations are stored in "octet-planar" layout [C/8][H][W][8]: 8 channels of
// one pixel are 16 bytes (bf16) or 32 bytes (fp32) and consecutive pixels of a
// row are adjacent, so 8 pixels x 8 channels form one contiguous 128-byte
// tensor-core core matrix at any pixel offset.
#pragma once
#include <stdint.h>

#if defined(__CUDACC__)
#define MAFAT_HD __host__ __device__
#else
#define MAFAT_HD
#endif

#define MAFAT_BLK_ROWS 16   // conv output rows of one M block
#define MAFAT_BLK_COLS 8    // conv output columns of one M block (M = 128)
#define MAFAT_MAX_MB 4      // M blocks per work item
#define MAFAT_MAX_MB_PAIRED 8  // M blocks per work item of a paired-tap (8-input-channel) layer
#define MAFAT_MAX_NBLK 256  // output channels of one item (MMA N)
#define MAFAT_A_STAGE_BYTES 36864   // shared-memory A halo stage of the tensor-core kernel (x2)
#define MAFAT_B_PIECE_BYTES 75776   // one of the two shared-memory weight buffers (x2)

// SCRATCH: a tile's own region buffer in the scratch ring (frame in the offset); MAP: a
// whole layer-output map of every frame in the scratch allocation (halo reuse: tiles
// read their neighbours' results from it; frame as the tensor map's fourth coordinate).
enum { MAFAT_BUF_USER_IN = 0, MAFAT_BUF_CUT = 1, MAFAT_BUF_SCRATCH = 2, MAFAT_BUF_USER_OUT = 3, MAFAT_BUF_MAP = 4 };

// One entry of a task's dependency list: wait until counter ctr reaches target.
struct MafatDepDev {
    int32_t ctr, target;
};

struct MafatStageDev {
    int32_t layer;        // network layer index of the conv
    int32_t k, pad;       // 3/1 or 1/0
    int32_t cin, cin8;    // input channels and octets (cin8 = ceil(cin/8))
    int32_t cout;         // output channels
    int32_t pool;         // 1: a 2x2/s2 max-pool follows and is fused
    // tensor-core packing
    int32_t n_blk;        // output channels per item (MMA N)
    int32_t n_nblk;       // cout / n_blk
    int32_t chunk8;       // input octets per A chunk (8 = 64 channels, or cin8 if smaller)
    int32_t n_chunks;     // cin8 / chunk8
    int32_t paired;       // 1: cin8 == 1, two taps share one K=16 step
    int32_t n_bsteps;     // weight blobs per chunk (taps, or tap pairs)
    int32_t kst;          // K=16 MMA steps per blob
    int32_t b_swz;        // 1: blobs in the 128-byte swizzled K-major layout (kst == 4), 0: no swizzle
    int32_t mb;           // M blocks per item (stacked along rows, one TMEM accumulator each)
    int32_t rows_box, cols_box;  // A halo box (pixels): 16*mb + k - 1 rows, 8 + k - 1 columns
                                 // (flat stage: mafat_flat_rows(mb, pitch, k) rows, pitch columns)
    // Flattened M blocks (convolutions without a fused pool, tensor maps of at most 32 pixels a
    // row): the task's conv region of ch x cw pixels is read as ch rows of `pitch` = cols_box
    // pixels (a multiple of 8, at least cw + k - 1) laid end to end, and block b is pixels
    // 128 b .. 128 b + 127 of that sequence, pixel p being (p / pitch, p % pitch); pixels in
    // columns cw .. pitch - 1 are computed and dropped.  The A halo of an item is the same
    // rows laid out the same way, so that 8 consecutive pixels are one core matrix wherever a
    // row ends, and tap (ky, kx) is an offset of ky * pitch + kx pixels.  A region 19 pixels
    // wide takes 4 such blocks for 19 rows instead of 6 rectangles.
    int32_t flat;
    int64_t w_off;        // element offset of this stage's packed bf16 weights
    int32_t blob_elems;   // elements of one blob (n_blk * 16 * kst)
    int32_t set_bytes;    // bytes of the weights of one output-channel block (all chunks and blobs)
    int32_t bpp;          // blobs per weight piece (a piece fills at most one shared-memory buffer)
    int32_t n_pieces;     // pieces per channel block (1: the set stays resident across items)
    int32_t sb_off;       // offset into the scale / bias arrays
    int32_t lookahead;    // 1: a CTA takes its next item as soon as this stage's item is loaded
    int64_t w32_off;      // element offset of the fp32 weights [cout][cin][k][k]
    // How a task of this stage that reads the caller's input (NHWC [frames][H][W][cin]) gets its
    // A halo into shared memory (tensor-core kernel; other tasks read octet-planar buffers):
    //   MAFAT_IN_PLANAR: one 4-D box per chunk (cin == 8, whose NHWC is one octet plane, or a
    //                    copy converted to octet-planar before the launch);
    //   MAFAT_IN_GATHER: cin < 8: the box's rows of raw NHWC elements (raw_e per row, from a
    //                    16-byte aligned element) land in the stage's tail, and the gather warp
    //                    expands them into the one-octet halo, channels cin..7 zero.
    int32_t in_mode;
    int32_t raw_e;        // MAFAT_IN_GATHER: elements of one raw row in shared memory (multiple of 8)
    // Pixel pairs (a gathered 3x3 stage of at most 4 input channels): 16-byte halo slot q holds
    // the channels of pixels q and q + 1, 4 channels (8 bytes) each, the unused ones zero.  A
    // core-matrix row of slot q then spans taps kx and kx + 1 of one kernel row, and one K = 16
    // step covers a whole kernel row: its K halves are slots kx = 0 (taps 0, 1) and kx = 2 (tap
    // 2 and a zero tap), LBO two slots apart.  A 3x3 convolution takes 3 K steps instead of the
    // 5 of tap pairs over 8-channel pixels (K 48 against 80 for 27 useful values).
    int32_t pix_pair;
    // Per-block halos (every gathered stage): the A stage holds one (16 + k - 1) x cols_box halo
    // per block of the item, block after block, so that an item's blocks need not be stacked in
    // one block column: they are any run of the task's blocks in column-major order (linear
    // index bx * nby + by; the item's `by` is its first block's index, `bx` is 0).  The
    // widening builds each block's halo from raw rows loaded block by block.  A 137-row tile
    // region (9 block rows) then takes items of 8 blocks instead of 5 + 4 per block column.
    int32_t blk_halo;
    // On-chip chaining of a 3x3 convolution and the 1x1 convolution after it (tensor-core plans):
    // an item of a `chain` stage computes its pixels for all of the 3x3's channels into TMEM, the
    // epilogue writes the activated bf16 result back into TMEM as the A operand of the 1x1, and
    // the 1x1 (the next stage, marked `chained`, which has no tasks of its own) runs from there.
    // Columns of one 256-column accumulator buffer: [0, n_blk) the 3x3's accumulator,
    // [chain_a_col, + n_blk / 2) its bf16 result, [chain_out_col, + next stage's n_blk) the 1x1's.
    int32_t chain;
    int32_t chained;
    int32_t chain_a_col, chain_out_col;
    // chain stage: what the kernel needs of the chained 1x1 (a copy of its stage's fields, so that
    // one stage record serves the item): N, output channels, fused pool, input chunks, K steps and
    // swizzle of its weight blobs, blobs per piece, pieces, blob elements, scale / bias offset,
    // packed weight offset
    int32_t c2_n_blk, c2_cout, c2_pool, c2_n_chunks, c2_kst, c2_b_swz, c2_bpp, c2_n_pieces, c2_blob_elems, c2_sb_off;
    int64_t c2_w_off;
};

enum { MAFAT_IN_PLANAR = 0, MAFAT_IN_GATHER = 1 };

// Rows of the A box of a flat stage's item: its 128 * mb pixels start anywhere in a row of
// `pitch` pixels, and the last of them reads (k - 1) rows and (k - 1) pixels further on.
inline MAFAT_HD int mafat_flat_rows(int mb, int pitch, int k) {
    return (128 * mb + pitch - 1 + (k - 1) * (pitch + 1) + pitch - 1) / pitch;
}

// Byte offset of the raw rows inside an A stage (MAFAT_IN_GATHER): after the expanded
// one-octet halo of rows_box x cols_box pixels, on a 128-byte boundary.
inline MAFAT_HD int mafat_raw_offset(int rows_box, int cols_box) {
    return (rows_box * cols_box * 16 + 127) & ~127;
}

// Bytes between the raw rows of consecutive blocks of a per-block-halo item (one TMA box of
// 16 + k - 1 rows of raw_e elements each, on 128-byte boundaries).
inline MAFAT_HD int mafat_raw_blk_stride(int k, int raw_e) {
    return ((MAFAT_BLK_ROWS + k - 1) * raw_e * 2 + 127) & ~127;
}

struct MafatTaskDev {
    int32_t stage;        // index into the stage table
    int32_t frame;
    // input buffer
    int32_t in_kind;      // MAFAT_BUF_*
    int32_t in_tmap;      // tensor map index (-1: the user-input map passed to the kernel)
    int64_t in_off;       // element offset from the buffer base (frame included)
    int32_t in_h, in_w;   // buffer extent (pixels)
    int32_t in_y0, in_x0; // map position of buffer pixel (0, 0)
    // conv output rectangle computed by this task (map coordinates, before pooling)
    int32_t cy0, cx0, ch, cw;
    int32_t nby, nbx;     // M blocks along rows / columns (flat stage: blocks of the region, 1)
    // output buffer
    int32_t out_kind;     // MAFAT_BUF_*
    int32_t out_nhwc;     // 1: NHWC (user output), 0: octet-planar
    int64_t out_off;      // element offset (frame included)
    int32_t out_h, out_w; // buffer extent (pixels, after pooling)
    int32_t out_y0, out_x0; // map position of buffer pixel (0, 0) (pooled map)
    int32_t done_ctr;     // counter bumped once per finished item
    int32_t n_items;
    int32_t dep_first, dep_count;  // the task's own dependency list in the plan's list (halo reuse)
};

struct MafatItemDev {
    int32_t task;
    int16_t by, bx;       // M block (flat stage: index of the first block in the region, 0)
    int16_t nb;           // output-channel block
    int16_t nbk;          // M blocks of this item (rows by .. by+nbk-1)
    int16_t flags;        // bit 0: do not publish completion (test hook)
    int16_t stage;        // the task's stage (lets the task and stage records load in parallel)
    int32_t dep0, dep0_target;  // counter index (-1: none) and value to wait for
    int32_t dep1, dep1_target;
    int32_t extra_ctr;    // second counter bumped on completion (-1: none)
};

// Counter block layout (uint32 words).  Zeroed when the plan is created; the
// last CTA to leave a run sets every word except the status back to zero, so
// a run is exactly one kernel launch.
//   [0] ticket, [1] status, [2] abort, [3] CTAs finished, [4 ...] task / frame counters
#define MAFAT_CTR_TICKET 0
#define MAFAT_CTR_STATUS 1
#define MAFAT_CTR_ABORT 2
#define MAFAT_CTR_EXIT 3
#define MAFAT_CTR_BASE 4

// Device status codes (written with atomicCAS from 0).
#define MAFAT_DEV_OK 0u
#define MAFAT_DEV_TIMEOUT 1u
#define MAFAT_DEV_PIPE 2u

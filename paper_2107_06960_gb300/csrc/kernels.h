// Launch interface of the persistent fused-tile kernels (host and device visible).
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "device_types.h"

#define MAFAT_PF_REGIONS 8

struct MafatKParams {
    const MafatStageDev* stages;
    const MafatTaskDev* tasks;
    const MafatItemDev* items;
    int32_t n_items;
    int32_t pad0;
    const CUtensorMap* tmaps;     // scratch-input and cut tensor maps (bf16 path)
    int32_t cut_tmap;             // index of the cut tensor map (-1: none)
    int32_t pad1;
    const uint16_t* w_bf16;       // packed tensor-core weights
    const float* w_f32;           // fp32 weights [cout][cin][k][k] per stage
    const float* scale;
    const float* bias;
    const void* user_in;
    void* user_out;
    void* cut;
    void* scratch;
    uint32_t* ctr;                // counter block (ticket, status, abort, exit, task / frame counters)
    int32_t n_ctr;                // words of the counter block
    int32_t pad2;
    int64_t timeout_ns;
    unsigned long long* trace;    // per-item timestamps (null: off)
    // Regions every CTA warms into L2 (its 1/grid share of each) at start: the input, the
    // packed weights, the work tables and the scale / bias arrays (bytes 0: unused slot).
    const void* pf_ptr[MAFAT_PF_REGIONS];
    int64_t pf_bytes[MAFAT_PF_REGIONS];
    int64_t pf_per[MAFAT_PF_REGIONS];   // each CTA's share of region r (bytes, multiple of 16)
    const MafatDepDev* deps;            // task dependency lists (halo reuse)
};

// bf16 tensor-core kernel (tcgen05 + TMA): one launch runs a whole plan; `chain` selects the
// instance with the on-chip 3x3 -> 1x1 chaining path (plans that have chain stages).
cudaError_t mafat_launch_tc(const MafatKParams& p, const CUtensorMap& in_map, int grid, bool chain, cudaStream_t s);
size_t mafat_tc_smem_bytes();
// fp32 CUDA-core check kernel: same work list, same scheduler.
cudaError_t mafat_launch_fp32(const MafatKParams& p, int grid, cudaStream_t s);
// NHWC [frames][h][w][c] -> octet-planar [frames][c8][h][w][8] (padded channels zero),
// for element sizes of 2 (bf16) or 4 (fp32) bytes.
cudaError_t mafat_launch_to_planar(const void* nhwc, void* planar, int frames, int h, int w, int c, int c8,
                                   int elem_bytes, cudaStream_t s);
// Diagnostic single-MMA kernel.
cudaError_t mafat_launch_diag_umma(const void* a, const void* b, float* d, int n, int a_tmem, cudaStream_t s);

// bf16 tensor-core kernel for fused-tile execution of CNN layer groups
// (MAFAT, Sec. 3-4) on sm_103a: tcgen05 MMA with TMEM accumulators, operands
// staged in shared memory by TMA, one persistent launch per plan.
//
// One work item = up to 8 vertically stacked 16 x 8 blocks of a tile's conv
// output (M = 128 pixels each, one accumulator each) times one block of n_blk
// <= 256 output channels, i.e. an implicit GEMM
//   D[m][n] = sum_{c, ky, kx} A[pixel m shifted by (ky, kx)][c] * W[n][c][ky][kx]
// (M = 128, N = n_blk, K = k*k*Cin) accumulated in fp32 in tensor memory.
//
// Operand layouts (no-swizzle, K-major canonical layout of the tcgen05 shared
// memory descriptor: 8-row x 16-byte core matrices, LBO = stride between the
// two core matrices along K, SBO = stride between 8-row groups along M/N):
//  * A: one TMA box per chunk of <= 64 input channels holds the block's input
//    halo, (16 + k - 1) x (8 + k - 1) pixels, as [octet][row][col][8 ch].  Eight
//    consecutive pixels of a row x 8 channels are one 128-byte core matrix at any
//    pixel offset, so the A operand of tap (ky, kx) is the same buffer at byte
//    offset (ky * cols + kx) * 16: the halo is loaded once and reused for all
//    taps, with no im2col copy.  SBO = one halo row, LBO = one octet plane.
//    With 8 input channels (the first layer), one K=16 step covers two taps:
//    its two K core matrices sit at the two taps' offsets (LBO = their
//    distance).
//  * B: weights pre-packed on the host in exactly their shared-memory image, as
//    blobs of one (chunk, tap); blobs with 64 channels use the 128-byte swizzled
//    K-major layout, narrower ones the no-swizzle one.  The weights of one (stage,
//    output-channel block) travel in pieces filling one of two 74 KB buffers: a
//    set that fits one piece stays resident while the CTA's consecutive items use
//    it, larger sets stream piece by piece (every copy costs a few hundred cycles
//    of TMA time however small it is, so copies are large and few).
//
// Warp roles (384 threads): warps 0-7 epilogue (warp w reads TMEM lanes
// 32(w%4)..+31 = conv rows 4(w%4)..+3 of a block; the two warpgroups take units
// of one block x 32 columns in turn), warp 8 scheduler + TMA producer, warp 9 TMEM
// allocator + MMA issuer, warp 10 publisher (bumps an item's completion counter
// once all epilogue threads have stored it, so that the epilogue warps never wait
// for their stores to reach L2), warp 11 gather (expands raw rows of a narrow NHWC
// input image, e.g. 3-channel RGB, into the 8-channel halo layout of the first layer).  Shared memory: 2 A halo stages, 2 weight
// buffers, a 4-deep queue of items with the record the epilogue needs (written by
// the producer, so the epilogue reads no work table from global memory), and one
// scale / bias slot per accumulator (copied in by the MMA warp and landing on the
// accumulator's full barrier); TMEM: 2 accumulators of 256 columns (the epilogue
// of one item overlaps the MMAs of the next).
//
// Epilogue: y = leaky_0.1(scale[n] * acc + bias[n]); for a fused 2x2/s2
// max-pool the quad of pixels {(r, c), (r, c+1), (r+1, c), (r+1, c+1)} are lanes
// {l, l^1, l^8, l^8^1} of one warp and are reduced with two shuffles; rounded
// to bf16 (nearest-even) and stored to the tile's region buffer (octet-planar),
// the cut tensor, or the NHWC output.
#include <cuda_bf16.h>

#include "sched.cuh"

namespace {

constexpr int kEpiGroups = 2;           // epilogue warpgroups, each over all 128 TMEM lanes
constexpr int kEpiWarps = 4 * kEpiGroups;
constexpr int kEpiThreads = kEpiWarps * 32;
constexpr int kProducerWarp = kEpiWarps;
constexpr int kMmaWarp = kEpiWarps + 1;
constexpr int kPubWarp = kEpiWarps + 2;
constexpr int kGatherWarp = kEpiWarps + 3;
constexpr int kThreads = (kEpiWarps + 4) * 32;
constexpr int kAStages = 2;
constexpr int kQDepth = 4;
constexpr int kAStageBytes = MAFAT_A_STAGE_BYTES;   // one A halo box, multiple of 1024
constexpr int kBPieceBytes = MAFAT_B_PIECE_BYTES;   // one of two weight buffers
constexpr int kTmemCols = 512;        // two accumulators of up to 256 fp32 columns
constexpr int kAccStride = 256;

// shared-memory map (offsets from a 1024-aligned base)
constexpr int kBarAFull = 0;
constexpr int kBarAEmpty = kBarAFull + kAStages;
constexpr int kBarBFull = kBarAEmpty + kAStages;   // a weight piece has landed in buffer b
constexpr int kBarBEmpty = kBarBFull + 2;          // the MMAs reading buffer b's previous piece are done
constexpr int kBarAccFull = kBarBEmpty + 2;
constexpr int kBarAccEmpty = kBarAccFull + 2;
constexpr int kBarQFull = kBarAccEmpty + 2;
constexpr int kBarQEmpty = kBarQFull + kQDepth;
constexpr int kBarDone = kBarQEmpty + kQDepth;
constexpr int kBarEpiDone = kBarDone + 1;          // every epilogue thread has stored item e (slot e % 2)
constexpr int kBarPubDone = kBarEpiDone + 2;       // the publisher has published item e (slot e % 2)
constexpr int kBarRawFull = kBarPubDone + 2;       // raw NHWC rows have landed in A stage s (gather items)
constexpr int kBarMidFull = kBarRawFull + kAStages; // chain items: the 3x3's bf16 result is in TMEM (buffer b)
constexpr int kNumBars = kBarMidFull + 2;
constexpr int kOffRec = 256;                        // kQDepth epilogue records
constexpr int kRecStride = 160;
constexpr int kOffQItems = kOffRec + kQDepth * kRecStride;
constexpr int kOffTmem = kOffQItems + 4 * kQDepth;
constexpr int kOffBroken = kOffTmem + 4;
constexpr int kOffA = 1024;
constexpr int kOffB = kOffA + kAStages * kAStageBytes;
constexpr int kSbSlotBytes = 2 * MAFAT_MAX_NBLK * 4;  // scale then bias of one item's channels
constexpr int kOffSb = kOffB + 2 * kBPieceBytes;
constexpr int kSmemUsed = kOffSb + 2 * kSbSlotBytes;
constexpr int kSmemBytes = kSmemUsed + 1024;  // slack for aligning the base
static_assert(kNumBars * 8 <= kOffRec, "barrier area");
static_assert(kOffBroken + 4 <= kOffA, "queue area");
static_assert(kSmemBytes <= 232448, "shared memory");

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

// The lane with el = 1 (one lane of the converged warp, from elect_one) adds 2 x bytes to
// the current phase of bar's expected transactions (without arriving) and copies bytes of
// scale and of bias into the slot (bias at slot + MAFAT_MAX_NBLK floats), completing on
// bar.  No branch on the lane: the MMA warp stays converged.
__device__ __forceinline__ void sb_load_el(uint32_t el, uint32_t bar, uint32_t slot, const float* scale,
                                           const float* bias, uint32_t bytes) {
    asm volatile(
        "{\n\t.reg .pred e;\n\t.reg .b32 tx;\n\t"
        "setp.ne.b32 e, %6, 0;\n\t"
        "add.u32 tx, %4, %4;\n\t"
        "@e mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], tx;\n\t"
        "@e cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%1], [%2], %4, [%0];\n\t"
        "@e cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%5], [%3], %4, [%0];\n\t}" ::"r"(bar),
        "r"(slot), "l"(scale), "l"(bias), "r"(bytes), "r"(slot + (uint32_t)(MAFAT_MAX_NBLK * 4)), "r"(el)
        : "memory");
}

// The same for a chain item: the 3x3's n1 channels at slot offset 0 and the chained 1x1's n2
// at slot offset n1 (scale and bias halves alike), all completing on bar.
__device__ __forceinline__ void sb_load2_el(uint32_t el, uint32_t bar, uint32_t slot, const float* scale1,
                                            const float* bias1, uint32_t bytes1, const float* scale2,
                                            const float* bias2, uint32_t bytes2) {
    asm volatile(
        "{\n\t.reg .pred e;\n\t.reg .b32 tx;\n\t"
        "setp.ne.b32 e, %11, 0;\n\t"
        "add.u32 tx, %4, %7;\n\t"
        "add.u32 tx, tx, tx;\n\t"
        "@e mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], tx;\n\t"
        "@e cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%1], [%2], %4, [%0];\n\t"
        "@e cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%8], [%3], %4, [%0];\n\t"
        "@e cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%9], [%5], %7, [%0];\n\t"
        "@e cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%10], [%6], %7, [%0];\n\t}" ::"r"(bar),
        "r"(slot), "l"(scale1), "l"(bias1), "r"(bytes1), "l"(scale2), "l"(bias2), "r"(bytes2),
        "r"(slot + (uint32_t)(MAFAT_MAX_NBLK * 4)), "r"(slot + bytes1), "r"(slot + (uint32_t)(MAFAT_MAX_NBLK * 4) + bytes1),
        "r"(el)
        : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(bar), "r"(parity)
        : "memory");
    return done != 0;
}

// Bounded wait on a pipeline barrier phase.  These waits depend only on work
// inside the CTA, so they always finish unless something is broken; as a safety
// net the first one to run out records MAFAT_DEV_PIPE and marks the CTA broken,
// after which every pipeline wait of the CTA gives up after 1 ms, so the launch
// still ends in bounded time (with garbage results and an error status).
__device__ __forceinline__ void mbar_wait(uint32_t bar, uint32_t parity, uint32_t* ctr, int64_t limit_ns,
                                          volatile int* broken, uint32_t sleep_ns = 0) {
    if (mbar_try_wait(bar, parity)) return;
    const int64_t lim = *broken ? 1000000LL : limit_ns;
    uint64_t t0 = mafat_dev::globaltimer_ns();
    for (uint32_t i = 1;; ++i) {
        // warps whose waits are off the critical path back off, leaving issue slots of
        // their sub-partition to the MMA issuer
        if (sleep_ns) __nanosleep(sleep_ns);
        if (mbar_try_wait(bar, parity)) return;
        if ((i & 255u) == 0u && (int64_t)(mafat_dev::globaltimer_ns() - t0) > lim) {
            mafat_dev::record_status(ctr, MAFAT_DEV_PIPE);
            *broken = 1;
            return;
        }
    }
}

// The MMA warp's wait.  Measured on GB300: a polling loop written in C++ anywhere in
// the MMA issue loop (even one whose exit is a warp vote) more than halves the MMA
// issue rate of the whole loop, while the same loop inside one asm statement costs
// nothing.  So the poll, with its deadline on %globaltimer, lives in the asm, and a
// timeout is recorded by every lane alike (no branch on the lane).  The lanes poll in
// step, so the result needs no vote: a vote and a warp barrier after every wait cost the
// first layer ~7 % of its MMA phase.
__device__ __forceinline__ void mbar_wait_mma(uint32_t bar, uint32_t parity, uint32_t* ctr, int64_t limit_ns,
                                              volatile int* broken) {
    const uint64_t lim = (uint64_t)(*broken ? 1000000LL : limit_ns);
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred P1, P2;\n\t.reg .u64 dl, t;\n\t"
        "mov.u32 %0, 1;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 P1, [%1], %2;\n\t"
        "@P1 bra MW_DONE_%=;\n\t"
        "mov.u64 dl, %%globaltimer;\n\t"
        "add.u64 dl, dl, %3;\n\t"
        "MW_POLL_%=:\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 P1, [%1], %2;\n\t"
        "@P1 bra MW_DONE_%=;\n\t"
        "mov.u64 t, %%globaltimer;\n\t"
        "setp.lt.u64 P2, t, dl;\n\t"
        "@P2 bra MW_POLL_%=;\n\t"
        "mov.u32 %0, 0;\n\t"
        "MW_DONE_%=:\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity), "l"(lim)
        : "memory");
    if (ok == 0u) {  // every lane polled the same barrier in step: ok is warp-uniform
        mafat_dev::record_status(ctr, MAFAT_DEV_PIPE);
        *broken = 1;
    }
}

// An arrive on bar by the lane with el = 1 (from elect_one).
__device__ __forceinline__ void mbar_arrive_el(uint32_t el, uint32_t bar) {
    asm volatile(
        "{\n\t.reg .pred e;\n\tsetp.ne.b32 e, %1, 0;\n\t"
        "@e mbarrier.arrive.shared::cta.b64 _, [%0];\n\t}" ::"r"(bar), "r"(el)
        : "memory");
}

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap* map, int c0, int c1, int c2, int c3,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int c0, int c1, int c2,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Broadcast from lane 0: marks the value warp-uniform for the compiler.
__device__ __forceinline__ int wu(int v) { return __shfl_sync(0xffffffffu, v, 0); }

// Warp-wide forms for the MMA warp, whose 32 lanes all run the issue loop (so that
// descriptors stay warp-uniform): elect.sync picks one lane, the same lane every time
// since the warp is converged, to issue the operation.
__device__ __forceinline__ void tc_commit_warp(uint32_t bar) {
    asm volatile(
        "{\n\t.reg .pred e;\n\t"
        "elect.sync _|e, 0xffffffff;\n\t"
        "@e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n\t}" ::"r"(bar)
        : "memory");
}

// tcgen05.commit and the A-in-tensor-memory MMA with the issuing lane chosen beforehand
// (el from elect_one), as mma_el.
__device__ __forceinline__ void tc_commit_el(uint32_t el, uint32_t bar) {
    asm volatile(
        "{\n\t.reg .pred e;\n\t"
        "setp.ne.b32 e, %0, 0;\n\t"
        "@e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%1];\n\t}" ::"r"(el), "r"(bar)
        : "memory");
}
__device__ __forceinline__ void mma_tmem_a_el(uint32_t el, uint32_t d_tmem, uint32_t a_tmem, uint32_t b_lo,
                                              uint32_t b_hi, uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p, e;\n\t.reg .b64 db;\n\t"
        "setp.ne.b32 e, %0, 0;\n\t"
        "setp.ne.b32 p, %6, 0;\n\t"
        "mov.b64 db, {%3, %4};\n\t"
        "@e tcgen05.mma.cta_group::1.kind::f16 [%1], [%2], db, %5, p;\n\t}" ::"r"(el), "r"(d_tmem),
        "r"(a_tmem), "r"(b_lo), "r"(b_hi), "r"(idesc), "r"(accumulate));
}

// Shared-memory matrix descriptor, no swizzle: start >> 4 in bits 0-13, LBO >> 4
// in 16-29, SBO >> 4 in 32-45, descriptor version 1 in bits 46-47, layout 0.  For
// the K-major no-swizzle layout LBO is the stride between the two core matrices
// along K and SBO the stride between 8-row groups along M / N (checked by
// mafat_diag_umma against a float64 product).
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t k_stride, uint32_t mn_stride) {
    const uint32_t lbo = k_stride, sbo = mn_stride;
    uint64_t d = (uint64_t)((addr & 0x3FFFFu) >> 4);
    d |= (uint64_t)((lbo & 0x3FFFFu) >> 4) << 16;
    d |= (uint64_t)((sbo & 0x3FFFFu) >> 4) << 32;
    d |= (uint64_t)1 << 46;
    return d;
}

// Instruction descriptor of kind::f16: fp32 accumulator (bits 4-5 = 1), bf16 A and
// B (bits 7-9 = 1, 10-12 = 1), both K-major, N >> 3 in bits 17-22, M >> 4 in 24-28.
__device__ __forceinline__ uint32_t instr_desc_bf16(int n, int m) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

// One MMA whose A operand is in tensor memory (a_tmem: column of K elements 0..1 of lane 0;
// a K=16 step spans 8 columns, two bf16 per 32-bit column, lane = row of A), B in shared
// memory, issued by one elected lane of the converged warp.
__device__ __forceinline__ void mma_tmem_a(uint32_t d_tmem, uint32_t a_tmem, uint32_t b_lo, uint32_t b_hi,
                                           uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p, e;\n\t.reg .b64 db;\n\t"
        "elect.sync _|e, 0xffffffff;\n\t"
        "setp.ne.b32 p, %5, 0;\n\t"
        "mov.b64 db, {%2, %3};\n\t"
        "@e tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], db, %4, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "r"(b_lo), "r"(b_hi), "r"(idesc), "r"(accumulate));
}

// Store 16 consecutive 32-bit TMEM columns of this thread's lane (warp w reaches lanes
// 32(w%4)..+31), then wait until the stores are done.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15, %16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]),
        "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
        : "memory");
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// The MMA warp runs its loop on all 32 lanes and one elected lane issues each MMA
// (a lone lane in diverged code issues far slower).  The hot loop keeps descriptors
// as 32-bit halves: the low word holds
// start address >> 4 (bits 0-13) and LBO >> 4 (bits 16-29), and advancing an
// operand only adds 16-byte units to it; the high word (SBO, version, swizzle
// mode) is fixed per operand.
__device__ __forceinline__ void mma_lo(uint32_t d_tmem, uint32_t a_lo, uint32_t a_hi, uint32_t b_lo, uint32_t b_hi,
                                       uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p, e;\n\t.reg .b64 da, db;\n\t"
        "elect.sync _|e, 0xffffffff;\n\t"
        "setp.ne.b32 p, %6, 0;\n\t"
        "mov.b64 da, {%1, %2};\n\t"
        "mov.b64 db, {%3, %4};\n\t"
        "@e tcgen05.mma.cta_group::1.kind::f16 [%0], da, db, %5, p;\n\t}" ::"r"(d_tmem),
        "r"(a_lo), "r"(a_hi), "r"(b_lo), "r"(b_hi), "r"(idesc), "r"(accumulate));
}

// Picks one lane of the converged warp (the same lane on every call) as 1, the others 0.
__device__ __forceinline__ uint32_t elect_one() {
    uint32_t el;
    asm volatile("{\n\t.reg .pred e;\n\telect.sync _|e, 0xffffffff;\n\tselp.u32 %0, 1, 0, e;\n\t}" : "=r"(el));
    return el;
}

// mma_lo with the issuing lane chosen beforehand (el from elect_one, taken once when the
// MMA warp starts): measured on GB300, an elect.sync per MMA cost ~3.5 % of the one-frame
// launch against this form.
__device__ __forceinline__ void mma_el(uint32_t el, uint32_t d_tmem, uint32_t a_lo, uint32_t a_hi, uint32_t b_lo,
                                       uint32_t b_hi, uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p, e;\n\t.reg .b64 da, db;\n\t"
        "setp.ne.b32 e, %0, 0;\n\t"
        "setp.ne.b32 p, %7, 0;\n\t"
        "mov.b64 da, {%2, %3};\n\t"
        "mov.b64 db, {%4, %5};\n\t"
        "@e tcgen05.mma.cta_group::1.kind::f16 [%1], da, db, %6, p;\n\t}" ::"r"(el), "r"(d_tmem),
        "r"(a_lo), "r"(a_hi), "r"(b_lo), "r"(b_hi), "r"(idesc), "r"(accumulate));
}

// 128-byte-swizzled, K-major B operand (weights packed so by the host): rows of
// 64 channels (128 bytes), 8-row atoms of 1024 bytes, SBO = 1024, one K=16 step =
// 32 bytes along the row.  Measured on GB300: when both operands change from one
// MMA to the next, no-swizzle operands cost ~2.4x the MMA time; with B swizzled
// the MMAs run at their own rate.
__device__ __forceinline__ uint32_t desc_hi_sw128(uint32_t sbo) {
    return ((sbo >> 4) & 0x3FFFu) | (1u << 14) | (2u << 29);
}
__device__ __forceinline__ uint32_t desc_lo_sw128(uint32_t addr) {
    return ((addr & 0x3FFFFu) >> 4) | (1u << 16);
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15}, [%16];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
        : "r"(taddr)
        : "memory");
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&h);
}
// Folded BN and leaky ReLU of two accumulator values with the packed fp32 instructions:
// z = s * acc + b (fma.rn per element) and 0.1 z (mul.rn per element), then
// max(z, 0.1 z) per element: the same roundings as the scalar form.
__device__ __forceinline__ void bn_leaky2(float s0, float s1, uint32_t a0, uint32_t a1, float b0, float b1, float& v0,
                                          float& v1) {
    float z0, z1, t0, t1;
    asm("{\n\t.reg .b64 s, a, b, z, t, c;\n\t"
        "mov.b64 s, {%4, %5};\n\t"
        "mov.b64 a, {%6, %7};\n\t"
        "mov.b64 b, {%8, %9};\n\t"
        "fma.rn.f32x2 z, s, a, b;\n\t"
        "mov.b64 c, {%10, %10};\n\t"
        "mul.rn.f32x2 t, z, c;\n\t"
        "mov.b64 {%0, %1}, z;\n\t"
        "mov.b64 {%2, %3}, t;\n\t}"
        : "=f"(z0), "=f"(z1), "=f"(t0), "=f"(t1)
        : "f"(s0), "f"(s1), "r"(a0), "r"(a1), "f"(b0), "f"(b1), "f"(0.1f));
    v0 = fmaxf(z0, t0);
    v1 = fmaxf(z1, t1);
}

__device__ __forceinline__ uint32_t max_bf16x2(uint32_t a, uint32_t b) {
    __nv_bfloat162 x = *reinterpret_cast<__nv_bfloat162*>(&a), y = *reinterpret_cast<__nv_bfloat162*>(&b);
    __nv_bfloat162 m = __hmax2(x, y);
    return *reinterpret_cast<uint32_t*>(&m);
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
          "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
          "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr)
        : "memory");
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// What the MMA issuer needs of an item, packed in 32-bit words that it reads with three
// 16-byte shared-memory loads and broadcasts word by word (the read is on the MMA warp's
// path between items, while the tensor core keeps shared memory busy with its operands):
//   w[0] key: stage * 256 + channel block, identifies a resident weight set
//   w[1] sb: offset of the item's first channel in the scale / bias arrays
//   w[2] bytes of one weight blob
//   w[3] n_mid: MMA N of the item's (first) convolution
//   w[4] k | K steps per blob << 8 | blocks << 16 | paired << 24 | swizzled B << 25 | chain << 26 |
//        pixel pairs << 27 | per-block halos << 28
//   w[5] A box columns | rows << 16
//   w[6] input chunks | blobs per chunk << 16
//   w[7] blobs per weight piece | pieces << 16
//   w[8] flat stage: A box pixel of the item's first pixel + 1 (0: 16x8 blocks) | box pixels << 16
struct __align__(16) MmaRec {
    uint32_t w[12];
};

// What the MMA issuer needs of a chain item's chained 1x1 (N, input chunks, K steps per blob,
// swizzled blobs, blobs per piece, pieces, TMEM columns of its A operand and accumulator,
// blob elements, scale / bias offset).  Read from the queue slot only on the chain path.
struct __align__(8) ChainRec {
    int16_t n2, nch2, kst2, swz2, bpp2, np2, a_col, out_col;
    int32_t blob2, sb2;
};

// What the MMA issuer, the epilogue and the publisher need of an item, written into its
// queue slot by the producer (which has the work tables in registers anyway), so that
// none of them reads a work table from global memory on its critical path.
// What the gather warp needs of an item that reads raw NHWC rows (MAFAT_IN_GATHER).
struct __align__(8) GatherRec {
    int16_t on;              // 1: this item's A halo is built from raw rows by the gather warp,
                             // one pixel per 16-byte slot; 2: two pixels per slot (pixel pairs)
    int16_t c;               // channels of the input (1..7)
    int16_t raw_e;           // elements of one raw row in shared memory
    int16_t s0;              // element of the first halo pixel's channel 0 within a raw row
};

struct __align__(16) EpiRec {  // 16-byte aligned: written and read with 16-byte accesses
    __nv_bfloat16* out;      // output buffer of the task (frame and tile offset applied)
    int32_t x0, xlim;        // conv column of the item's block column; end of the task's columns
    int32_t y0, ylim;        // conv row of the item's first block row; end of the task's rows
    int32_t out_y0, out_x0;  // map position of output buffer pixel (0, 0)
    int32_t out_w, out_h;    // output buffer extent (pixels, after pooling)
    int16_t nbk;             // blocks of the item
    int16_t nby;             // per-block-halo item: block rows of its task (0: blocks stacked from y0)
    int32_t n_blk;           // output channels per item (accumulator columns per block)
    int32_t cout, ch_base;   // channels of the layer; first channel of the item
    int32_t flags;           // bit 0: fused max-pool, bit 1: NHWC output, bit 2: never published (test hook)
    int32_t done_ctr, extra_ctr;
    int16_t chain;           // 1: chain item (first pass turns the 3x3's result into the 1x1's A operand)
    int16_t n_mid;           // chain item: columns of the 3x3's accumulator
    int16_t a_col, out_col;  // chain item: TMEM columns of the 1x1's A operand and of its accumulator
    int16_t pitch;           // flat stage: row pitch of the region (pixels); 0: 16x8 blocks
    int16_t flat_by;         // flat stage: the item's first block in the region; per-block-halo item:
                             // its first block's index in the task's column-major block order
};

// A queue slot: the record of one item, in parts, so that every role copies only its own.
struct ItemRec {
    EpiRec epi;
    MmaRec mma;
    ChainRec chain;
    GatherRec gather;
};
static_assert(sizeof(ItemRec) <= kRecStride, "item record");
static_assert(kRecStride % 16 == 0 && offsetof(ItemRec, mma) % 16 == 0, "16-byte loads of the MMA record");

// Where one thread's epilogue results go: its pixel's element offset in the
// output buffer (octet-planar: offset inside an 8-channel plane; NHWC: offset
// of channel 0), the plane stride, and whether this lane stores at all.
struct EpiDst {
    __nv_bfloat16* out;
    uint32_t pix, plane;  // element offsets within the output buffer (a frame's region: < 2^31)
    int nhwc, cout, pool;
    bool store;
};

// Epilogue of NC accumulator columns (output channels ch0 .. ch0+NC-1, NC = 16 or 32)
// of one pixel per thread: folded BN, leaky ReLU 0.1 (as max(z, 0.1 z), the same value),
// bf16 (nearest-even), 16-byte stores per octet of channels.
//
// A fused 2x2 max-pool reduces the window {(r, c), (r, c+1), (r+1, c), (r+1, c+1)},
// lanes {l, l^1, l^8, l^9}, on packed bf16 pairs (rounding is monotonic, so the max of
// rounded values is the rounded max) in two exchange rounds that each halve the octets a
// lane holds: with the partner lane^1, a lane keeps octets 2m + (l & 1) and sends the
// others; with lane^8, it keeps every other remaining octet.  Every shuffle carries data
// both lanes need, and each lane of the window ends with its own octet(s) of the pooled
// pixel to store (two octets: both lanes l and l^8 end with the same one; one stores).
template <int NC>
__device__ __forceinline__ void epi_chunk(uint32_t taddr, const float* sc, const float* bi, int ch0,
                                          const EpiDst& d, int lane) {
    static_assert(NC == 16 || NC == 32, "unit width");
    constexpr int NO = NC / 8;  // octets
    uint32_t raw[NC];
    if constexpr (NC == 32)
        tmem_ld32(taddr, raw);
    else
        tmem_ld16(taddr, raw);
    uint32_t pk[NC / 2];
#pragma unroll
    for (int i = 0; i < NC; i += 4) {
        const float4 s4 = *reinterpret_cast<const float4*>(sc + i);  // shared memory, same address
        const float4 b4 = *reinterpret_cast<const float4*>(bi + i);  // for the whole warp
        float v[4];
        bn_leaky2(s4.x, s4.y, raw[i], raw[i + 1], b4.x, b4.y, v[0], v[1]);
        bn_leaky2(s4.z, s4.w, raw[i + 2], raw[i + 3], b4.z, b4.w, v[2], v[3]);
        pk[i / 2] = pack_bf16x2(v[0], v[1]);
        pk[i / 2 + 1] = pack_bf16x2(v[2], v[3]);
    }
    if (!d.pool) {
        if (!d.store) return;
#pragma unroll
        for (int o = 0; o < NO; ++o) {
            const int ch = ch0 + 8 * o;
            if (ch >= d.cout) break;  // channels past cout belong to the zero-padded MMA N
            const uint4 w = make_uint4(pk[4 * o], pk[4 * o + 1], pk[4 * o + 2], pk[4 * o + 3]);
            __nv_bfloat16* p = d.out + (d.nhwc ? d.pix + (uint32_t)ch : (uint32_t)(ch >> 3) * d.plane + d.pix);
            *reinterpret_cast<uint4*>(p) = w;
        }
        return;
    }
    const bool h0 = (lane & 1) != 0, h3 = (lane & 8) != 0;
    // first exchange, partner lane ^ 1: keep octet 2m + h0 of each pair (2m, 2m + 1)
    uint32_t r1[NC / 4];
#pragma unroll
    for (int m = 0; m < NO / 2; ++m)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const uint32_t lo = pk[8 * m + j], hi = pk[8 * m + 4 + j];
            const uint32_t got = __shfl_xor_sync(0xffffffffu, h0 ? lo : hi, 1);
            r1[4 * m + j] = max_bf16x2(h0 ? hi : lo, got);
        }
    if constexpr (NO == 4) {
        // second exchange, partner lane ^ 8: keep octet 2 * h3 + h0
        uint32_t r2[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const uint32_t lo = r1[j], hi = r1[4 + j];
            const uint32_t got = __shfl_xor_sync(0xffffffffu, h3 ? lo : hi, 8);
            r2[j] = max_bf16x2(h3 ? hi : lo, got);
        }
        const int ch = ch0 + 8 * (2 * (int)h3 + (int)h0);
        if (!d.store || ch >= d.cout) return;
        __nv_bfloat16* p = d.out + (d.nhwc ? d.pix + (uint32_t)ch : (uint32_t)(ch >> 3) * d.plane + d.pix);
        *reinterpret_cast<uint4*>(p) = make_uint4(r2[0], r2[1], r2[2], r2[3]);
    } else {
        // two octets: the second exchange is a plain max with lane ^ 8, and lanes with h3 set leave the store
#pragma unroll
        for (int j = 0; j < 4; ++j) r1[j] = max_bf16x2(r1[j], __shfl_xor_sync(0xffffffffu, r1[j], 8));
        const int ch = ch0 + 8 * (int)h0;
        if (!d.store || h3 || ch >= d.cout) return;
        __nv_bfloat16* p = d.out + (d.nhwc ? d.pix + (uint32_t)ch : (uint32_t)(ch >> 3) * d.plane + d.pix);
        *reinterpret_cast<uint4*>(p) = make_uint4(r1[0], r1[1], r1[2], r1[3]);
    }
}

// Sixteen TMEM lanes from `taddr` x 32 columns in the 16x256b shape (then wait): lane l of the
// warp gets, for column group g = 0..3, v[4g + e] = column 8g + 2 (l % 4) + (e & 1) of TMEM lane
// l / 4 (e < 2) or l / 4 + 8 (e >= 2) counted from taddr's lane (pinned on GB300 by a probe that
// wrote lane << 8 | column into every cell).
__device__ __forceinline__ void tmem_ld16x256_x4(uint32_t taddr, uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.16x256b.x4.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15}, [%16];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
        : "r"(taddr)
        : "memory");
}

// Epilogue of one block x 32 accumulator columns (channels ch0 .. ch0 + 31) with the fused 2x2
// max-pool, read in the 16x256b shape so that both rows of a pool window sit in one lane: the
// warp's quarter holds conv rows 4 wq .. 4 wq + 3 of the block (TMEM lane = 8 row + column), and
// its two loads (lanes +0 and +16) give lane l the pixels (2h, l / 4) and (2h + 1, l / 4) of
// load h, channels 8g + 2 (l % 4) + {0, 1}.  Folded BN, leaky ReLU and bf16 rounding as in
// epi_chunk, the vertical max in the lane, then one exchange with lane l ^ 4 (the next column):
// a lane of an even column keeps pooled row 0 of its quarter, one of an odd column row 1.  Each
// lane then stores 4 bytes (two channels) of each of its pooled pixel's four octets.
struct EpiPoolDst {
    __nv_bfloat16* out;
    uint32_t pix, plane;  // element offset of the pooled pixel (NHWC: of its channel 0); octet plane
    int nhwc, cout;
    bool store;
};
__device__ __forceinline__ void epi_pool32(uint32_t taddr, const float* sc, const float* bi, int ch0,
                                           const EpiPoolDst& d, int lane) {
    uint32_t raw0[16], raw1[16];
    tmem_ld16x256_x4(taddr, raw0);
    tmem_ld16x256_x4(taddr + (16u << 16), raw1);
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
    const int q2 = 2 * (lane & 3);
    uint32_t pv0[4], pv1[4];  // per column group: bf16x2 of channels 8g + q2, + 1 after the vertical max
#pragma unroll
    for (int g = 0; g < 4; ++g) {
        const float2 s = *reinterpret_cast<const float2*>(sc + 8 * g + q2);  // shared memory
        const float2 c = *reinterpret_cast<const float2*>(bi + 8 * g + q2);
        float a0, a1, b0, b1;
        bn_leaky2(s.x, s.y, raw0[4 * g], raw0[4 * g + 1], c.x, c.y, a0, a1);
        bn_leaky2(s.x, s.y, raw0[4 * g + 2], raw0[4 * g + 3], c.x, c.y, b0, b1);
        pv0[g] = max_bf16x2(pack_bf16x2(a0, a1), pack_bf16x2(b0, b1));
        bn_leaky2(s.x, s.y, raw1[4 * g], raw1[4 * g + 1], c.x, c.y, a0, a1);
        bn_leaky2(s.x, s.y, raw1[4 * g + 2], raw1[4 * g + 3], c.x, c.y, b0, b1);
        pv1[g] = max_bf16x2(pack_bf16x2(a0, a1), pack_bf16x2(b0, b1));
    }
    const bool odd = ((lane >> 2) & 1) != 0;
    uint32_t res[4];
#pragma unroll
    for (int g = 0; g < 4; ++g) {
        const uint32_t got = __shfl_xor_sync(0xffffffffu, odd ? pv0[g] : pv1[g], 4);
        res[g] = max_bf16x2(odd ? pv1[g] : pv0[g], got);
    }
    if (!d.store) return;
#pragma unroll
    for (int g = 0; g < 4; ++g) {
        const int ch = ch0 + 8 * g;
        if (ch >= d.cout) break;  // channels past cout belong to the zero-padded MMA N
        __nv_bfloat16* p = d.out + (d.nhwc ? d.pix + (uint32_t)(ch + q2) : (uint32_t)(ch >> 3) * d.plane + d.pix + q2);
        *reinterpret_cast<uint32_t*>(p) = res[g];
    }
}

// Weight-buffer bookkeeping.  The producer and the MMA issuer each keep a copy and
// apply the same transitions to the same item sequence, so they agree without
// talking on which of the two buffers holds which weights.  A set that fits one
// piece stays resident in its buffer (key >= 0) across items that use it; larger
// sets stream through both buffers piece by piece.
struct WeightBufs {
    // two buffers as scalar fields: a runtime-indexed local array would live in
    // local memory, next to the MMA issue loop
    int key0 = -1, key1 = -1;        // resident set held by buffer b (-1: streamed piece or nothing)
    uint32_t loads0 = 0, loads1 = 0; // pieces loaded into buffer b so far
    int next = 0;                    // buffer of the next load
    bool held0 = false, held1 = false;  // MMA side: b holds a resident set that is not yet released
    __device__ __forceinline__ int resident(int k) const { return key0 == k ? 0 : (key1 == k ? 1 : -1); }
    __device__ __forceinline__ uint32_t loads(int b) const { return b ? loads1 : loads0; }
    __device__ __forceinline__ bool held(int b) const { return b ? held1 : held0; }
    __device__ __forceinline__ void set_loaded(int b, int k, bool hold) {
        if (b) {
            ++loads1;
            key1 = k;
            held1 = hold;
        } else {
            ++loads0;
            key0 = k;
            held0 = hold;
        }
    }
    __device__ __forceinline__ void release(int b) {
        if (b)
            held1 = false;
        else
            held0 = false;
    }
};

// L2 prefetch of this CTA's share (per bytes, computed on the host) of a buffer
// (16-byte aligned base), in bulk prefetches of at most 64 KB; the tail below 16 bytes
// is left out.
__device__ __forceinline__ void prefetch_l2_share(const void* base, int64_t bytes, int64_t per) {
    if (base == nullptr || bytes <= 0) return;
    int64_t off = (int64_t)blockIdx.x * per;
    const int64_t end = min(bytes, off + per);
    for (; off < end; off += 65536) {
        const uint32_t n = (uint32_t)min((int64_t)65536, end - off) & ~15u;
        if (n == 0) break;
        asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"((const char*)base + off), "r"(n) : "memory");
    }
}

// ----------------------------------------------------------------------------- MMA warp
// State of the MMA warp that lives across items.
struct MmaState {
    WeightBufs wb;
    uint32_t a_cnt;                 // A halo stages consumed
    uint32_t sbase;                 // shared-memory base (warp-uniform)
    uint32_t* ctr;
    int64_t pipe_limit;
    volatile int* broken;
    unsigned long long* trace;
    uint32_t el;                    // 1 on the lane that issues tensor-core operations
    __device__ __forceinline__ uint32_t bar(int i) const { return sbase + (uint32_t)(i * 8); }
};

// One item's MMA parameters, all warp-uniform.
struct MmaJob {
    uint32_t d_tmem, idesc;
    uint32_t a_plane, a_row, a_step, blk16;  // A: octet-plane and row strides (bytes), K step and block (16-B units)
    uint32_t a_off16;                        // A: first pixel of the item in the box (16-B units; flat stages)
    uint32_t b_hi, b_half, b_step, blob_bytes, n_blk;
    int k, cols_box, n_chunks, n_bsteps, bpp, P, G, key, ticket, cur_b;
    bool bswz;
    bool pp;   // paired form with pixel pairs: blob t is kernel row t (K halves at kx = 0 and 2)
    uint64_t wait_a, wait_b;
};

// Start consuming the next weight piece: release the buffer's previous resident set
// (its MMAs finish first), then wait for the piece.
__device__ __forceinline__ void mma_begin_piece(MmaState& s, MmaJob& j) {
    const int b = s.wb.next;
    s.wb.next ^= 1;
    if (s.wb.held(b)) {
        tc_commit_el(s.el, s.bar(kBarBEmpty + b));
        s.wb.release(b);
    }
    mbar_wait_mma(s.bar(kBarBFull + b), s.wb.loads(b) & 1u, s.ctr, s.pipe_limit, s.broken);
    s.wb.set_loaded(b, j.P == 1 ? j.key : -1, j.P == 1);
    tc_fence_after();
    j.cur_b = b;
}

// Low word of the B descriptor of the first blob of buffer b (start address in bits 0-13;
// a later blob of the buffer only adds its offset >> 4 to it).
__device__ __forceinline__ uint32_t b_lo_of(const MmaState& s, const MmaJob& j, int b) {
    const uint32_t addr = s.sbase + kOffB + (uint32_t)b * kBPieceBytes;
    return j.bswz ? desc_lo_sw128(addr) : (uint32_t)smem_desc(addr, j.b_half, 128u);
}

// All MMAs of one item, for KST K=16 steps per weight blob, NBK M blocks (sharing every
// B operand) and the paired-tap form (8 input channels, two taps per K step).  One
// instance per shape keeps every blob's KST x NBK MMAs one straight run of code: on
// GB300, MMAs separated by a runtime loop or a branch per MMA, or by a jump per blob into
// a large switch, issued at half the tensor core's rate or worse; so does an MMA that
// is issued predicated off (measured: a block-count-generic instance with absent
// blocks' MMAs predicated off doubled the MMA time of one-block items).  Between blobs
// the loop does as little as it can: the descriptors advance by adds, and one countdown
// marks the end of a weight piece.  Measured on GB300 with eight epilogue-like warps
// sharing the SM, a loop that rebuilt the B descriptor and tested the piece bounds
// twice per blob issued N=64 MMAs every ~87 cycles; this form every ~52 (the shared
// memory bound of a 128x64x16 MMA is ~49).
template <int KST, int NBK, bool PAIRED, bool TR>
__device__ __forceinline__ void mma_item(MmaState& s, MmaJob& j) {
    uint32_t accumulate = 0;
    int g = 0;                        // blob index within the weight set
    int rem = j.P > 1 ? j.bpp : j.G;  // blobs left in the current buffer
    uint32_t b_lo = b_lo_of(s, j, j.cur_b);
    const uint32_t blob16 = j.blob_bytes >> 4;
    const int taps = j.k * j.k;
    for (int c = 0; c < j.n_chunks; ++c) {
        const int as = (int)(s.a_cnt % kAStages);
        const uint64_t tw0 = (TR && s.trace) ? mafat_dev::globaltimer_ns() : 0;
        mbar_wait_mma(s.bar(kBarAFull + as), (s.a_cnt / kAStages) & 1u, s.ctr, s.pipe_limit, s.broken);
        if (TR && s.trace) {  // every lane stores (one value wins): no branch on the lane
            const uint64_t tw1 = mafat_dev::globaltimer_ns();
            if (c > 0)
                j.wait_a += tw1 - tw0;
            else
                mafat_dev::trace_put(s.trace, j.ticket, 6, tw1);
        }
        tc_fence_after();
        const uint32_t a_base = s.sbase + kOffA + (uint32_t)as * kAStageBytes;
        const uint64_t a_desc0 = smem_desc(a_base, j.a_plane, j.a_row);
        const uint32_t a_hi = (uint32_t)(a_desc0 >> 32);
        uint32_t a_lo = (uint32_t)a_desc0 + j.a_off16;  // tap (ky, kx) of the plain form: + ky * cols_box + kx
        int kx = 0;
        // paired form: offset (16-byte units) and column of tap 2t, advanced by two taps per blob;
        // with pixel pairs, the offset of kernel row t's slot kx = 0, advanced by a halo row
        const uint32_t a_base16 = (a_base & 0x3FFFFu) >> 4;
        uint32_t oa16 = 0, or16 = 0;
        int xa = 0;
        for (int t = 0; t < j.n_bsteps; ++t) {
            uint32_t a_lo_t, a_hi_t;
            if (PAIRED) {
                // taps (2t, 2t+1) as the two K halves: LBO = their distance (in the low word's
                // bits 16-29; the high word, SBO = one halo row, is the plain form's); for an odd
                // tap count (3x3: a 1x1 layer needs more than 8 input channels) the last blob
                // pairs zero weights with the last tap, the walk's current position, and both
                // halves read that tap (LBO 0)
                uint32_t pa, pb;
                if (2 * t + 1 < taps) {
                    pa = oa16;
                    pb = xa + 1 == j.k ? oa16 + (uint32_t)(j.cols_box - j.k + 1) : oa16 + 1u;
                } else {
                    pa = oa16;
                    pb = oa16;
                }
                // pixel pairs: the row's slots kx = 0 (taps 0, 1) and kx = 2 (tap 2, zero weights)
                pa = j.pp ? or16 : pa;
                pb = j.pp ? or16 + 2u : pb;
                or16 += (uint32_t)j.cols_box;
                a_lo_t = (a_base16 + pa) | ((pb - pa) << 16);
                a_hi_t = a_hi;
                oa16 += 2u;
                xa += 2;
                if (xa >= j.k) {  // paired stages are 3x3 (a 1x1 layer needs more than 8 channels)
                    xa -= j.k;
                    oa16 += (uint32_t)(j.cols_box - j.k);
                }
            } else {
                a_lo_t = a_lo;
                a_hi_t = a_hi;
            }
            {
                const uint32_t el = s.el;
#pragma unroll
                for (int q = 0; q < KST; ++q)
#pragma unroll
                    for (int b = 0; b < NBK; ++b)
                        mma_el(el, j.d_tmem + (uint32_t)b * j.n_blk,
                               a_lo_t + (uint32_t)q * j.a_step + (uint32_t)b * j.blk16, a_hi_t,
                               b_lo + (uint32_t)q * j.b_step, j.b_hi, j.idesc, q == 0 ? accumulate : 1u);
            }
            accumulate = 1;
            b_lo += blob16;
            if (!PAIRED) {
                ++a_lo;
                if (++kx == j.k) {
                    kx = 0;
                    a_lo += (uint32_t)(j.cols_box - j.k);
                }
            }
            ++g;
            if (--rem == 0) {
                // end of the buffer's blobs for this item: a streamed piece is released as soon
                // as its last blob has been issued, and the next piece (if any) is waited for;
                // a piece that ends with the chunk is followed only after the A stage is
                // released below, so that the producer can refill the stage meanwhile
                if (j.P > 1) tc_commit_el(s.el, s.bar(kBarBEmpty + j.cur_b));
                if (g < j.G && t + 1 < j.n_bsteps) {
                    const uint64_t tp0 = (TR && s.trace) ? mafat_dev::globaltimer_ns() : 0;
                    mma_begin_piece(s, j);
                    if (TR && s.trace) j.wait_b += mafat_dev::globaltimer_ns() - tp0;
                    rem = min(j.bpp, j.G - g);
                    b_lo = b_lo_of(s, j, j.cur_b);
                }
            }
        }
        tc_commit_el(s.el, s.bar(kBarAEmpty + as));
        ++s.a_cnt;
        if (rem == 0 && g < j.G) {
            const uint64_t tp0 = (TR && s.trace) ? mafat_dev::globaltimer_ns() : 0;
            mma_begin_piece(s, j);
            if (TR && s.trace) j.wait_b += mafat_dev::globaltimer_ns() - tp0;
            rem = min(j.bpp, j.G - g);
            b_lo = b_lo_of(s, j, j.cur_b);
        }
    }
}

// Widening of raw rows of c < 8 channels (other than the RGB fast path), slot by slot
// (idx = r * cols + x dealt to the lanes); out of line, as it is off the common path.  With
// pixel pairs (pp, c <= 4) slot x holds pixel x in its first 8 bytes and pixel x + 1 in the
// last 8.  The item's blocks have a halo of hr rows each, and their raw rows come block by
// block, blk_stride bytes apart.
__device__ __noinline__ void gather_generic(const uint8_t* raw_b, uint8_t* stage, int rows, int cols, int raw_e,
                                            int s0, int c, bool pp, int hr, int blk_stride, int lane) {
    uint4* dst = reinterpret_cast<uint4*>(stage);
    if (cols <= 0) return;  // only a record read after a pipeline wait ran out can hold this
    int r = 0, x = lane;
    while (x >= cols) {
        x -= cols;
        ++r;
    }
    for (int idx = lane; idx < rows * cols; idx += 32) {
        // widened row r is row r % hr of block r / hr, whose raw rows start blk_stride bytes apart
        const uint16_t* src = reinterpret_cast<const uint16_t*>(raw_b + (r / hr) * blk_stride) + (r % hr) * raw_e +
                              s0 + x * c;
        uint32_t w[4] = {0u, 0u, 0u, 0u};
        if (pp) {
#pragma unroll
            for (int ch = 0; ch < 4; ++ch)
                if (ch < c) {
                    w[ch >> 1] |= (uint32_t)src[ch] << (16 * (ch & 1));
                    w[2 + (ch >> 1)] |= (uint32_t)src[c + ch] << (16 * (ch & 1));
                }
        } else {
#pragma unroll
            for (int ch = 0; ch < 7; ++ch)
                if (ch < c) w[ch >> 1] |= (uint32_t)src[ch] << (16 * (ch & 1));
        }
        dst[idx] = make_uint4(w[0], w[1], w[2], w[3]);
        x += 32;
        while (x >= cols) {
            x -= cols;
            ++r;
        }
    }
}

// The chained 1x1 of a chain item: A = the 3x3's activated bf16 result in TMEM (columns
// acc + a_col .., 8 per K=16 step), B = the 1x1's weights streamed through the two
// buffers piece by piece (never resident), D = TMEM columns acc + out_col .., N = n2.  The
// K order is the 1x1's packed blob order: input chunk c, K step q = channels (c kst2 + q) 16 ...
__device__ __forceinline__ void mma_chain_1x1(MmaState& s, uint32_t acc, int n2, int nch2, int kst2, bool swz2,
                                              int bpp2, int np2, uint32_t blob_bytes2, int a_col, int out_col) {
    const uint32_t idesc = instr_desc_bf16(n2, 128);
    const uint32_t b_half = (uint32_t)n2 * 16u;
    const uint32_t b_hi = swz2 ? desc_hi_sw128(1024u) : (uint32_t)(smem_desc(0u, b_half, 128u) >> 32);
    const uint32_t b_step = swz2 ? 2u : 2u * (b_half >> 4);
    const uint32_t blob16 = blob_bytes2 >> 4;
    const uint32_t d = acc + (uint32_t)out_col;
    uint32_t a = acc + (uint32_t)a_col;
    uint32_t accumulate = 0;
    int g = 0;
    for (int pc = 0; pc < np2; ++pc) {
        const int b = s.wb.next;
        s.wb.next ^= 1;
        if (s.wb.held(b)) {
            tc_commit_el(s.el, s.bar(kBarBEmpty + b));
            s.wb.release(b);
        }
        mbar_wait_mma(s.bar(kBarBFull + b), s.wb.loads(b) & 1u, s.ctr, s.pipe_limit, s.broken);
        s.wb.set_loaded(b, -1, false);
        tc_fence_after();
        const uint32_t addr = s.sbase + kOffB + (uint32_t)b * kBPieceBytes;
        uint32_t b_lo = swz2 ? desc_lo_sw128(addr) : (uint32_t)smem_desc(addr, b_half, 128u);
        const int nb = min(bpp2, nch2 - g);
        for (int k = 0; k < nb; ++k, ++g) {
            for (int q = 0; q < kst2; ++q) {
                mma_tmem_a_el(s.el, d, a, b_lo + (uint32_t)q * b_step, b_hi, idesc, accumulate);
                accumulate = 1u;
                a += 8u;
            }
            b_lo += blob16;
        }
        tc_commit_el(s.el, s.bar(kBarBEmpty + b));  // the piece is free once these MMAs are done
    }
}

// Gather of a 3x3 halo row from raw NHWC elements: the 16-byte slot x of a halo row holds
// elements S0 + C x .. S0 + C x + C - 1 of the raw row (the rest zero), or with pixel pairs
// (PP, C <= 4) those of pixel x in its first 8 bytes and of pixel x + 1 in its last 8.  One
// lane builds whole rows: the row's RAW_E elements come in as 16-byte loads, and with C, S0
// and the row length fixed at compile time every slot is a few byte permutes and one 16-byte
// store.  The rows of a halo are dealt to the lanes in turn.  Row r of the item is row r % 18
// of its block r / 18, whose raw rows start on a 128-byte boundary.
template <int C, int S0, int RAW_E, bool PP>
__device__ __forceinline__ void gather_rows(const uint8_t* raw, uint8_t* dst, int rows, int lane) {
    constexpr int kCols = MAFAT_BLK_COLS + 2;  // a gathered stage is a 3x3 convolution
    constexpr int kWords = RAW_E / 2;
    static_assert(RAW_E % 8 == 0 && S0 + C * (kCols + (PP ? 1 : 0)) <= RAW_E && (!PP || C <= 4), "raw row");
    constexpr int kHR = MAFAT_BLK_ROWS + 2;                          // halo rows of one block
    constexpr int kStride = (kHR * RAW_E * 2 + 127) / 128 * 128;     // raw bytes of one block
    for (int r = lane; r < rows; r += 32) {
        uint32_t w[kWords];
        const uint4* src = reinterpret_cast<const uint4*>(raw + (r / kHR) * kStride + (r % kHR) * RAW_E * 2);
#pragma unroll
        for (int q = 0; q < kWords / 4; ++q) {
            const uint4 v = src[q];
            w[4 * q] = v.x;
            w[4 * q + 1] = v.y;
            w[4 * q + 2] = v.z;
            w[4 * q + 3] = v.w;
        }
        uint4* out = reinterpret_cast<uint4*>(dst + (size_t)r * kCols * 16);
#pragma unroll
        for (int x = 0; x < kCols; ++x) {
            uint32_t o[4] = {0u, 0u, 0u, 0u};
#pragma unroll
            for (int px = 0; px < (PP ? 2 : 1); ++px)
#pragma unroll
                for (int ch = 0; ch < C; ++ch) {
                    const int i = S0 + C * (x + px) + ch;
                    const uint32_t e = (w[i >> 1] >> (16 * (i & 1))) & 0xFFFFu;
                    o[2 * px + (ch >> 1)] |= e << (16 * (ch & 1));
                }
            out[x] = make_uint4(o[0], o[1], o[2], o[3]);
        }
    }
}

// kChain: the instance for plans with chain stages; plans without them run the instance
// compiled without that path.  kTrace: the instance that records the per-item trace (plans
// made with trace = 1); the others carry none of its code (measured on GB300: with the
// trace code present but switched off, the 608x608 frame took 2.4 us longer).
template <bool kChain, bool kTrace>
__global__ void __launch_bounds__(kThreads, 1)
    mafat_tc_kernel(const __grid_constant__ MafatKParams p, const __grid_constant__ CUtensorMap in_map) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const uint32_t sbase = smem_u32(smem);
    volatile int* q_items = reinterpret_cast<volatile int*>(smem + kOffQItems);
    volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(smem + kOffTmem);
    volatile int* broken = reinterpret_cast<volatile int*>(smem + kOffBroken);
    ItemRec* recs = reinterpret_cast<ItemRec*>(smem + kOffRec);
    auto bar = [&](int i) { return sbase + (uint32_t)(i * 8); };

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int64_t pipe_limit = 4 * p.timeout_ns + 1000000000LL;
    unsigned long long* const trace = kTrace ? p.trace : nullptr;
    // the producer's first item record, in flight while the CTA sets up
    MafatItemDev it_first{};
    if (warp == kProducerWarp && lane == 0 && (int)blockIdx.x < p.n_items) it_first = p.items[blockIdx.x];

    if (threadIdx.x == 0) {
        for (int i = 0; i < kAStages; ++i) {
            mbar_init(bar(kBarAFull + i), 1);
            mbar_init(bar(kBarAEmpty + i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(kBarBFull + i), 1);
            mbar_init(bar(kBarBEmpty + i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(kBarAccFull + i), 1);
            mbar_init(bar(kBarAccEmpty + i), kEpiThreads);
        }
        for (int i = 0; i < kQDepth; ++i) {
            mbar_init(bar(kBarQFull + i), 1);
            mbar_init(bar(kBarQEmpty + i), kEpiWarps + 3);  // epilogue warps, MMA warp, publisher, gather warp
        }
        for (int i = 0; i < kAStages; ++i) mbar_init(bar(kBarRawFull + i), 1);
        for (int i = 0; i < 2; ++i) mbar_init(bar(kBarMidFull + i), kEpiThreads);
        mbar_init(bar(kBarDone), 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(kBarEpiDone + i), kEpiThreads);
            mbar_init(bar(kBarPubDone + i), 1);
        }
        *broken = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == kMmaWarp) {
        __syncwarp();  // .sync.aligned: the whole warp, converged
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         sbase + (uint32_t)kOffTmem),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == kProducerWarp) {
        // ------------------------------------------------------------ scheduler + TMA producer
        if (lane == 0) {
            // The input, the weights, the work tables and scale / bias are read from DRAM
            // once per run, mostly by loads that wait for them (the first layer's halos, the
            // first use of every weight set and table entry on each SM); fetching them into
            // L2 at once, spread over all CTAs, overlaps those DRAM latencies instead of
            // paying them item by item.
            for (int r = 0; r < MAFAT_PF_REGIONS; ++r) prefetch_l2_share(p.pf_ptr[r], p.pf_bytes[r], p.pf_per[r]);
            uint32_t a_cnt = 0, q_cnt = 0;
            WeightBufs wb;
            // dependency counters already seen at (or above) a target: items of one task
            // usually follow each other, so most items skip the round trip to L2
            int ok_idx0 = -1, ok_idx1 = -1, ok_tgt0 = 0, ok_tgt1 = 0;
            int ok_task = -1;  // the last task whose dependency list was found complete
            // A ticket is taken (and its item record loaded) at the end of the previous item,
            // once the A stage the new item will use is about to free: early enough to hide
            // the new item's loads behind the current MMAs, late enough that a CTA busy with a
            // long item does not hold work another CTA could start now.  After an item of a
            // stage with many items (lookahead) it is taken at once: every CTA has work then,
            // and the hand-out latency (atomic, record loads) is hidden behind the A stage's
            // release instead of added to it.
            // The first ticket is the CTA's index (the first gridDim.x items go out at once
            // anyway), its record loaded during the setup; later tickets come from the atomic
            // counter, offset by gridDim.x.
            int next = (int)blockIdx.x;
            MafatItemDev it_next = it_first;
            while (true) {
                const int ticket = next < p.n_items ? next : -1;
                const MafatItemDev it = it_next;
                if (ticket >= 0 && trace) {
                    mafat_dev::trace_put(trace, ticket, 0, mafat_dev::globaltimer_ns());
                    mafat_dev::trace_put(trace, ticket, 4, mafat_dev::smid());
                }
                MafatTaskDev tk;
                MafatStageDev st;
                if (ticket >= 0) {  // two independent loads (the item names its stage)
                    tk = p.tasks[it.task];
                    st = p.stages[it.stage];
                }
                // a flat stage's item starts at pixel 128 by of its region read row by row: its A box
                // starts at that pixel's row, the pixel being flat_off pixels into the box
                int y_lo = 0, flat_off = -1;
                if (ticket >= 0 && st.flat) {
                    const int p0 = it.by * 128;
                    y_lo = p0 / st.cols_box;
                    flat_off = p0 - y_lo * st.cols_box;
                }
                const int qs = (int)(q_cnt % kQDepth);
                mbar_wait(bar(kBarQEmpty + qs), ((q_cnt / kQDepth) & 1u) ^ 1u, p.ctr, pipe_limit, broken, 64);
                q_items[qs] = ticket;
                if (ticket >= 0) {
                    // the records are built in registers and stored whole (a few wide stores rather
                    // than one per field, on this single thread while the tensor core keeps the
                    // shared memory busy)
                    EpiRec rc{};
                    MmaRec& rm = recs[qs].mma;
                    GatherRec rg{};
                    rc.out = (__nv_bfloat16*)(tk.out_kind == MAFAT_BUF_USER_OUT ? p.user_out
                                              : tk.out_kind == MAFAT_BUF_CUT    ? p.cut
                                                                                : p.scratch) +
                             tk.out_off;
                    rc.x0 = tk.cx0 + it.bx * MAFAT_BLK_COLS;
                    rc.xlim = tk.cx0 + tk.cw;
                    rc.y0 = (flat_off >= 0 || st.blk_halo) ? tk.cy0 : tk.cy0 + it.by * MAFAT_BLK_ROWS;
                    rc.nby = (int16_t)(st.blk_halo ? tk.nby : 0);
                    rc.pitch = (int16_t)(flat_off >= 0 ? st.cols_box : 0);
                    rc.flat_by = it.by;
                    rc.ylim = tk.cy0 + tk.ch;
                    rc.out_y0 = tk.out_y0;
                    rc.out_x0 = tk.out_x0;
                    rc.out_w = tk.out_w;
                    rc.out_h = tk.out_h;
                    rc.nbk = (int16_t)it.nbk;
                    // what the epilogue stores: the item's own output, or a chain item's 1x1 output
                    const bool chain = kChain && st.chain;
                    rc.n_blk = chain ? st.c2_n_blk : st.n_blk;
                    rc.cout = chain ? st.c2_cout : st.cout;
                    rc.ch_base = chain ? 0 : it.nb * st.n_blk;
                    rc.flags = ((chain ? st.c2_pool : st.pool) ? 1 : 0) | (tk.out_nhwc ? 2 : 0) | ((it.flags & 1) ? 4 : 0);
                    rc.done_ctr = tk.done_ctr;
                    rc.extra_ctr = it.extra_ctr;
                    {
                        uint4* w = reinterpret_cast<uint4*>(rm.w);
                        w[0] = make_uint4((uint32_t)(tk.stage * 256 + it.nb), (uint32_t)(st.sb_off + it.nb * st.n_blk),
                                          (uint32_t)(st.blob_elems * 2), (uint32_t)st.n_blk);
                        w[1] = make_uint4((uint32_t)st.k | ((uint32_t)st.kst << 8) | ((uint32_t)it.nbk << 16) |
                                              ((uint32_t)st.paired << 24) | ((uint32_t)st.b_swz << 25) |
                                              ((uint32_t)chain << 26) | ((uint32_t)st.pix_pair << 27) |
                                              ((uint32_t)st.blk_halo << 28),
                                          (uint32_t)st.cols_box | ((uint32_t)st.rows_box << 16),
                                          (uint32_t)st.n_chunks | ((uint32_t)st.n_bsteps << 16),
                                          (uint32_t)st.bpp | ((uint32_t)st.n_pieces << 16));
                        w[2] = make_uint4((uint32_t)(flat_off + 1) | ((uint32_t)(st.rows_box * st.cols_box) << 16), 0u, 0u,
                                          0u);
                    }
                    rc.n_mid = (int16_t)st.n_blk;
                    rc.chain = (int16_t)chain;
                    if (chain) {
                        ChainRec rh{};
                        rh.n2 = (int16_t)st.c2_n_blk;
                        rh.nch2 = (int16_t)st.c2_n_chunks;
                        rh.kst2 = (int16_t)st.c2_kst;
                        rh.swz2 = (int16_t)st.c2_b_swz;
                        rh.bpp2 = (int16_t)st.c2_bpp;
                        rh.np2 = (int16_t)st.c2_n_pieces;
                        rh.a_col = (int16_t)st.chain_a_col;
                        rh.out_col = (int16_t)st.chain_out_col;
                        rh.blob2 = st.c2_blob_elems;
                        rh.sb2 = st.c2_sb_off;
                        recs[qs].chain = rh;
                        rc.a_col = (int16_t)st.chain_a_col;
                        rc.out_col = (int16_t)st.chain_out_col;
                    }
                    rg.on = 0;
                    if (tk.in_kind == MAFAT_BUF_USER_IN && st.in_mode == MAFAT_IN_GATHER) {
                        const int e_start = (tk.cx0 + it.bx * MAFAT_BLK_COLS - st.pad - tk.in_x0) * st.cin;
                        rg.on = (int16_t)(st.pix_pair ? 2 : 1);
                        rg.c = (int16_t)st.cin;
                        rg.raw_e = (int16_t)st.raw_e;
                        rg.s0 = (int16_t)(e_start - (e_start & ~7));
                    }
                    recs[qs].epi = rc;
                    recs[qs].gather = rg;
                }
                mbar_arrive(bar(kBarQFull + qs));  // release: the record is visible to the consumers
                ++q_cnt;
                if (ticket < 0) break;
                // the tensor map of the item's input (a table in global memory, cold after the
                // launch) into the TMA unit's descriptor cache while the item waits for its inputs
                if (tk.in_kind != MAFAT_BUF_USER_IN) {
                    const CUtensorMap* pm = tk.in_kind == MAFAT_BUF_CUT ? p.tmaps + p.cut_tmap : p.tmaps + tk.in_tmap;
                    asm volatile("prefetch.tensormap [%0];" ::"l"(pm) : "memory");
                }
                const int key = tk.stage * 256 + it.nb;
                const int P = st.n_pieces, G = st.n_chunks * st.n_bsteps;
                const uint32_t blob_bytes = (uint32_t)(st.blob_elems * 2);
                const uint16_t* wset = p.w_bf16 + st.w_off + (size_t)it.nb * (size_t)(st.set_bytes / 2);
                const bool resident = P == 1 && wb.resident(key) >= 0;
                // Loads go out in the order the MMA issuer consumes them: piece 0, then for
                // every chunk its A halo and the pieces that start inside it.  A piece goes
                // into the next buffer once the buffer's previous contents are released.
#define MAFAT_LOAD_PIECE(pc)                                                                                   \
    do {                                                                                                      \
        const int b_ = wb.next;                                                                               \
        wb.next ^= 1;                                                                                         \
        mbar_wait(bar(kBarBEmpty + b_), (wb.loads(b_) & 1u) ^ 1u, p.ctr, pipe_limit, broken, 64);             \
        const int nblob_ = min(st.bpp, G - (pc) * st.bpp);                                                    \
        const uint32_t bytes_ = (uint32_t)nblob_ * blob_bytes;                                                \
        mbar_arrive_expect_tx(bar(kBarBFull + b_), bytes_);                                                   \
        bulk_load(sbase + kOffB + b_ * kBPieceBytes, wset + (size_t)(pc) * st.bpp * st.blob_elems, bytes_,    \
                  bar(kBarBFull + b_));                                                                        \
        wb.set_loaded(b_, P == 1 ? key : -1, false);                                                          \
    } while (0)
                if (!resident) MAFAT_LOAD_PIECE(0);  // weights do not depend on other tiles: fetch first
                const CUtensorMap* map = tk.in_kind == MAFAT_BUF_USER_IN ? &in_map
                                         : tk.in_kind == MAFAT_BUF_CUT   ? p.tmaps + p.cut_tmap
                                                                         : p.tmaps + tk.in_tmap;
                const int c3 = tk.in_kind == MAFAT_BUF_SCRATCH ? 0 : tk.frame;
                const int in_mode = tk.in_kind == MAFAT_BUF_USER_IN ? st.in_mode : MAFAT_IN_PLANAR;
                const int px0 = tk.cx0 + it.bx * MAFAT_BLK_COLS - st.pad - tk.in_x0;  // first halo column
                const int x0 = px0 * 8;
                const int y0 = tk.cy0 + (flat_off >= 0 ? y_lo : it.by * MAFAT_BLK_ROWS) - st.pad - tk.in_y0;
                const uint32_t a_bytes = (uint32_t)(st.chunk8 * st.rows_box * st.cols_box * 16);
                bool waited = false;
                if (it.dep0 >= 0 && !(it.dep0 == ok_idx0 && it.dep0_target <= ok_tgt0)) {
                    mafat_dev::wait_counter(p.ctr, it.dep0, it.dep0_target, p.timeout_ns);
                    ok_idx0 = it.dep0;
                    ok_tgt0 = it.dep0_target;
                    waited = true;
                }
                if (it.dep1 >= 0 && !(it.dep1 == ok_idx1 && it.dep1_target <= ok_tgt1)) {
                    mafat_dev::wait_counter(p.ctr, it.dep1, it.dep1_target, p.timeout_ns);
                    ok_idx1 = it.dep1;
                    ok_tgt1 = it.dep1_target;
                    waited = true;
                }
                if (tk.dep_count > 0 && it.task != ok_task) {
                    mafat_dev::wait_dep_list(p.ctr, p.deps, tk.dep_first, tk.dep_count, p.timeout_ns);
                    ok_task = it.task;
                    waited = true;
                }
                if (waited) mafat_dev::fence_proxy_async_global();
                if (trace) mafat_dev::trace_put(trace, ticket, 1, mafat_dev::globaltimer_ns());
                int next_pc = 1;  // the next weight piece to load (piece 0 went first)
                for (int c = 0; c < st.n_chunks; ++c) {
                    const int as = (int)(a_cnt % kAStages);
                    const uint32_t a_dst = sbase + kOffA + as * kAStageBytes;
                    mbar_wait(bar(kBarAEmpty + as), ((a_cnt / kAStages) & 1u) ^ 1u, p.ctr, pipe_limit, broken, 64);
                    if (in_mode == MAFAT_IN_GATHER) {
                        // raw NHWC rows of each block's halo, from the 16-byte aligned element at
                        // or before the halo's first one, into the stage's tail block after block;
                        // the gather warp builds the halos from them and completes the stage's
                        // full barrier itself.  The item's blocks run down its task's block
                        // columns (column-major order from block it.by).
                        const int hr = MAFAT_BLK_ROWS + st.k - 1;
                        const uint32_t stride = (uint32_t)mafat_raw_blk_stride(st.k, st.raw_e);
                        uint32_t dst = a_dst + (uint32_t)mafat_raw_offset(st.rows_box, st.cols_box);
                        mbar_arrive_expect_tx(bar(kBarRawFull + as), (uint32_t)(it.nbk * hr * st.raw_e * 2));
                        int bxx = it.by / tk.nby, byy = it.by - bxx * tk.nby;
                        for (int j = 0; j < it.nbk; ++j, dst += stride) {
                            const int e = (tk.cx0 + bxx * MAFAT_BLK_COLS - st.pad - tk.in_x0) * st.cin;
                            tma_load_3d(dst, map, e & ~7, tk.cy0 + byy * MAFAT_BLK_ROWS - st.pad - tk.in_y0, c3,
                                        bar(kBarRawFull + as));
                            if (++byy == tk.nby) {
                                byy = 0;
                                ++bxx;
                            }
                        }
                    } else {
                        mbar_arrive_expect_tx(bar(kBarAFull + as), a_bytes);
                        tma_load_4d(a_dst, map, x0, y0, c * st.chunk8, c3, bar(kBarAFull + as));
                    }
                    ++a_cnt;
                    // the pieces that start inside this chunk (piece pc starts at blob pc * bpp);
                    // no division: on this single thread, a runtime modulo per blob cost ~1.5 us
                    // per chunk of a 3x3 256->512 item
                    while (next_pc < P && next_pc * st.bpp < (c + 1) * st.n_bsteps) {
                        MAFAT_LOAD_PIECE(next_pc);
                        ++next_pc;
                    }
                }
#undef MAFAT_LOAD_PIECE
                if (kChain && st.chain) {
                    // the chained 1x1's weights follow the 3x3's, streamed piece by piece (never
                    // resident), in the order the MMA issuer consumes them
                    const uint16_t* wset2 = p.w_bf16 + st.c2_w_off;
                    const int G2 = st.c2_n_chunks;  // one tap per blob
                    const uint32_t blob_bytes2 = (uint32_t)(st.c2_blob_elems * 2);
                    for (int pc = 0; pc < st.c2_n_pieces; ++pc) {
                        const int b_ = wb.next;
                        wb.next ^= 1;
                        mbar_wait(bar(kBarBEmpty + b_), (wb.loads(b_) & 1u) ^ 1u, p.ctr, pipe_limit, broken, 64);
                        const int nblob_ = min(st.c2_bpp, G2 - pc * st.c2_bpp);
                        const uint32_t bytes_ = (uint32_t)nblob_ * blob_bytes2;
                        mbar_arrive_expect_tx(bar(kBarBFull + b_), bytes_);
                        bulk_load(sbase + kOffB + b_ * kBPieceBytes, wset2 + (size_t)pc * st.c2_bpp * st.c2_blob_elems,
                                  bytes_, bar(kBarBFull + b_));
                        wb.set_loaded(b_, -1, false);
                    }
                }
                if (!st.lookahead)
                    mbar_wait(bar(kBarAEmpty + (int)(a_cnt % kAStages)), ((a_cnt / kAStages) & 1u) ^ 1u, p.ctr,
                              pipe_limit, broken, 64);
                next = (int)(atomicAdd(&p.ctr[MAFAT_CTR_TICKET], 1u) + gridDim.x);
                if (next < p.n_items) it_next = p.items[next];
            }
            // Drain: every copy issued has landed before the CTA may exit.
            for (uint32_t i = 0; i < kAStages && i < a_cnt; ++i) {
                uint32_t n = a_cnt - 1 - i;
                mbar_wait(bar(kBarAFull + (int)(n % kAStages)), (n / kAStages) & 1u, p.ctr, pipe_limit, broken);
            }
            for (int b = 0; b < 2; ++b)
                if (wb.loads(b) > 0)
                    mbar_wait(bar(kBarBFull + b), (wb.loads(b) - 1u) & 1u, p.ctr, pipe_limit, broken);
        }
        __syncwarp();
    } else if (warp == kMmaWarp) {
        // ------------------------------------------------------------ MMA issuer (whole warp)
        // Every value that feeds an MMA operand passes through wu() (a broadcast from lane
        // 0), so that the compiler knows it is warp-uniform.
        {
            MmaState ms;
            ms.a_cnt = 0;
            ms.sbase = (uint32_t)wu((int)sbase);
            ms.ctr = p.ctr;
            ms.pipe_limit = pipe_limit;
            ms.broken = broken;
            ms.trace = trace;
            ms.el = elect_one();
            const uint32_t tmem_u = (uint32_t)wu((int)tmem_base);
            uint32_t q_cnt = 0, acc_cnt = 0;
            uint32_t mid_ph0 = 0, mid_ph1 = 0;  // MidFull phases consumed, per accumulator buffer
            bool issued = false;
            while (true) {
                const int qs = (int)(q_cnt % kQDepth);
                mbar_wait_mma(ms.bar(kBarQFull + qs), (q_cnt / kQDepth) & 1u, p.ctr, pipe_limit, broken);
                const int ticket = wu(q_items[qs]);
                uint4 m0 = make_uint4(0u, 0u, 0u, 0u), m1 = m0, m2 = m0;
                if (ticket >= 0) {
                    const uint4* src = reinterpret_cast<const uint4*>(recs[qs].mma.w);
                    m0 = src[0];
                    m1 = src[1];
                    m2 = src[2];
                }
                const uint32_t w4 = (uint32_t)wu((int)m1.x);
                // release the slot once the record has been read (a chain item's slot is held until
                // its chained 1x1's fields have been read, on the chain path)
                const bool chain = kChain && ticket >= 0 && ((w4 >> 26) & 1u) != 0;
                if (!chain) mbar_arrive_el(ms.el, ms.bar(kBarQEmpty + qs));
                ++q_cnt;
                if (ticket < 0) break;
                MmaJob j;
                j.ticket = ticket;
                const uint32_t w5 = (uint32_t)wu((int)m1.y), w6 = (uint32_t)wu((int)m1.z), w7 = (uint32_t)wu((int)m1.w);
                const uint32_t w8 = (uint32_t)wu((int)m2.x);
                j.k = (int)(w4 & 0xFFu);
                j.cols_box = (int)(w5 & 0xFFFFu);
                j.n_blk = (uint32_t)wu((int)m0.w);
                j.n_chunks = (int)(w6 & 0xFFFFu);
                j.n_bsteps = (int)(w6 >> 16);
                j.bpp = (int)(w7 & 0xFFFFu);
                j.P = (int)(w7 >> 16);
                j.G = j.n_chunks * j.n_bsteps;
                j.key = wu((int)m0.x);
                j.blob_bytes = (uint32_t)wu((int)m0.z);
                j.a_plane = (w8 >> 16) * 16u;
                j.bswz = ((w4 >> 25) & 1u) != 0;
                j.pp = ((w4 >> 27) & 1u) != 0;
                const int kst = (int)((w4 >> 8) & 0xFFu), nbk = (int)((w4 >> 16) & 0xFFu), paired = (int)((w4 >> 24) & 1u);
                const int sb = wu((int)m0.y);
                j.cur_b = j.P == 1 ? ms.wb.resident(j.key) : -1;
                if (j.P > 1) {
                    // a streamed set takes both buffers: a resident set held in the one its
                    // second piece goes to is released now (its MMAs are long done), not when
                    // that piece is needed, so that the producer can load the piece meanwhile
                    const int o = ms.wb.next ^ 1;
                    if (ms.wb.held(o)) {
                        tc_commit_el(ms.el, ms.bar(kBarBEmpty + o));
                        ms.wb.release(o);
                    }
                }
                if (j.cur_b < 0) mma_begin_piece(ms, j);
                const int buf = (int)(acc_cnt & 1u);
                mbar_wait_mma(ms.bar(kBarAccEmpty + buf), ((acc_cnt >> 1) & 1u) ^ 1u, p.ctr, pipe_limit, broken);
                tc_fence_after();
                {
                    // the item's scale and bias go into the accumulator's slot (the epilogue of
                    // the slot's previous item is past it); the accumulator's full barrier then
                    // completes only once they have landed as well
                    const uint32_t slot = ms.sbase + (uint32_t)(kOffSb + buf * kSbSlotBytes);
                    if (chain) {
                        const int sb2 = wu(recs[qs].chain.sb2);
                        sb_load2_el(ms.el, ms.bar(kBarAccFull + buf), slot, p.scale + sb, p.bias + sb, j.n_blk * 4u,
                                       p.scale + sb2, p.bias + sb2, (uint32_t)wu(recs[qs].chain.n2) * 4u);
                    } else {
                        sb_load_el(ms.el, ms.bar(kBarAccFull + buf), slot, p.scale + sb, p.bias + sb, j.n_blk * 4u);
                    }
                }
                j.d_tmem = tmem_u + (uint32_t)(buf * kAccStride);
                j.idesc = instr_desc_bf16((int)j.n_blk, 128);
                // 8-pixel groups of a block: one halo row apart in a 16x8 block, adjacent in a flat one
                const int flat_off = (int)(w8 & 0xFFFFu) - 1;
                j.a_row = flat_off >= 0 ? 128u : (uint32_t)(j.cols_box * 16);
                j.b_half = j.n_blk * 16u;
                // next block (16-B units): one halo row apart in stacked 16x8 blocks; a block-halo apart
                // with per-block halos; 128 pixels on in a flat stage
                j.blk16 = flat_off >= 0             ? 128u
                          : ((w4 >> 28) & 1u) != 0u ? (uint32_t)((MAFAT_BLK_ROWS + j.k - 1) * j.cols_box)
                                                    : (uint32_t)(MAFAT_BLK_ROWS * j.cols_box);
                j.a_off16 = flat_off >= 0 ? (uint32_t)flat_off : 0u;
                j.a_step = 2u * (j.a_plane >> 4);                   // next K=16 step: two octet planes
                // B descriptor: 128-byte swizzled blobs (64 channels per row) or no-swizzle core matrices
                j.b_hi = j.bswz ? desc_hi_sw128(1024u) : (uint32_t)(smem_desc(0u, j.b_half, 128u) >> 32);
                j.b_step = j.bswz ? 2u : 2u * (j.b_half >> 4);
                j.wait_a = 0;
                j.wait_b = 0;
                // one jump per item into the instance for its shape
                switch ((paired << 8) | (kst << 4) | nbk) {
#define MAFAT_MMA_CASE(PA, K, B) \
    case ((PA) << 8) | ((K) << 4) | (B): mma_item<K, B, PA, kTrace>(ms, j); break;
                    MAFAT_MMA_CASE(0, 4, 1) MAFAT_MMA_CASE(0, 4, 2) MAFAT_MMA_CASE(0, 4, 3) MAFAT_MMA_CASE(0, 4, 4)
                    MAFAT_MMA_CASE(0, 2, 1) MAFAT_MMA_CASE(0, 2, 2) MAFAT_MMA_CASE(0, 2, 3) MAFAT_MMA_CASE(0, 2, 4)
                    MAFAT_MMA_CASE(0, 1, 1) MAFAT_MMA_CASE(0, 1, 2) MAFAT_MMA_CASE(0, 1, 3) MAFAT_MMA_CASE(0, 1, 4)
                    MAFAT_MMA_CASE(1, 1, 1) MAFAT_MMA_CASE(1, 1, 2) MAFAT_MMA_CASE(1, 1, 3) MAFAT_MMA_CASE(1, 1, 4)
                    MAFAT_MMA_CASE(1, 1, 5) MAFAT_MMA_CASE(1, 1, 6) MAFAT_MMA_CASE(1, 1, 7) MAFAT_MMA_CASE(1, 1, 8)
#undef MAFAT_MMA_CASE
                    default:  // a shape the planner never makes: fail loudly, never compute silently wrong
                        mafat_dev::record_status(p.ctr, MAFAT_DEV_PIPE);
                        *broken = 1;
                        break;
                }
                issued = true;
                if (trace) {
                    mafat_dev::trace_put(trace, ticket, 7, mafat_dev::globaltimer_ns());
                    mafat_dev::trace_put(trace, ticket, 8, j.wait_a);
                    mafat_dev::trace_put(trace, ticket, 9, j.wait_b);
                }
                if (chain) {
                    // chain item: the 3x3's accumulator goes to the epilogue, which writes its activated
                    // bf16 result back into TMEM; the chained 1x1 then runs from there
                    tc_commit_el(ms.el, ms.bar(kBarAccFull + buf));
                    const ChainRec ch = recs[qs].chain;
                    mbar_arrive_el(ms.el, ms.bar(kBarQEmpty + qs));  // the slot is no longer read
                    const uint32_t mph = buf ? mid_ph1++ : mid_ph0++;
                    mbar_wait_mma(ms.bar(kBarMidFull + buf), mph & 1u, p.ctr, pipe_limit, broken);
                    tc_fence_after();
                    mma_chain_1x1(ms, j.d_tmem, wu(ch.n2), wu(ch.nch2), wu(ch.kst2), wu(ch.swz2) != 0, wu(ch.bpp2),
                                  wu(ch.np2), (uint32_t)wu(ch.blob2 * 2), wu(ch.a_col), wu(ch.out_col));
                }
                tc_commit_el(ms.el, ms.bar(kBarAccFull + buf));
                ++acc_cnt;
            }
            // Every MMA this warp issued has completed before TMEM is released.
            if (issued) {
                tc_commit_el(ms.el, ms.bar(kBarDone));
                mbar_wait_mma(ms.bar(kBarDone), 0u, p.ctr, pipe_limit, broken);
            }
        }
        __syncwarp();
    } else if (warp == kPubWarp) {
        // ------------------------------------------------------------ publisher (warp 10)
        // An item is done once every epilogue thread has stored its share and fenced it
        // for the async proxy, then arrived on the item's EpiDone slot (release, CTA
        // scope).  The publisher's gpu-scope release reduction is cumulative over those
        // arrivals, so a consumer that acquires the counter sees every store; waiting for
        // the stores to reach L2 is this warp's job, not the epilogue warps'.
        if (lane == 0) {
            uint32_t q_cnt = 0, e_cnt = 0;
            while (true) {
                const int qs = (int)(q_cnt % kQDepth);
                mbar_wait(bar(kBarQFull + qs), (q_cnt / kQDepth) & 1u, p.ctr, pipe_limit, broken, 256);
                const int ticket = q_items[qs];
                int done_ctr = 0, extra_ctr = -1, flags = 0;
                if (ticket >= 0) {
                    done_ctr = recs[qs].epi.done_ctr;
                    extra_ctr = recs[qs].epi.extra_ctr;
                    flags = recs[qs].epi.flags;
                }
                mbar_arrive(bar(kBarQEmpty + qs));
                ++q_cnt;
                if (ticket < 0) break;
                const int es = (int)(e_cnt & 1u);
                mbar_wait(bar(kBarEpiDone + es), (e_cnt >> 1) & 1u, p.ctr, pipe_limit, broken, 32);
                if (!(flags & 4)) mafat_dev::publish_counters(p.ctr, done_ctr, extra_ctr);
                if (trace) mafat_dev::trace_put(trace, ticket, 3, mafat_dev::globaltimer_ns());
                mbar_arrive(bar(kBarPubDone + es));
                ++e_cnt;
            }
        }
        __syncwarp();
    } else if (warp == kGatherWarp) {
        // ------------------------------------------------------------ gather warp (warp 11)
        // For items whose input is a narrow NHWC image (fewer than 8 channels, e.g. RGB), the
        // producer lands raw rows of the image in the A stage's tail; this warp expands them
        // into the one-octet halo the MMAs read ([rows][cols][8 channels], channels c..7
        // zero), makes the stores visible to the tensor core (async proxy) and completes the
        // stage's full barrier.  It walks the item queue like the other consumers, counting A
        // stages as the producer and the MMA warp do.
        uint32_t q_cnt = 0, a_cnt = 0, raw_uses0 = 0, raw_uses1 = 0;
        while (true) {
            const int qs = (int)(q_cnt % kQDepth);
            mbar_wait(bar(kBarQFull + qs), (q_cnt / kQDepth) & 1u, p.ctr, pipe_limit, broken, 256);
            const int ticket = q_items[qs];
            GatherRec g{};
            int n_chunks = 0, rows_box = 0, rows = 0, cols = 0, hr = 0;
            if (ticket >= 0) {
                g = recs[qs].gather;
                const uint32_t w4 = recs[qs].mma.w[4], w5 = recs[qs].mma.w[5], w6 = recs[qs].mma.w[6];
                n_chunks = (int)(w6 & 0xFFFFu);
                rows_box = (int)(w5 >> 16);
                cols = (int)(w5 & 0xFFFFu);
                // a gathered item holds one halo of hr rows per block, block after block
                hr = MAFAT_BLK_ROWS + (int)(w4 & 0xFFu) - 1;
                rows = (int)((w4 >> 16) & 0xFFu) * hr;
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kBarQEmpty + qs));
            ++q_cnt;
            if (ticket < 0) break;
            if (g.on) {
                const int as = (int)(a_cnt % kAStages);
                const uint32_t uses = as ? raw_uses1++ : raw_uses0++;
                mbar_wait(bar(kBarRawFull + as), uses & 1u, p.ctr, pipe_limit, broken, 32);
                uint8_t* stage = smem + kOffA + as * kAStageBytes;
                // the raw rows start after the widened halos of the stage's largest item
                const uint8_t* raw_b = stage + mafat_raw_offset(rows_box, cols);
                if (g.on == 2 && g.c == 3 && g.raw_e == 40 && cols == MAFAT_BLK_COLS + 2) {
                    // RGB in pixel pairs: the common case, one instance per alignment of the first element
                    switch (g.s0) {
#define MAFAT_GATHER_CASE(S) \
    case S: gather_rows<3, S, 40, true>(raw_b, stage, rows, lane); break;
                        MAFAT_GATHER_CASE(0) MAFAT_GATHER_CASE(1) MAFAT_GATHER_CASE(2) MAFAT_GATHER_CASE(3)
                        MAFAT_GATHER_CASE(4) MAFAT_GATHER_CASE(5) MAFAT_GATHER_CASE(6) MAFAT_GATHER_CASE(7)
#undef MAFAT_GATHER_CASE
                        default: break;
                    }
                } else {
                    gather_generic(raw_b, stage, rows, cols, g.raw_e, g.s0, g.c, g.on == 2, hr,
                                   mafat_raw_blk_stride(hr - MAFAT_BLK_ROWS + 1, g.raw_e), lane);
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(kBarAFull + as));
            }
            a_cnt += (uint32_t)n_chunks;
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue (warps 0-7)
        // Warp w reads TMEM lanes 32*(w%4) .. +31 (conv rows 4*(w%4) .. +3 of a block);
        // the two warpgroups (h = w/4) take units of one block x 32 columns in turn.
        uint32_t q_cnt = 0, acc_cnt = 0;
        uint32_t full_ph0 = 0, full_ph1 = 0;  // AccFull phases consumed, per buffer (chain items take two)
        const int wq = warp & 3, h = warp >> 2;  // lane quarter, warpgroup
        const int r = wq * 4 + (lane >> 3);  // conv row within the block
        const int cc = lane & 7;             // conv column within the block
        while (true) {
            const int qs = (int)(q_cnt % kQDepth);
            mbar_wait(bar(kBarQFull + qs), (q_cnt / kQDepth) & 1u, p.ctr, pipe_limit, broken, 256);
            const int ticket = q_items[qs];
            EpiRec rc;
            if (ticket >= 0) rc = recs[qs].epi;
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kBarQEmpty + qs));
            ++q_cnt;
            if (ticket < 0) break;
            const int buf = (int)(acc_cnt & 1u);
            // completes once the item's MMAs are done and its scale / bias have landed
            mbar_wait(bar(kBarAccFull + buf), (buf ? full_ph1++ : full_ph0++) & 1u, p.ctr, pipe_limit, broken, 128);
            if (trace && threadIdx.x == 0) mafat_dev::trace_put(trace, ticket, 2, mafat_dev::globaltimer_ns());
            __syncwarp();
            tc_fence_after();

            const float* sc = reinterpret_cast<const float*>(smem + kOffSb + buf * kSbSlotBytes);
            const float* bi = sc + MAFAT_MAX_NBLK;
            const uint32_t acc_lanes = tmem_base + ((uint32_t)(wq * 32) << 16) + (uint32_t)(buf * kAccStride);
            uint32_t col0 = 0;  // accumulator column of what is stored
            if (kChain && rc.chain) {
                // Chain item, first pass: the 3x3's accumulator (n_mid columns of one block),
                // activated and rounded as for a stored output, into TMEM at column a_col as the
                // chained 1x1's A operand (two bf16 per column), 32 columns per unit, every other
                // unit to this warpgroup; then, once the 1x1's MMAs are done, its accumulator
                // (from column out_col) is stored like any output below.
                for (int q = 32 * h; q < rc.n_mid; q += 32 * kEpiGroups) {
                    uint32_t raw[32];
                    tmem_ld32(acc_lanes + (uint32_t)q, raw);
                    uint32_t pk[16];
#pragma unroll
                    for (int i = 0; i < 32; i += 4) {
                        const float4 s4 = *reinterpret_cast<const float4*>(sc + q + i);
                        const float4 b4 = *reinterpret_cast<const float4*>(bi + q + i);
                        float v[4];
                        bn_leaky2(s4.x, s4.y, raw[i], raw[i + 1], b4.x, b4.y, v[0], v[1]);
                        bn_leaky2(s4.z, s4.w, raw[i + 2], raw[i + 3], b4.z, b4.w, v[2], v[3]);
                        pk[i / 2] = pack_bf16x2(v[0], v[1]);
                        pk[i / 2 + 1] = pack_bf16x2(v[2], v[3]);
                    }
                    tmem_st16(acc_lanes + (uint32_t)(rc.a_col + q / 2), pk);
                }
                tmem_st_wait();
                tc_fence_before();
                mbar_arrive(bar(kBarMidFull + buf));
                mbar_wait(bar(kBarAccFull + buf), (buf ? full_ph1++ : full_ph0++) & 1u, p.ctr, pipe_limit, broken, 64);
                __syncwarp();
                tc_fence_after();
                col0 = (uint32_t)rc.out_col;
                sc += rc.n_mid;
                bi += rc.n_mid;
            }
            const bool pool = (rc.flags & 1) != 0, nhwc = (rc.flags & 2) != 0;
            // Work split between the warpgroups in units of one block x 32 output columns
            // (16 when N is an odd multiple of 16), dealt round-robin.
            const int uw = (rc.n_blk & 31) == 0 ? 32 : 16;
            // units per block (at least 1: only a record read after a pipeline wait ran out
            // can hold a smaller N, and the unit walk below must end)
            const int upb = max(1, uw == 32 ? rc.n_blk >> 5 : rc.n_blk >> 4);
            // unit u = b * upb + qi, from u = h in steps of kEpiGroups (no division per unit)
            for (int b = 0, qi = h;; qi += kEpiGroups) {
                while (qi >= upb) {
                    qi -= upb;
                    ++b;
                }
                if (b >= rc.nbk) break;
                const int q = qi * uw;
                const uint32_t taddr = acc_lanes + col0 + (uint32_t)(b * rc.n_blk + q);
                // conv position of the block's top-left pixel
                int yb = rc.y0 + b * MAFAT_BLK_ROWS, xb = rc.x0;
                if (rc.nby > 0) {
                    // per-block halos: the item's block b is block flat_by + b of its task in
                    // column-major order
                    const int lin = rc.flat_by + b;
                    const int bxx = lin / rc.nby;
                    yb = rc.y0 + (lin - bxx * rc.nby) * MAFAT_BLK_ROWS;
                    xb = rc.x0 + bxx * MAFAT_BLK_COLS;
                }
                if (pool && uw == 32) {
                    // the window of this lane's pooled pixel (epi_pool32): rows 4 wq + 2 (c & 1) + {0, 1},
                    // columns (c & ~1) + {0, 1} of the block, c = lane / 4
                    const int c = lane >> 2;
                    const int Yw = yb + wq * 4 + 2 * (c & 1), Xw = xb + (c & ~1);
                    const uint32_t pix = (uint32_t)(((Yw >> 1) - rc.out_y0) * rc.out_w + ((Xw >> 1) - rc.out_x0));
                    EpiPoolDst pd;
                    pd.out = rc.out;
                    pd.nhwc = nhwc;
                    pd.pix = nhwc ? pix * (uint32_t)rc.cout : pix * 8u;
                    pd.plane = (uint32_t)(rc.out_h * rc.out_w * 8);
                    pd.cout = rc.cout;
                    pd.store = (Yw < rc.ylim) && (Xw < rc.xlim);
                    epi_pool32(taddr, sc + q, bi + q, rc.ch_base + q, pd, lane);
                    continue;
                }
                int Y = yb + r, Xb = xb + cc;
                if (rc.pitch > 0) {
                    // flat stage (never pooled): pixel 128 (flat_by + b) + 32 wq + lane of the
                    // region read row after row, rc.pitch pixels a row
                    const int pf = (rc.flat_by + b) * 128 + wq * 32 + lane;
                    const int yy = pf / rc.pitch;
                    Y = rc.y0 + yy;
                    Xb = rc.x0 + (pf - yy * rc.pitch);
                }
                const bool valid = (Y < rc.ylim) && (Xb < rc.xlim);
                // a pooled stage's conv region starts on even rows and columns and has even
                // extents, so a window's four lanes agree on valid
                int oy = Y, ox = Xb;
                if (pool) {
                    oy = Y >> 1;
                    ox = Xb >> 1;
                }
                const uint32_t pix = (uint32_t)((oy - rc.out_y0) * rc.out_w + (ox - rc.out_x0));
                EpiDst dst;
                dst.out = rc.out;
                dst.nhwc = nhwc;
                dst.pix = nhwc ? pix * (uint32_t)rc.cout : pix * 8u;
                dst.plane = (uint32_t)(rc.out_h * rc.out_w * 8);
                dst.cout = rc.cout;
                dst.store = valid;
                dst.pool = pool;
                if (uw == 32)
                    epi_chunk<32>(taddr, sc + q, bi + q, rc.ch_base + q, dst, lane);
                else
                    epi_chunk<16>(taddr, sc + q, bi + q, rc.ch_base + q, dst, lane);
            }
            tc_fence_before();
            mbar_arrive(bar(kBarAccEmpty + buf));  // also frees the scale / bias slot
            // Hand the item to the publisher: the stores are fenced for the async proxy (TMA
            // reads of them by later items), then every thread arrives on the item's EpiDone
            // slot.  A slot is reused two items later, once the publisher is past it.
            mafat_dev::fence_proxy_async_global();
            if (acc_cnt >= 2)
                mbar_wait(bar(kBarPubDone + buf), ((acc_cnt >> 1) & 1u) ^ 1u, p.ctr, pipe_limit, broken, 32);
            mbar_arrive(bar(kBarEpiDone + buf));
            ++acc_cnt;
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == kMmaWarp) {
        __syncwarp();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(kTmemCols)
                     : "memory");
    }
    mafat_dev::finish_cta(p.ctr, p.n_ctr);
}

// ---------------------------------------------------------------------------
// Diagnostic: one 128 x n x 16 MMA with the operand and accumulator layouts of
// the fused kernel.  Operands are written to shared memory as K-major no-swizzle
// core matrices, [8-row group][K half][8 rows][8 k] (K-direction core-matrix
// stride 128 B, M / N stride 256 B), read through smem_desc as the kernel does.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(128, 1)
    mafat_diag_umma_kernel(const __nv_bfloat16* a, const __nv_bfloat16* b, float* d, int n, int a_tmem) {
    __shared__ __align__(1024) __nv_bfloat16 sa[128 * 16];
    __shared__ __align__(1024) __nv_bfloat16 sb[256 * 16];
    __shared__ __align__(8) uint64_t done_bar;
    __shared__ uint32_t tmem_slot;
    const int tid = threadIdx.x;
    for (int idx = tid; idx < 128 * 16; idx += 128) {
        int m = idx / 16, kk = idx % 16;
        sa[((m / 8) * 2 + kk / 8) * 64 + (m % 8) * 8 + kk % 8] = a[idx];
    }
    for (int idx = tid; idx < n * 16; idx += 128) {
        int m = idx / 16, kk = idx % 16;
        sb[((m / 8) * 2 + kk / 8) * 64 + (m % 8) * 8 + kk % 8] = b[idx];
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    if (tid == 0) {
        mbar_init(smem_u32(&done_bar), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if ((tid >> 5) == 0) {
        __syncwarp();  // thread 0 just left a branch of its own; .sync.aligned needs the warp converged
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_slot)),
                     "r"(512)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    const int warp0 = tid >> 5;
    if (a_tmem) {
        // row tid of A (lane tid) into TMEM columns 256..263, two bf16 per column
        uint32_t v[16];
        for (int i = 0; i < 8; ++i) {
            const uint16_t lo = reinterpret_cast<const uint16_t*>(a)[tid * 16 + 2 * i];
            const uint16_t hi = reinterpret_cast<const uint16_t*>(a)[tid * 16 + 2 * i + 1];
            v[i] = (uint32_t)lo | ((uint32_t)hi << 16);
        }
        for (int i = 8; i < 16; ++i) v[i] = 0u;
        tmem_st16(tmem + ((uint32_t)(warp0 * 32) << 16) + 256u, v);
        tmem_st_wait();
        tc_fence_before();
    }
    __syncthreads();
    tc_fence_after();
    if (warp0 == 0) {
        // one converged warp issues (elect.sync inside the issue helpers)
        const uint64_t bdesc = smem_desc(smem_u32(sb), 128u, 256u);
        if (a_tmem) {
            mma_tmem_a(tmem, tmem + 256u, (uint32_t)bdesc, (uint32_t)(bdesc >> 32), instr_desc_bf16(n, 128), 0u);
        } else {
            const uint64_t adesc = smem_desc(smem_u32(sa), 128u, 256u);
            mma_lo(tmem, (uint32_t)adesc, (uint32_t)(adesc >> 32), (uint32_t)bdesc, (uint32_t)(bdesc >> 32),
                   instr_desc_bf16(n, 128), 0u);
        }
        tc_commit_warp(smem_u32(&done_bar));
    }
    __syncwarp();
    // bounded wait (1 s) for the product
    {
        uint64_t t0 = mafat_dev::globaltimer_ns();
        while (!mbar_try_wait(smem_u32(&done_bar), 0u)) {
            if ((int64_t)(mafat_dev::globaltimer_ns() - t0) > 1000000000LL) break;
        }
    }
    __syncwarp();
    tc_fence_after();
    const int warp = tid >> 5;
    for (int q = 0; q < n / 16; ++q) {
        uint32_t raw[16];
        tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)(q * 16), raw);
#pragma unroll
        for (int i = 0; i < 16; ++i) d[(size_t)tid * n + q * 16 + i] = __uint_as_float(raw[i]);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) {
        __syncwarp();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512) : "memory");
    }
}

}  // namespace

size_t mafat_tc_smem_bytes() { return (size_t)kSmemBytes; }

namespace {
template <bool kChain, bool kTrace>
cudaError_t launch_tc(const MafatKParams& p, const CUtensorMap& in_map, int grid, cudaStream_t s) {
    // the large dynamic shared memory is opted into once per device
    static bool attr_set[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || !attr_set[dev]) {
        e = cudaFuncSetAttribute(mafat_tc_kernel<kChain, kTrace>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kSmemBytes);
        if (e != cudaSuccess) return e;
        if (dev >= 0 && dev < 64) attr_set[dev] = true;
    }
    mafat_tc_kernel<kChain, kTrace><<<grid, kThreads, kSmemBytes, s>>>(p, in_map);
    return cudaGetLastError();
}
}  // namespace

cudaError_t mafat_launch_tc(const MafatKParams& p, const CUtensorMap& in_map, int grid, bool chain, cudaStream_t s) {
    const bool trace = p.trace != nullptr;
    if (chain) return trace ? launch_tc<true, true>(p, in_map, grid, s) : launch_tc<true, false>(p, in_map, grid, s);
    return trace ? launch_tc<false, true>(p, in_map, grid, s) : launch_tc<false, false>(p, in_map, grid, s);
}

cudaError_t mafat_launch_diag_umma(const void* a, const void* b, float* d, int n, int a_tmem, cudaStream_t s) {
    mafat_diag_umma_kernel<<<1, 128, 0, s>>>((const __nv_bfloat16*)a, (const __nv_bfloat16*)b, d, n, a_tmem);
    return cudaGetLastError();
}

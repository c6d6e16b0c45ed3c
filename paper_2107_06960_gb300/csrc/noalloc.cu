// Allocation-free run of an fp32 plan.
//
// Some callers cannot have device memory allocated for them while they run:
// code that executes while a stream is being captured into a CUDA graph in
// global mode (cudaMalloc is refused there), real-time loops that forbid
// allocator calls, or host processes whose device memory is owned by another
// allocator and budgeted up front.  mafat_run_fp32_noalloc serves them: it runs
// the fp32 check kernel of an already-created plan, taking every byte of
// per-run scratch (the ring of tile buffers, the cut tensor between the two
// layer groups, and the scheduler counters) from one fixed device array that
// is part of this library, instead of from the plan's own workspace.  It makes
// no allocation of any kind.
//
// The array is MAFAT_NOALLOC_SCRATCH_BYTES (32 MiB) of device memory that every
// GPU which loads this library keeps until the process exits.  All calls share
// it, so calls that overlap in time on the GPU (different streams, or different
// host threads without ordering) race with each other.  What must start at zero
// is cleared at the start of every call: the scheduler counters (all but the
// status word, which keeps the first device error until
// mafat_noalloc_sync_status reads and clears it).  The tile buffers and the cut
// tensor need no clearing: a stage reads only the part of its input buffer that
// the previous stage of the same tile (or the first group) wrote earlier in the
// same run, and reads outside that part are bounds-checked to zero.
// The device address of the array is looked up once per device, on the first
// call made with that device current; make that first call before any stream
// capture begins.
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/mafat.h"
#include "kernels.h"

#define MAFAT_NOALLOC_SCRATCH_BYTES (32u << 20)

static __device__ __align__(256) unsigned char g_noalloc_scratch[MAFAT_NOALLOC_SCRATCH_BYTES];

mafat_status mafat_internal_fp32_params(const mafat_plan_t* plan, MafatKParams* kp, size_t* ctr_bytes,
                                        size_t* cut_bytes, size_t* scratch_bytes, size_t* in_bytes,
                                        size_t* out_bytes, int* grid, int* device);
mafat_status mafat_internal_fail(mafat_status s, const char* msg);

namespace {

constexpr int kMaxDevices = 256;
std::mutex g_mu;
void* g_addr[kMaxDevices];  // device address of g_noalloc_scratch, per device ordinal

size_t round256(size_t x) { return (x + 255) / 256 * 256; }

// Device address of the static area on the current device (looked up on first use).
mafat_status area_of_current_device(char** out) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return mafat_internal_fail(MAFAT_ECUDA, cudaGetErrorString(e));
    if (dev < 0 || dev >= kMaxDevices) return mafat_internal_fail(MAFAT_EINVAL, "device ordinal out of range");
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_addr[dev]) {
        // In host code the array's name is only a stand-in; its device address
        // has to be asked for, once per device, with that device current.
        void* ptr = nullptr;
        e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
        if (e != cudaSuccess || !ptr)
            return mafat_internal_fail(MAFAT_ECUDA, "cudaGetSymbolAddress of the static scratch area failed");
        // the status word starts clear on this device (a synchronous memset: this set-up
        // runs before any stream capture)
        e = cudaMemset((uint32_t*)ptr + MAFAT_CTR_STATUS, 0, sizeof(uint32_t));
        if (e != cudaSuccess) return mafat_internal_fail(MAFAT_ECUDA, cudaGetErrorString(e));
        g_addr[dev] = ptr;
    }
    *out = (char*)g_addr[dev];
    return MAFAT_OK;
}

}  // namespace

extern "C" mafat_status mafat_run_fp32_noalloc(const mafat_plan_t* plan, const void* input, void* output,
                                               void* stream) {
    if (!plan || !input || !output) return mafat_internal_fail(MAFAT_EINVAL, "null argument");
    if (((uintptr_t)input & 15u) || ((uintptr_t)output & 15u))
        return mafat_internal_fail(MAFAT_EINVAL, "input and output must be 16-byte aligned");
    MafatKParams kp;
    size_t ctr_b = 0, cut_b = 0, scr_b = 0, in_b = 0, out_b = 0;
    int grid = 0, plan_dev = 0;
    mafat_status st =
        mafat_internal_fp32_params(plan, &kp, &ctr_b, &cut_b, &scr_b, &in_b, &out_b, &grid, &plan_dev);
    if (st != MAFAT_OK) return st;
    const char* ib = (const char*)input;
    const char* ob = (const char*)output;
    if (ib < ob + out_b && ob < ib + in_b) return mafat_internal_fail(MAFAT_EINVAL, "input and output overlap");
    const size_t need = round256(ctr_b) + round256(cut_b) + round256(scr_b);
    if (need > MAFAT_NOALLOC_SCRATCH_BYTES)
        return mafat_internal_fail(MAFAT_EINVAL,
                                   "plan needs more scratch than the 32 MiB static area of mafat_run_fp32_noalloc "
                                   "(use fewer ring slots, a finer grid or a smaller batch)");
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return mafat_internal_fail(MAFAT_ECUDA, cudaGetErrorString(e));
    if (dev != plan_dev) return mafat_internal_fail(MAFAT_EINVAL, "the plan's device is not the current device");
    char* b = nullptr;
    if ((st = area_of_current_device(&b)) != MAFAT_OK) return st;
    uint32_t* ctr = (uint32_t*)b;
    void* cut = b + round256(ctr_b);
    void* scratch = b + round256(ctr_b) + round256(cut_b);
    cudaStream_t s = (cudaStream_t)stream;
    // the scheduler counters must start at zero, all but the status word (it keeps an
    // earlier call's device error until mafat_noalloc_sync_status reads it)
    static_assert(MAFAT_CTR_STATUS == 1, "counter layout");
    e = cudaMemsetAsync(ctr, 0, sizeof(uint32_t) * MAFAT_CTR_STATUS, s);
    if (e == cudaSuccess && ctr_b > sizeof(uint32_t) * (MAFAT_CTR_STATUS + 1))
        e = cudaMemsetAsync(ctr + MAFAT_CTR_STATUS + 1, 0, ctr_b - sizeof(uint32_t) * (MAFAT_CTR_STATUS + 1), s);
    if (e != cudaSuccess) return mafat_internal_fail(MAFAT_ECUDA, cudaGetErrorString(e));
    kp.user_in = input;
    kp.user_out = output;
    kp.cut = cut_b ? cut : nullptr;
    kp.scratch = scratch;
    kp.ctr = ctr;
    e = mafat_launch_fp32(kp, grid, s);
    if (e != cudaSuccess) return mafat_internal_fail(MAFAT_ECUDA, cudaGetErrorString(e));
    return MAFAT_OK;
}

extern "C" mafat_status mafat_noalloc_sync_status(void* stream) {
    char* b = nullptr;
    mafat_status st = area_of_current_device(&b);
    if (st != MAFAT_OK) return st;
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return mafat_internal_fail(MAFAT_ECUDA, cudaGetErrorString(e));
    uint32_t* status = (uint32_t*)b + MAFAT_CTR_STATUS;
    uint32_t v = 0;
    e = cudaMemcpy(&v, status, sizeof(v), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return mafat_internal_fail(MAFAT_ECUDA, cudaGetErrorString(e));
    if (v == MAFAT_DEV_OK) return MAFAT_OK;
    e = cudaMemset(status, 0, sizeof(uint32_t));
    if (e != cudaSuccess) return mafat_internal_fail(MAFAT_ECUDA, cudaGetErrorString(e));
    if (v == MAFAT_DEV_TIMEOUT)
        return mafat_internal_fail(MAFAT_ETIMEOUT, "a tile waited on another tile that never completed");
    return mafat_internal_fail(MAFAT_EDEVICE, "a device pipeline wait ran out");
}

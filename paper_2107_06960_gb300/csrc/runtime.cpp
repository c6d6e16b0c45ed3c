// C ABI of the fused-tile runtime: network description, planning, device
// workspace, weight packing, tensor maps and launches.  See include/mafat.h.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cstdint>
#include <algorithm>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/mafat.h"
#include "kernels.h"
#include "planner.h"

struct mafat_net_s {
    mafat::Net net;
};

struct mafat_plan_s {
    mafat::Net shapes;  // layers only (no weights)
    mafat::PlanTables t;
    int device = 0;
    int dtype = 0;
    int esz = 2;
    bool dry_run = false;
    int grid = 0;
    int64_t timeout_ns = 2000000000LL;
    std::vector<void*> allocs;
    int64_t workspace_bytes = 0;
    MafatStageDev* d_stages = nullptr;
    MafatTaskDev* d_tasks = nullptr;
    MafatItemDev* d_items = nullptr;
    MafatDepDev* d_deps = nullptr;
    CUtensorMap* d_tmaps = nullptr;
    void* d_w = nullptr;
    float* d_scale = nullptr;
    float* d_bias = nullptr;
    void* d_cut = nullptr;
    void* d_scratch = nullptr;
    uint32_t* d_ctr = nullptr;
    unsigned long long* d_trace = nullptr;
    size_t ctr_bytes = 0;
    int64_t weight_bytes = 0, scratch_bytes = 0;
    size_t in_bytes = 0, out_bytes = 0, cut_bytes = 0;
    // user-input tensor map, re-encoded when the input pointer changes
    CUtensorMap in_map;
    const void* in_map_ptr = nullptr;
    // octet-planar copy of the input for tensor-core plans whose raw NHWC rows are not a
    // multiple of 16 bytes (t.in_convert), made by a small kernel before each launch
    void* d_in_planar = nullptr;
    size_t in_planar_bytes = 0;
    bool has_chain = false;  // the plan has chain stages (selects the kernel instance)
    // staging for mafat_run_host: the NHWC input batch as copied from the host, the output
    void* d_in_stage = nullptr;
    void* d_out_stage = nullptr;
    // two staging slots of mafat_run_host_async (frames in flight), its copy streams
    struct HostSlot {
        void* d_in = nullptr;
        void* d_out = nullptr;
        cudaEvent_t h2d_done = nullptr, compute_done = nullptr, d2h_done = nullptr;
        bool used = false;
    } hs[2];
    int hs_next = 0, hs_last = -1;
    cudaStream_t s_h2d = nullptr, s_d2h = nullptr;
    std::mutex mu;
};

namespace {

thread_local std::string g_err;

mafat_status fail(mafat_status s, const std::string& msg) {
    g_err = msg;
    return s;
}

mafat_status cuda_fail(cudaError_t e, const char* what) {
    g_err = std::string(what) + ": " + cudaGetErrorString(e);
    return e == cudaErrorMemoryAllocation ? MAFAT_ENOMEM : MAFAT_ECUDA;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (PFN_cuTensorMapEncodeTiled_v12000)p;
    });
    return fn;
}

// 4-D tiled map over an octet-planar bf16 tensor [frames][c8][h][w][8]:
// dim0 = w*8 elements (one row of pixels), dim1 = h, dim2 = c8, dim3 = frames.
// Box = one A halo: cols_box pixels x rows_box rows x chunk8 octets x 1 frame.
// Out-of-range elements read as zero (the convolution's zero padding).
bool encode_planar_map(CUtensorMap* m, const void* base, int w, int h, int c8, int frames, int cols_box,
                       int rows_box, int chunk8, std::string* err) {
    auto fn = encode_fn();
    if (!fn) {
        *err = "cuTensorMapEncodeTiled unavailable";
        return false;
    }
    cuuint64_t dims[4] = {(cuuint64_t)w * 8, (cuuint64_t)h, (cuuint64_t)c8, (cuuint64_t)frames};
    cuuint64_t strides[3] = {(cuuint64_t)w * 16, (cuuint64_t)h * w * 16, (cuuint64_t)c8 * h * w * 16};
    cuuint32_t box[4] = {(cuuint32_t)cols_box * 8, (cuuint32_t)rows_box, (cuuint32_t)chunk8, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        *err = "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")";
        return false;
    }
    return true;
}

// 3-D tiled map over a narrow NHWC bf16 input (c < 8 channels) seen as rows of raw
// elements [frames][h][w*c]: dim0 = w*c elements, dim1 = h, dim2 = frames.  Box = raw_e
// elements (from a 16-byte aligned element) x one block's halo rows x 1 frame; elements outside
// the image read as zero (the convolution's zero padding, left and right included).
bool encode_raw_rows_map(CUtensorMap* m, const void* base, int w, int h, int c, int frames, int raw_e,
                         int rows_box, std::string* err) {
    auto fn = encode_fn();
    if (!fn) {
        *err = "cuTensorMapEncodeTiled unavailable";
        return false;
    }
    cuuint64_t dims[3] = {(cuuint64_t)w * c, (cuuint64_t)h, (cuuint64_t)frames};
    cuuint64_t strides[2] = {(cuuint64_t)w * c * 2, (cuuint64_t)h * w * c * 2};
    cuuint32_t box[3] = {(cuuint32_t)raw_e, (cuuint32_t)rows_box, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        *err = "cuTensorMapEncodeTiled (raw rows) failed (" + std::to_string((int)r) + ")";
        return false;
    }
    return true;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

void free_plan_memory(mafat_plan_s* p) {
    for (void* a : p->allocs) cudaFree(a);
    p->allocs.clear();
    if (p->d_in_stage) cudaFree(p->d_in_stage);
    if (p->d_out_stage) cudaFree(p->d_out_stage);
    p->d_in_stage = p->d_out_stage = nullptr;
    for (auto& h : p->hs) {
        if (h.d_in) cudaFree(h.d_in);
        if (h.d_out) cudaFree(h.d_out);
        if (h.h2d_done) cudaEventDestroy(h.h2d_done);
        if (h.compute_done) cudaEventDestroy(h.compute_done);
        if (h.d2h_done) cudaEventDestroy(h.d2h_done);
        h = mafat_plan_s::HostSlot{};
    }
    if (p->s_h2d) cudaStreamDestroy(p->s_h2d);
    if (p->s_d2h) cudaStreamDestroy(p->s_d2h);
    p->s_h2d = p->s_d2h = nullptr;
    p->hs_last = -1;
}

template <class T>
cudaError_t dalloc(mafat_plan_s* p, T** out, size_t bytes) {
    void* d = nullptr;
    if (bytes == 0) bytes = 256;
    cudaError_t e = cudaMalloc(&d, bytes);
    if (e != cudaSuccess) return e;
    p->allocs.push_back(d);
    p->workspace_bytes += (int64_t)bytes;
    *out = (T*)d;
    return cudaSuccess;
}

mafat_status launch(mafat_plan_s* p, const void* input, void* output, cudaStream_t s) {
    if (p->dry_run) return fail(MAFAT_EINVAL, "plan was created with dry_run");
    if (!input || !output) return fail(MAFAT_EINVAL, "null input or output");
    if (!aligned16(input) || !aligned16(output)) return fail(MAFAT_EINVAL, "input and output must be 16-byte aligned");
    const char* ib = (const char*)input;
    const char* ob = (const char*)output;
    if (ib < ob + p->out_bytes && ob < ib + p->in_bytes) return fail(MAFAT_EINVAL, "input and output overlap");
    cudaError_t e;
    MafatKParams kp{};
    kp.stages = p->d_stages;
    kp.tasks = p->d_tasks;
    kp.items = p->d_items;
    kp.deps = p->d_deps;
    kp.n_items = (int32_t)p->t.items.size();
    kp.tmaps = p->d_tmaps;
    kp.cut_tmap = p->t.cfg.n_groups >= 2 ? (int)p->t.tmaps.size() : -1;
    kp.w_bf16 = (const uint16_t*)p->d_w;
    kp.w_f32 = (const float*)p->d_w;
    kp.scale = p->d_scale;
    kp.bias = p->d_bias;
    kp.user_in = input;
    kp.user_out = output;
    kp.cut = p->d_cut;
    kp.scratch = p->d_scratch;
    kp.ctr = p->d_ctr;
    kp.n_ctr = (int32_t)(p->ctr_bytes / sizeof(uint32_t));
    kp.timeout_ns = p->timeout_ns;
    kp.trace = p->d_trace;
    if (p->dtype == MAFAT_BF16) {
        const mafat::Layer& L0 = p->shapes.layers[0];
        const MafatStageDev& s0 = p->t.stages[p->t.stage_first[0]];
        const void* in_dev = input;
        int64_t in_dev_bytes = (int64_t)p->in_bytes;
        if (p->t.in_convert) {
            // raw rows of this input are no multiple of 16 bytes (TMA strides must be): one small
            // kernel writes the octet-planar copy the first stage reads
            e = mafat_launch_to_planar(input, p->d_in_planar, p->t.cfg.batch, L0.h_in, L0.w_in, L0.c_in, p->t.in_c8,
                                       2, s);
            if (e != cudaSuccess) return cuda_fail(e, "layout conversion launch");
            in_dev = p->d_in_planar;
            in_dev_bytes = (int64_t)p->in_planar_bytes;
        }
        const void* pf[] = {in_dev, p->d_w, p->d_items, p->d_tasks, p->d_stages, p->d_scale, p->d_bias};
        const int64_t pb[] = {in_dev_bytes, (int64_t)p->t.weight_elems * 2,
                              (int64_t)(p->t.items.size() * sizeof(MafatItemDev)),
                              (int64_t)(p->t.tasks.size() * sizeof(MafatTaskDev)),
                              (int64_t)(p->t.stages.size() * sizeof(MafatStageDev)), (int64_t)p->t.sb_elems * 4,
                              (int64_t)p->t.sb_elems * 4};
        for (int i = 0; i < 7; ++i) {
            kp.pf_ptr[i] = pf[i];
            kp.pf_bytes[i] = pb[i];
            kp.pf_per[i] = ((pb[i] + p->grid - 1) / p->grid + 15) & ~(int64_t)15;
        }
        if (p->in_map_ptr != in_dev) {
            std::string err;
            bool ok;
            if (s0.in_mode == MAFAT_IN_GATHER)
                ok = encode_raw_rows_map(&p->in_map, in_dev, L0.w_in, L0.h_in, L0.c_in, p->t.cfg.batch, s0.raw_e,
                                         MAFAT_BLK_ROWS + s0.k - 1, &err);  // one block's halo rows
            else  // octet-planar: an 8-channel NHWC input is one octet plane, or the converted copy
                ok = encode_planar_map(&p->in_map, in_dev, L0.w_in, L0.h_in, p->t.in_c8, p->t.cfg.batch,
                                       p->t.in_cols_box, p->t.in_rows_box, p->t.in_chunk8, &err);
            if (!ok) return fail(MAFAT_ECUDA, err);
            p->in_map_ptr = in_dev;
        }
        e = mafat_launch_tc(kp, p->in_map, p->grid, p->has_chain, s);
    } else {
        e = mafat_launch_fp32(kp, p->grid, s);
    }
    if (e != cudaSuccess) return cuda_fail(e, "kernel launch");
    return MAFAT_OK;
}

}  // namespace

// Internal accessor for the allocation-free entry point (noalloc.cu): kernel
// parameters of an fp32 plan with its own scratch, cut tensor and counters left
// out (the caller supplies them), plus the sizes those three need.
mafat_status mafat_internal_fp32_params(const mafat_plan_t* plan, MafatKParams* kp, size_t* ctr_bytes,
                                        size_t* cut_bytes, size_t* scratch_bytes, size_t* in_bytes,
                                        size_t* out_bytes, int* grid, int* device) {
    const mafat_plan_s* p = plan;
    if (p->dry_run) return fail(MAFAT_EINVAL, "plan was created with dry_run");
    if (p->dtype != MAFAT_FP32) return fail(MAFAT_EUNSUPPORTED, "this entry point runs fp32 plans only");
    MafatKParams k{};
    k.stages = p->d_stages;
    k.tasks = p->d_tasks;
    k.items = p->d_items;
    k.deps = p->d_deps;
    k.n_items = (int32_t)p->t.items.size();
    k.tmaps = nullptr;
    k.cut_tmap = -1;
    k.w_f32 = (const float*)p->d_w;
    k.scale = p->d_scale;
    k.bias = p->d_bias;
    k.n_ctr = (int32_t)(p->ctr_bytes / sizeof(uint32_t));
    k.timeout_ns = p->timeout_ns;
    *kp = k;
    *ctr_bytes = p->ctr_bytes;
    *cut_bytes = p->t.cfg.n_groups >= 2 ? p->cut_bytes : 0;
    *scratch_bytes = (size_t)p->scratch_bytes;
    *in_bytes = p->in_bytes;
    *out_bytes = p->out_bytes;
    *grid = p->grid;
    *device = p->device;
    return MAFAT_OK;
}

mafat_status mafat_internal_fail(mafat_status s, const char* msg) { return fail(s, msg); }
int32_t mafat_internal_net_layers(const mafat_net_t* net) { return net ? (int32_t)net->net.layers.size() : 0; }
void mafat_internal_clear_error() { g_err.clear(); }

extern "C" {

const char* mafat_last_error(void) { return g_err.c_str(); }

const char* mafat_version(void) { return "mafat-gb300 0.1 (sm_103a tcgen05)"; }

mafat_status mafat_describe_net(const mafat_layer_desc* layers, int32_t n, int32_t in_h, int32_t in_w, int32_t in_c,
                                mafat_net_t** out) {
    if (!layers || !out) return fail(MAFAT_EINVAL, "null argument");
    *out = nullptr;
    static_assert(sizeof(mafat_layer_desc) == 5 * sizeof(int32_t), "layer desc layout");
    mafat_net_s* net = new (std::nothrow) mafat_net_s();
    if (!net) return fail(MAFAT_ENOMEM, "host allocation failed");
    std::string err = mafat::build_net((const int32_t*)layers, n, in_h, in_w, in_c, net->net);
    if (!err.empty()) {
        delete net;
        bool unsup = err.find("only") != std::string::npos || err.find("multiple of") != std::string::npos ||
                     err.find("even") != std::string::npos || err.find("needs more") != std::string::npos;
        return fail(unsup ? MAFAT_EUNSUPPORTED : MAFAT_EINVAL, err);
    }
    *out = net;
    g_err.clear();
    return MAFAT_OK;
}

mafat_status mafat_net_shape(const mafat_net_t* net, int32_t layer, int32_t shape[6]) {
    if (!net || !shape) return fail(MAFAT_EINVAL, "null argument");
    if (layer < 0 || layer >= (int)net->net.layers.size()) return fail(MAFAT_EINVAL, "layer out of range");
    const mafat::Layer& L = net->net.layers[layer];
    shape[0] = L.h_in;
    shape[1] = L.w_in;
    shape[2] = L.c_in;
    shape[3] = L.h_out;
    shape[4] = L.w_out;
    shape[5] = L.c_out;
    return MAFAT_OK;
}

mafat_status mafat_set_weights(mafat_net_t* net, int32_t layer, const float* w, const float* scale,
                               const float* bias) {
    if (!net || !w || !scale || !bias) return fail(MAFAT_EINVAL, "null argument");
    if (layer < 0 || layer >= (int)net->net.layers.size()) return fail(MAFAT_EINVAL, "layer out of range");
    const mafat::Layer& L = net->net.layers[layer];
    if (L.type != mafat::L_CONV) return fail(MAFAT_EINVAL, "layer is not a convolution");
    size_t nw = (size_t)L.c_out * L.c_in * L.k * L.k;
    net->net.w[layer].assign(w, w + nw);
    net->net.scale[layer].assign(scale, scale + L.c_out);
    net->net.bias[layer].assign(bias, bias + L.c_out);
    net->net.has_w[layer] = 1;
    return MAFAT_OK;
}

mafat_status mafat_plan_ex(const mafat_net_t* net, int32_t n_groups, const int32_t* cuts, const int32_t* grid_n,
                           const int32_t* grid_m, int32_t batch, int32_t dt, const mafat_plan_options* opt,
                           mafat_plan_t** out) {
    if (!net || !grid_n || !grid_m || !out) return fail(MAFAT_EINVAL, "null argument");
    *out = nullptr;
    if (n_groups >= 2 && !cuts) return fail(MAFAT_EINVAL, "several groups need cuts");
    if (n_groups < 1 || n_groups > MAFAT_MAX_GROUPS) return fail(MAFAT_EINVAL, "n_groups must be 1..4");
    if (dt != MAFAT_BF16 && dt != MAFAT_FP32) return fail(MAFAT_EINVAL, "unknown dtype");
    mafat_plan_options o{};
    if (opt) {
        if (opt->struct_size < (int32_t)offsetof(mafat_plan_options, dry_run))
            return fail(MAFAT_EINVAL, "mafat_plan_options.struct_size too small");
        std::memcpy(&o, opt, std::min((size_t)opt->struct_size, sizeof(o)));
    } else {
        o.test_unpublished_task = -1;
    }
    mafat::PlanConfig cfg;
    cfg.n_groups = n_groups;
    for (int c = 0; c + 1 < n_groups; ++c) cfg.cuts[c] = cuts[c];
    for (int g = 0; g < n_groups; ++g) {
        cfg.grid_n[g] = grid_n[g];
        cfg.grid_m[g] = grid_m[g];
    }
    cfg.batch = batch;
    cfg.dtype = dt;
    cfg.ring_slots = o.ring_slots;
    cfg.wave_tiles = o.wave_tiles;
    cfg.unpublished_task = o.test_unpublished_task;
    cfg.fixed_nblk = o.force_nblk;
    cfg.fixed_mb = o.force_mb;
    cfg.lookahead_items = o.lookahead_items;
    cfg.halo_reuse = o.halo_reuse != 0;
    cfg.frame_major = o.frame_major != 0;
    cfg.chain = o.chain != 0;
    cfg.rect_blocks = o.rect_blocks != 0;
    if (o.tile_bounds) {
        // per group: grid_n + 1 row bounds, then grid_m + 1 column bounds
        const int32_t* b = o.tile_bounds;
        for (int g = 0; g < n_groups; ++g) {
            cfg.row_bounds[g].assign(b, b + grid_n[g] + 1);
            b += grid_n[g] + 1;
            cfg.col_bounds[g].assign(b, b + grid_m[g] + 1);
            b += grid_m[g] + 1;
        }
    }
    int sms = 0;
    if (!o.dry_run) {
        int dev = 0;
        if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    }
    if (sms <= 0) sms = 152;
    cfg.n_ctas = o.max_ctas > 0 ? o.max_ctas : sms;

    mafat_plan_s* p = new (std::nothrow) mafat_plan_s();
    if (!p) return fail(MAFAT_ENOMEM, "host allocation failed");
    bool unsup = false;
    std::string err = mafat::build_plan(net->net, cfg, p->t, &unsup);
    if (!err.empty()) {
        delete p;
        return fail(unsup ? MAFAT_EUNSUPPORTED : MAFAT_EINVAL, err);
    }
    p->shapes.layers = net->net.layers;
    p->shapes.in_h = net->net.in_h;
    p->shapes.in_w = net->net.in_w;
    p->shapes.in_c = net->net.in_c;
    p->dtype = dt;
    p->esz = dt == MAFAT_BF16 ? 2 : 4;
    p->timeout_ns = o.wait_timeout_ns > 0 ? o.wait_timeout_ns : 2000000000LL;
    p->dry_run = o.dry_run != 0;
    const mafat::PlanTables& t = p->t;
    const mafat::Layer& L0 = net->net.layers[0];
    p->in_bytes = (size_t)t.cfg.batch * L0.c_in * L0.h_in * L0.w_in * p->esz;  // NHWC, as the caller holds it
    p->in_planar_bytes = t.in_convert ? (size_t)t.cfg.batch * t.in_c8 * 8 * L0.h_in * L0.w_in * p->esz : 0;
    for (const MafatStageDev& st : t.stages) p->has_chain = p->has_chain || st.chain != 0;
    p->out_bytes = (size_t)t.cfg.batch * t.out_h * t.out_w * t.out_c * p->esz;
    p->cut_bytes = (size_t)t.cfg.batch * t.cut_c8 * 8 * t.cut_h * t.cut_w * p->esz;
    p->ctr_bytes = (size_t)(MAFAT_CTR_BASE + t.n_counters) * sizeof(uint32_t);
    p->scratch_bytes = t.scratch_elems * p->esz;
    p->weight_bytes = (dt == MAFAT_BF16 ? t.weight_elems * 2 : t.weight32_elems * 4) + 2 * t.sb_elems * 4;
    if (p->dry_run) {
        *out = p;
        return MAFAT_OK;
    }

    cudaError_t e = cudaGetDevice(&p->device);
    if (e != cudaSuccess) {
        delete p;
        return cuda_fail(e, "cudaGetDevice");
    }
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, p->device);
    // tensor-core kernel: one CTA per SM (shared memory and TMEM); check kernel: 8 small CTAs per SM
    p->grid = o.max_ctas > 0 ? o.max_ctas : (dt == MAFAT_BF16 ? sms : 8 * sms);
    if (p->grid <= 0) p->grid = 1;

    auto bail = [&](cudaError_t ee, const char* what) {
        free_plan_memory(p);
        delete p;
        return cuda_fail(ee, what);
    };
    if ((e = dalloc(p, &p->d_stages, t.stages.size() * sizeof(MafatStageDev))) != cudaSuccess) return bail(e, "cudaMalloc");
    if ((e = dalloc(p, &p->d_tasks, t.tasks.size() * sizeof(MafatTaskDev))) != cudaSuccess) return bail(e, "cudaMalloc");
    if ((e = dalloc(p, &p->d_items, t.items.size() * sizeof(MafatItemDev))) != cudaSuccess) return bail(e, "cudaMalloc");
    if (!t.deps.empty()) {
        if ((e = dalloc(p, &p->d_deps, t.deps.size() * sizeof(MafatDepDev))) != cudaSuccess) return bail(e, "cudaMalloc");
        if ((e = cudaMemcpy(p->d_deps, t.deps.data(), t.deps.size() * sizeof(MafatDepDev), cudaMemcpyHostToDevice)) !=
            cudaSuccess)
            return bail(e, "cudaMemcpy");
    }
    if ((e = dalloc(p, &p->d_ctr, p->ctr_bytes)) != cudaSuccess) return bail(e, "cudaMalloc");
    if ((e = dalloc(p, &p->d_scale, t.sb_elems * 4)) != cudaSuccess) return bail(e, "cudaMalloc");
    if ((e = dalloc(p, &p->d_bias, t.sb_elems * 4)) != cudaSuccess) return bail(e, "cudaMalloc");
    if ((e = dalloc(p, &p->d_scratch, (size_t)p->scratch_bytes)) != cudaSuccess) return bail(e, "cudaMalloc");
    if (t.cfg.n_groups >= 2 && (e = dalloc(p, &p->d_cut, p->cut_bytes)) != cudaSuccess) return bail(e, "cudaMalloc");
    if (t.in_convert && (e = dalloc(p, &p->d_in_planar, p->in_planar_bytes)) != cudaSuccess) return bail(e, "cudaMalloc");

    std::vector<float> w32, sc, bi;
    mafat::pack_weights_fp32(net->net, t, w32, sc, bi);
    if (dt == MAFAT_BF16) {
        std::vector<uint16_t> wb;
        mafat::pack_weights_bf16(net->net, t, wb);
        if ((e = dalloc(p, &p->d_w, wb.size() * 2)) != cudaSuccess) return bail(e, "cudaMalloc");
        if ((e = cudaMemcpy(p->d_w, wb.data(), wb.size() * 2, cudaMemcpyHostToDevice)) != cudaSuccess)
            return bail(e, "cudaMemcpy");
    } else {
        if ((e = dalloc(p, &p->d_w, w32.size() * 4)) != cudaSuccess) return bail(e, "cudaMalloc");
        if ((e = cudaMemcpy(p->d_w, w32.data(), w32.size() * 4, cudaMemcpyHostToDevice)) != cudaSuccess)
            return bail(e, "cudaMemcpy");
    }
    if ((e = cudaMemcpy(p->d_scale, sc.data(), sc.size() * 4, cudaMemcpyHostToDevice)) != cudaSuccess) return bail(e, "cudaMemcpy");
    if ((e = cudaMemcpy(p->d_bias, bi.data(), bi.size() * 4, cudaMemcpyHostToDevice)) != cudaSuccess) return bail(e, "cudaMemcpy");
    if ((e = cudaMemcpy(p->d_stages, t.stages.data(), t.stages.size() * sizeof(MafatStageDev), cudaMemcpyHostToDevice)) != cudaSuccess) return bail(e, "cudaMemcpy");
    if ((e = cudaMemcpy(p->d_tasks, t.tasks.data(), t.tasks.size() * sizeof(MafatTaskDev), cudaMemcpyHostToDevice)) != cudaSuccess) return bail(e, "cudaMemcpy");
    if ((e = cudaMemcpy(p->d_items, t.items.data(), t.items.size() * sizeof(MafatItemDev), cudaMemcpyHostToDevice)) != cudaSuccess) return bail(e, "cudaMemcpy");
    if ((e = cudaMemset(p->d_scratch, 0, (size_t)p->scratch_bytes)) != cudaSuccess) return bail(e, "cudaMemset");
    if ((e = cudaMemset(p->d_ctr, 0, p->ctr_bytes)) != cudaSuccess) return bail(e, "cudaMemset");
    if (o.trace &&
        (e = dalloc(p, &p->d_trace, t.items.size() * MAFAT_TRACE_WORDS * sizeof(unsigned long long))) != cudaSuccess)
        return bail(e, "cudaMalloc");

    if (dt == MAFAT_BF16) {
        // one map per scratch-input task, then the cut tensor map
        std::vector<CUtensorMap> maps(t.tmaps.size() + (t.cfg.n_groups >= 2 ? 1 : 0));
        std::string merr;
        for (size_t i = 0; i < t.tmaps.size(); ++i) {
            const mafat::TmapReq& q = t.tmaps[i];
            const char* base = (const char*)p->d_scratch + (size_t)q.elem_off * 2;
            if (!encode_planar_map(&maps[i], base, q.w, q.h, q.c8, q.frames, q.cols_box, q.rows_box, q.chunk8, &merr)) {
                free_plan_memory(p);
                delete p;
                return fail(MAFAT_ECUDA, merr);
            }
        }
        if (t.cfg.n_groups >= 2) {
            if (!encode_planar_map(&maps.back(), p->d_cut, t.cut_w, t.cut_h, t.cut_c8, t.cfg.batch, t.cut_cols_box,
                                   t.cut_rows_box, t.cut_chunk8, &merr)) {
                free_plan_memory(p);
                delete p;
                return fail(MAFAT_ECUDA, merr);
            }
        }
        if ((e = dalloc(p, &p->d_tmaps, maps.size() * sizeof(CUtensorMap))) != cudaSuccess) return bail(e, "cudaMalloc");
        if (!maps.empty() &&
            (e = cudaMemcpy(p->d_tmaps, maps.data(), maps.size() * sizeof(CUtensorMap), cudaMemcpyHostToDevice)) !=
                cudaSuccess)
            return bail(e, "cudaMemcpy");
    }
    *out = p;
    g_err.clear();
    return MAFAT_OK;
}

mafat_status mafat_plan(const mafat_net_t* net, int32_t n_groups, const int32_t* cuts, const int32_t* grid_n,
                        const int32_t* grid_m, int32_t batch, int32_t dt, mafat_plan_t** out) {
    return mafat_plan_ex(net, n_groups, cuts, grid_n, grid_m, batch, dt, nullptr, out);
}

mafat_status mafat_run(const mafat_plan_t* plan, const void* input, void* output, void* stream) {
    if (!plan) return fail(MAFAT_EINVAL, "null plan");
    mafat_plan_s* p = const_cast<mafat_plan_s*>(plan);
    std::lock_guard<std::mutex> lk(p->mu);
    return launch(p, input, output, (cudaStream_t)stream);
}

mafat_status mafat_run_debug(const mafat_plan_t* plan, const void* input, void* cut_out, void* output,
                             void* stream) {
    if (!plan) return fail(MAFAT_EINVAL, "null plan");
    mafat_plan_s* p = const_cast<mafat_plan_s*>(plan);
    std::lock_guard<std::mutex> lk(p->mu);
    mafat_status s = launch(p, input, output, (cudaStream_t)stream);
    if (s != MAFAT_OK) return s;
    if (p->t.cfg.n_groups >= 2 && cut_out) {
        cudaError_t e = cudaMemcpyAsync(cut_out, p->d_cut, p->cut_bytes, cudaMemcpyDeviceToDevice, (cudaStream_t)stream);
        if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync");
    }
    return MAFAT_OK;
}

mafat_status mafat_run_host_async(const mafat_plan_t* plan, const void* input_host, void* output_host,
                                  void* stream) {
    if (!plan || !input_host || !output_host) return fail(MAFAT_EINVAL, "null argument");
    mafat_plan_s* p = const_cast<mafat_plan_s*>(plan);
    if (p->dry_run) return fail(MAFAT_EINVAL, "plan was created with dry_run");
    cudaStream_t s = (cudaStream_t)stream;
    std::lock_guard<std::mutex> lk(p->mu);
    cudaError_t e;
    if (!p->s_h2d) {
        // set up into locals and publish only when everything exists, so that a failure
        // part-way leaves nothing half-made behind (the next call starts over)
        mafat_plan_s::HostSlot hs[2];
        cudaStream_t s_h2d = nullptr, s_d2h = nullptr;
        auto undo = [&](cudaError_t err, const char* what) {
            for (auto& h : hs) {
                if (h.d_in) cudaFree(h.d_in);
                if (h.d_out) cudaFree(h.d_out);
                if (h.h2d_done) cudaEventDestroy(h.h2d_done);
                if (h.compute_done) cudaEventDestroy(h.compute_done);
                if (h.d2h_done) cudaEventDestroy(h.d2h_done);
            }
            if (s_h2d) cudaStreamDestroy(s_h2d);
            if (s_d2h) cudaStreamDestroy(s_d2h);
            return cuda_fail(err, what);
        };
        if ((e = cudaStreamCreateWithFlags(&s_h2d, cudaStreamNonBlocking)) != cudaSuccess ||
            (e = cudaStreamCreateWithFlags(&s_d2h, cudaStreamNonBlocking)) != cudaSuccess)
            return undo(e, "cudaStreamCreate");
        for (auto& h : hs) {
            if ((e = cudaMalloc(&h.d_in, p->in_bytes)) != cudaSuccess ||
                (e = cudaMalloc(&h.d_out, p->out_bytes)) != cudaSuccess)
                return undo(e, "cudaMalloc");
            if ((e = cudaEventCreateWithFlags(&h.h2d_done, cudaEventDisableTiming)) != cudaSuccess ||
                (e = cudaEventCreateWithFlags(&h.compute_done, cudaEventDisableTiming)) != cudaSuccess ||
                (e = cudaEventCreateWithFlags(&h.d2h_done, cudaEventDisableTiming)) != cudaSuccess)
                return undo(e, "cudaEventCreate");
        }
        p->hs[0] = hs[0];
        p->hs[1] = hs[1];
        p->s_d2h = s_d2h;
        p->s_h2d = s_h2d;  // last: its presence marks the set-up as done
    }
    const int k = p->hs_next;
    mafat_plan_s::HostSlot& h = p->hs[k];
    // upload into slot k once the run that last read it is done
    if (h.used && (e = cudaStreamWaitEvent(p->s_h2d, h.compute_done, 0)) != cudaSuccess)
        return cuda_fail(e, "cudaStreamWaitEvent");
    if ((e = cudaMemcpyAsync(h.d_in, input_host, p->in_bytes, cudaMemcpyHostToDevice, p->s_h2d)) != cudaSuccess ||
        (e = cudaEventRecord(h.h2d_done, p->s_h2d)) != cudaSuccess)
        return cuda_fail(e, "upload");
    // run on the caller's stream once the upload landed and slot k's last result was read back
    if ((e = cudaStreamWaitEvent(s, h.h2d_done, 0)) != cudaSuccess ||
        (h.used && (e = cudaStreamWaitEvent(s, h.d2h_done, 0)) != cudaSuccess))
        return cuda_fail(e, "cudaStreamWaitEvent");
    mafat_status st = launch(p, h.d_in, h.d_out, s);
    if (st != MAFAT_OK) return st;
    if ((e = cudaEventRecord(h.compute_done, s)) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
    // read the result back on its own stream
    if ((e = cudaStreamWaitEvent(p->s_d2h, h.compute_done, 0)) != cudaSuccess ||
        (e = cudaMemcpyAsync(output_host, h.d_out, p->out_bytes, cudaMemcpyDeviceToHost, p->s_d2h)) != cudaSuccess ||
        (e = cudaEventRecord(h.d2h_done, p->s_d2h)) != cudaSuccess)
        return cuda_fail(e, "download");
    h.used = true;
    p->hs_last = k;
    p->hs_next = k ^ 1;
    return MAFAT_OK;
}

mafat_status mafat_run_host_wait(const mafat_plan_t* plan) {
    if (!plan) return fail(MAFAT_EINVAL, "null plan");
    mafat_plan_s* p = const_cast<mafat_plan_s*>(plan);
    if (p->dry_run) return fail(MAFAT_EINVAL, "plan was created with dry_run");
    {
        std::lock_guard<std::mutex> lk(p->mu);
        if (p->hs_last < 0) return MAFAT_OK;
        // read-backs run in order on one stream: the last one done means all are
        cudaError_t e = cudaEventSynchronize(p->hs[p->hs_last].d2h_done);
        if (e != cudaSuccess) return cuda_fail(e, "cudaEventSynchronize");
    }
    return mafat_sync_status(plan, p->s_d2h);
}

mafat_status mafat_sync_status(const mafat_plan_t* plan, void* stream) {
    if (!plan) return fail(MAFAT_EINVAL, "null plan");
    mafat_plan_s* p = const_cast<mafat_plan_s*>(plan);
    if (p->dry_run) return fail(MAFAT_EINVAL, "plan was created with dry_run");
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    uint32_t st = 0;
    e = cudaMemcpy(&st, p->d_ctr + MAFAT_CTR_STATUS, sizeof(st), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy");
    if (st == MAFAT_DEV_OK) return MAFAT_OK;
    cudaMemset(p->d_ctr + MAFAT_CTR_STATUS, 0, sizeof(uint32_t));
    if (st == MAFAT_DEV_TIMEOUT) return fail(MAFAT_ETIMEOUT, "a tile waited on another tile that never completed");
    return fail(MAFAT_EDEVICE, "a device pipeline wait ran out");
}

mafat_status mafat_run_host(const mafat_plan_t* plan, const void* input_host, void* output_host, void* stream) {
    if (!plan || !input_host || !output_host) return fail(MAFAT_EINVAL, "null argument");
    mafat_plan_s* p = const_cast<mafat_plan_s*>(plan);
    if (p->dry_run) return fail(MAFAT_EINVAL, "plan was created with dry_run");
    cudaStream_t s = (cudaStream_t)stream;
    {
        std::lock_guard<std::mutex> lk(p->mu);
        cudaError_t e;
        if (!p->d_in_stage) {
            // both buffers or none (a failure part-way frees what it made)
            void *in_stage = nullptr, *out_stage = nullptr;
            if ((e = cudaMalloc(&in_stage, p->in_bytes)) != cudaSuccess ||
                (e = cudaMalloc(&out_stage, p->out_bytes)) != cudaSuccess) {
                if (in_stage) cudaFree(in_stage);
                return cuda_fail(e, "cudaMalloc");
            }
            p->d_out_stage = out_stage;
            p->d_in_stage = in_stage;  // last: its presence marks the set-up as done
        }
        if ((e = cudaMemcpyAsync(p->d_in_stage, input_host, p->in_bytes, cudaMemcpyHostToDevice, s)) != cudaSuccess)
            return cuda_fail(e, "cudaMemcpyAsync");
        mafat_status st = launch(p, p->d_in_stage, p->d_out_stage, s);
        if (st != MAFAT_OK) return st;
        if ((e = cudaMemcpyAsync(output_host, p->d_out_stage, p->out_bytes, cudaMemcpyDeviceToHost, s)) != cudaSuccess)
            return cuda_fail(e, "cudaMemcpyAsync");
    }
    return mafat_sync_status(plan, stream);
}

mafat_status mafat_tile_region(const mafat_plan_t* plan, int32_t group, int32_t ti, int32_t tj, int32_t layer,
                               int32_t in_rect[4], int32_t out_rect[4]) {
    if (!plan || !in_rect || !out_rect) return fail(MAFAT_EINVAL, "null argument");
    const mafat::PlanTables& t = plan->t;
    if (group < 0 || group >= t.cfg.n_groups) return fail(MAFAT_EINVAL, "group out of range");
    if (ti < 0 || ti >= t.cfg.grid_n[group] || tj < 0 || tj >= t.cfg.grid_m[group])
        return fail(MAFAT_EINVAL, "tile out of range");
    if (layer < t.groups[group][0] || layer > t.groups[group][1]) return fail(MAFAT_EINVAL, "layer not in group");
    std::vector<mafat::Rect> outs, ins;
    mafat::Rect r;
    r.y0 = t.rows[group][ti];
    r.y1 = t.rows[group][ti + 1];
    r.x0 = t.cols[group][tj];
    r.x1 = t.cols[group][tj + 1];
    if (t.cfg.halo_reuse)
        mafat::owned_regions(plan->shapes, t.groups[group][0], t.groups[group][1], r, outs, ins);
    else
        mafat::rect_regions(plan->shapes, t.groups[group][0], t.groups[group][1], r, outs, ins);
    const mafat::Rect& i = ins[layer];
    const mafat::Rect& o = outs[layer];
    in_rect[0] = i.y0; in_rect[1] = i.y1; in_rect[2] = i.x0; in_rect[3] = i.x1;
    out_rect[0] = o.y0; out_rect[1] = o.y1; out_rect[2] = o.x0; out_rect[3] = o.x1;
    return MAFAT_OK;
}

mafat_status mafat_net_tile_region(const mafat_net_t* net, int32_t first, int32_t last, int32_t n, int32_t m,
                                   int32_t ti, int32_t tj, int32_t layer, int32_t in_rect[4], int32_t out_rect[4]) {
    if (!net || !in_rect || !out_rect) return fail(MAFAT_EINVAL, "null argument");
    const int nl = (int)net->net.layers.size();
    if (first < 0 || last >= nl || first > last) return fail(MAFAT_EINVAL, "bad layer range");
    if (n <= 0 || m <= 0 || ti < 0 || ti >= n || tj < 0 || tj >= m) return fail(MAFAT_EINVAL, "tile out of range");
    if (layer < first || layer > last) return fail(MAFAT_EINVAL, "layer not in range");
    std::vector<mafat::Rect> outs, ins;
    mafat::tile_regions(net->net, first, last, n, m, ti, tj, outs, ins);
    const mafat::Rect& i = ins[layer];
    const mafat::Rect& o = outs[layer];
    in_rect[0] = i.y0; in_rect[1] = i.y1; in_rect[2] = i.x0; in_rect[3] = i.x1;
    out_rect[0] = o.y0; out_rect[1] = o.y1; out_rect[2] = o.x0; out_rect[3] = o.x1;
    return MAFAT_OK;
}

mafat_status mafat_predict_layer_group(const mafat_net_t* net, int32_t first, int32_t last, int32_t n, int32_t m,
                                       double bias_mib, int32_t input_factor, double* out_mib) {
    if (!net || !out_mib) return fail(MAFAT_EINVAL, "null argument");
    const int nl = (int)net->net.layers.size();
    if (first < 0 || last >= nl || first > last || n <= 0 || m <= 0) return fail(MAFAT_EINVAL, "bad arguments");
    *out_mib = mafat::predict_layer_group(net->net, first, last, n, m, bias_mib, input_factor);
    return MAFAT_OK;
}

mafat_status mafat_predict_mem(const mafat_net_t* net, int32_t cut, int32_t n1, int32_t m1, int32_t n2, int32_t m2,
                               double bias_mib, double* out_mib) {
    if (!net || !out_mib) return fail(MAFAT_EINVAL, "null argument");
    if (n1 <= 0 || m1 <= 0 || n2 <= 0 || m2 <= 0) return fail(MAFAT_EINVAL, "grid sizes must be positive");
    *out_mib = mafat::predict_mem(net->net, cut, n1, m1, n2, m2, bias_mib);
    return MAFAT_OK;
}

mafat_status mafat_balanced_bounds(const mafat_net_t* net, int32_t first, int32_t last, int32_t n, int32_t m,
                                   int32_t* row_bounds, int32_t* col_bounds) {
    if (!net || !row_bounds || !col_bounds) return fail(MAFAT_EINVAL, "null argument");
    const int nl = (int)net->net.layers.size();
    if (first < 0 || last >= nl || first > last) return fail(MAFAT_EINVAL, "bad layer range");
    const mafat::Layer& L = net->net.layers[last];
    if (n <= 0 || m <= 0 || n > L.h_out || m > L.w_out) return fail(MAFAT_EINVAL, "bad grid size");
    const std::vector<int> r = mafat::balanced_bounds(net->net, first, last, n, 0);
    const std::vector<int> c = mafat::balanced_bounds(net->net, first, last, m, 1);
    std::copy(r.begin(), r.end(), row_bounds);
    std::copy(c.begin(), c.end(), col_bounds);
    return MAFAT_OK;
}

mafat_status mafat_search(const mafat_net_t* net, double limit_mib, double bias_mib, int32_t* top_tile,
                          int32_t* cut, int32_t* bottom_tile) {
    if (!net || !top_tile || !cut || !bottom_tile) return fail(MAFAT_EINVAL, "null argument");
    int a, b, c;
    mafat::search(net->net, limit_mib, bias_mib, &a, &b, &c);
    *top_tile = a;
    *cut = b;
    *bottom_tile = c;
    return MAFAT_OK;
}

mafat_status mafat_plan_stats(const mafat_plan_t* plan, mafat_plan_stats_t* out) {
    if (!plan || !out) return fail(MAFAT_EINVAL, "null argument");
    if (out->struct_size < (int32_t)sizeof(mafat_plan_stats_t)) return fail(MAFAT_EINVAL, "struct_size too small");
    const mafat::PlanTables& t = plan->t;
    mafat_plan_stats_t s{};
    s.struct_size = (int32_t)sizeof(mafat_plan_stats_t);
    s.n_groups = t.cfg.n_groups;
    s.n_tiles = t.n_tiles;
    s.n_tasks = (int32_t)t.tasks.size();
    s.n_items = (int64_t)t.items.size();
    s.useful_flops = t.useful_flops;
    s.executed_flops = t.executed_flops * 1.0;
    s.issued_flops = t.issued_flops;
    s.predicted_mib = t.predicted_mib;
    s.group_io_bytes = t.group_io_elems * plan->esz;
    s.weight_bytes = plan->weight_bytes;
    s.scratch_bytes = plan->scratch_bytes;
    s.workspace_bytes = plan->workspace_bytes;
    s.smem_bytes_per_cta = plan->dtype == MAFAT_BF16 ? (int64_t)mafat_tc_smem_bytes() : 4;
    s.ring_slots = t.ring_slots;
    s.wave_tiles = t.wave_tiles;
    s.max_ctas = plan->grid;
    s.dtype = plan->dtype;
    s.frames_overlapped = t.frames_overlapped;
    *out = s;
    return MAFAT_OK;
}

int32_t mafat_launches_per_run(const mafat_plan_t* plan) {
    if (!plan) return 0;
    return plan->dtype == MAFAT_BF16 && plan->t.in_convert ? 2 : 1;
}

mafat_status mafat_plan_trace(const mafat_plan_t* plan, uint64_t* out, int64_t max_words, void* stream) {
    if (!plan || !out) return fail(MAFAT_EINVAL, "null argument");
    if (!plan->d_trace) return fail(MAFAT_EINVAL, "plan was not created with options.trace = 1");
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    int64_t words = std::min<int64_t>(max_words, (int64_t)plan->t.items.size() * MAFAT_TRACE_WORDS);
    if (words <= 0) return MAFAT_OK;
    e = cudaMemcpy(out, plan->d_trace, (size_t)words * sizeof(uint64_t), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy");
    for (int64_t i = 0; (i + 1) * MAFAT_TRACE_WORDS <= words; ++i) {
        const MafatItemDev& it = plan->t.items[(size_t)i];
        const int layer = plan->t.stages[plan->t.tasks[it.task].stage].layer;
        out[i * MAFAT_TRACE_WORDS + 5] = ((uint64_t)it.task << 16) | (uint64_t)layer;
    }
    return MAFAT_OK;
}

void mafat_plan_destroy(mafat_plan_t* plan) {
    if (!plan) return;
    free_plan_memory(plan);
    delete plan;
}

void mafat_net_destroy(mafat_net_t* net) { delete net; }

mafat_status mafat_diag_umma(const void* a_dev, const void* b_dev, float* d_dev, int32_t n, int32_t a_in_tmem,
                             void* stream) {
    if (!a_dev || !b_dev || !d_dev) return fail(MAFAT_EINVAL, "null argument");
    if (n < 16 || n > 256 || n % 16 != 0) return fail(MAFAT_EINVAL, "n must be a multiple of 16 in 16..256");
    cudaError_t e = mafat_launch_diag_umma(a_dev, b_dev, d_dev, n, a_in_tmem ? 1 : 0, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "diag launch");
    e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "diag sync");
    return MAFAT_OK;
}

}  // extern "C"

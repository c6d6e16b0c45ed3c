// Measured plan search (Algorithm 2 of Sec. 4.1 re-targeted at the GPU): enumerate
// cut x tiling candidates, keep those whose intermediates fit the L2 budget, time each
// on the device and report the fastest.  Built on the library's own C ABI.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <string>
#include <vector>

#include "../../include/mafat.h"

mafat_status mafat_internal_fail(mafat_status s, const char* msg);
int32_t mafat_internal_net_layers(const mafat_net_t* net);
void mafat_internal_clear_error();

namespace {

struct Candidate {
    int n_groups, cut, gn[2], gm[2];
};

std::vector<std::pair<int, int>> grids_of(int max_grid, bool square_only) {
    std::vector<std::pair<int, int>> g;
    for (int n = 1; n <= max_grid; ++n)
        for (int m = 1; m <= max_grid; ++m)
            if (square_only ? n == m : (n - m <= 1 && m - n <= 1)) g.emplace_back(n, m);
    return g;
}

struct DeviceBuffers {
    void* in = nullptr;
    void* out = nullptr;
    void* flush = nullptr;
    cudaEvent_t a = nullptr, b = nullptr;
    ~DeviceBuffers() {
        if (in) cudaFree(in);
        if (out) cudaFree(out);
        if (flush) cudaFree(flush);
        if (a) cudaEventDestroy(a);
        if (b) cudaEventDestroy(b);
    }
};

constexpr size_t kFlushBytes = 256u << 20;  // twice the L2

}  // namespace

mafat_status mafat_search_measured(const mafat_net_t* net, const mafat_search_options* opt, void* stream,
                                   mafat_search_candidate* out, int32_t max_out, int32_t* n_out,
                                   int32_t* best) {
    if (!net || !opt || !n_out || !best) return mafat_internal_fail(MAFAT_EINVAL, "null argument");
    if (opt->struct_size != (int32_t)sizeof(mafat_search_options))
        return mafat_internal_fail(MAFAT_EINVAL, "mafat_search_options.struct_size mismatch");
    if (opt->n_cuts < 0 || (opt->n_cuts > 0 && !opt->cuts) || max_out < 0 || (max_out > 0 && !out))
        return mafat_internal_fail(MAFAT_EINVAL, "bad candidate list");
    if (opt->dtype != MAFAT_BF16 && opt->dtype != MAFAT_FP32) return mafat_internal_fail(MAFAT_EINVAL, "bad dtype");
    const int batch = opt->batch > 0 ? opt->batch : 1;
    const int max_grid = opt->max_grid > 0 ? opt->max_grid : 5;
    const int runs = opt->runs > 0 ? opt->runs : 10;
    const bool dry = opt->dry_run != 0;
    *n_out = 0;
    *best = -1;

    int32_t s_in[6], s_out[6];
    mafat_status st = mafat_net_shape(net, 0, s_in);
    if (st != MAFAT_OK) return st;
    if ((st = mafat_net_shape(net, mafat_internal_net_layers(net) - 1, s_out)) != MAFAT_OK) return st;

    int64_t budget = opt->budget_bytes;
    if (budget == 0) {
        budget = 128ll << 20;
        int dev = 0, l2 = 0;
        if (!dry && cudaGetDevice(&dev) == cudaSuccess &&
            cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev) == cudaSuccess && l2 > 0)
            budget = l2;
    }

    std::vector<Candidate> cands;
    const auto grids = grids_of(max_grid, opt->square_only != 0);
    if (opt->include_one_group)
        for (auto g : grids) cands.push_back({1, 0, {g.first, 1}, {g.second, 1}});
    for (int c = 0; c < opt->n_cuts; ++c)
        for (auto g1 : grids)
            for (auto g2 : grids) cands.push_back({2, opt->cuts[c], {g1.first, g2.first}, {g1.second, g2.second}});

    const size_t esz = opt->dtype == MAFAT_BF16 ? 2 : 4;
    // input [batch][ceil(C/8)][H][W][8], output NHWC (shape = {.., .., .., H, W, C} of layer outputs)
    const size_t in_bytes = (size_t)batch * ((s_in[2] + 7) / 8) * 8 * s_in[0] * s_in[1] * esz;
    const size_t out_bytes = (size_t)batch * s_out[3] * s_out[4] * s_out[5] * esz;
    DeviceBuffers buf;
    cudaStream_t s = (cudaStream_t)stream;
    if (!dry) {
        cudaError_t e;
        if ((e = cudaMalloc(&buf.in, in_bytes)) != cudaSuccess || (e = cudaMalloc(&buf.out, out_bytes)) != cudaSuccess ||
            (opt->flush_l2 && (e = cudaMalloc(&buf.flush, kFlushBytes)) != cudaSuccess) ||
            (e = cudaEventCreate(&buf.a)) != cudaSuccess || (e = cudaEventCreate(&buf.b)) != cudaSuccess ||
            (e = cudaMemsetAsync(buf.in, 0, in_bytes, s)) != cudaSuccess)
            return mafat_internal_fail(MAFAT_ECUDA, cudaGetErrorString(e));
    }

    double best_us = 0.0;
    for (size_t i = 0; i < cands.size(); ++i) {
        const Candidate& c = cands[i];
        mafat_search_candidate r{};
        r.n_groups = c.n_groups;
        r.cut = c.cut;
        for (int g = 0; g < 2; ++g) {
            r.grid_n[g] = g < c.n_groups ? c.gn[g] : 0;
            r.grid_m[g] = g < c.n_groups ? c.gm[g] : 0;
        }
        r.us_per_run = -1.0;
        r.status = MAFAT_OK;
        const int32_t cut = c.cut;
        mafat_plan_options po{};
        po.struct_size = (int32_t)sizeof(po);
        po.dry_run = 1;
        mafat_plan_t* plan = nullptr;
        st = mafat_plan_ex(net, c.n_groups, &cut, c.gn, c.gm, batch, opt->dtype, &po, &plan);
        if (st == MAFAT_OK) {
            mafat_plan_stats_t ps{};
            ps.struct_size = (int32_t)sizeof(ps);
            mafat_plan_stats(plan, &ps);
            mafat_plan_destroy(plan);
            plan = nullptr;
            int64_t cut_bytes = 0;
            if (c.n_groups == 2) {
                int32_t sh[6];
                if (mafat_net_shape(net, c.cut - 1, sh) == MAFAT_OK)
                    cut_bytes = (int64_t)batch * ((sh[5] + 7) / 8) * 8 * sh[3] * sh[4] * (int64_t)esz;
            }
            r.intermediate_bytes = ps.scratch_bytes + cut_bytes;
            r.predicted_mib = ps.predicted_mib;
            r.executed_flops = ps.executed_flops;
            if (budget > 0 && r.intermediate_bytes > budget) r.status = MAFAT_ENOFIT;
        } else {
            r.status = st;
        }
        if (!dry && r.status == MAFAT_OK) {
            st = mafat_plan_ex(net, c.n_groups, &cut, c.gn, c.gm, batch, opt->dtype, nullptr, &plan);
            if (st != MAFAT_OK) {
                r.status = st;
            } else {
                std::vector<float> t;
                bool ok = true;
                for (int k = 0; k < 2 + runs && ok; ++k) {
                    if (opt->flush_l2 && cudaMemsetAsync(buf.flush, k & 0xff, kFlushBytes, s) != cudaSuccess) ok = false;
                    if (ok && cudaEventRecord(buf.a, s) != cudaSuccess) ok = false;
                    if (ok && mafat_run(plan, buf.in, buf.out, stream) != MAFAT_OK) ok = false;
                    if (ok && cudaEventRecord(buf.b, s) != cudaSuccess) ok = false;
                    if (ok && cudaEventSynchronize(buf.b) != cudaSuccess) ok = false;
                    float ms = 0.f;
                    if (ok && cudaEventElapsedTime(&ms, buf.a, buf.b) != cudaSuccess) ok = false;
                    if (ok && k >= 2) t.push_back(ms);
                }
                const mafat_status ds = mafat_sync_status(plan, stream);
                mafat_plan_destroy(plan);
                if (!ok) {
                    r.status = MAFAT_ECUDA;
                } else if (ds != MAFAT_OK) {
                    r.status = ds;
                } else {
                    std::sort(t.begin(), t.end());
                    r.us_per_run = 1e3 * t[t.size() / 2];
                    if (*best < 0 || r.us_per_run < best_us) {
                        *best = (int32_t)i;
                        best_us = r.us_per_run;
                    }
                }
            }
        }
        if ((int32_t)i < max_out) out[i] = r;
    }
    *n_out = (int32_t)cands.size();
    mafat_internal_clear_error();  // candidates that could not be planned are reported in their status
    return MAFAT_OK;
}

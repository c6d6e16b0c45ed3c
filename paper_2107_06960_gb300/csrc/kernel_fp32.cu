// fp32 check-mode kernel: fused-tile execution (MAFAT, Sec. 4) on CUDA cores.
//
// Runs the same work list and persistent scheduler as the tensor-core kernel,
// with fp32 activations, weights and accumulation, so that the tiling, the
// region arithmetic and the dependency chain can be checked against the
// oracle at a tight tolerance.  One CTA of 128 threads computes one item: a
// block of 128 conv output pixels (thread = pixel; a 16 x 8 rectangle, or a run
// of a flat stage's region) for one block of output channels, 8 channels at a
// time:
//   acc[o] = sum_{c, ky, kx} w[o][c][ky][kx] * in[y + ky - p][x + kx - p][c]
//   z = scale[o] * acc + bias[o];  out = z > 0 ? z : 0.1 z
// followed, for a fused max-pool, by the 2x2 maximum over neighbouring lanes.
#include "sched.cuh"

namespace {

__device__ __forceinline__ const float* buf_ptr(const MafatKParams& p, int kind) {
    switch (kind) {
        case MAFAT_BUF_USER_IN: return (const float*)p.user_in;
        case MAFAT_BUF_CUT: return (const float*)p.cut;
        case MAFAT_BUF_SCRATCH:
        case MAFAT_BUF_MAP: return (const float*)p.scratch;
        default: return (const float*)p.user_out;
    }
}

__global__ void __launch_bounds__(128) mafat_fp32_kernel(const __grid_constant__ MafatKParams p) {
    __shared__ int s_ticket;
    const int tid = threadIdx.x;
    const int r = tid >> 3, c = tid & 7;  // pixel of the 16 x 8 block; lane = (r % 4) * 8 + c
    while (true) {
        if (tid == 0) s_ticket = (int)atomicAdd(&p.ctr[MAFAT_CTR_TICKET], 1u);
        __syncthreads();
        const int ticket = s_ticket;
        if (ticket >= p.n_items) break;
        const MafatItemDev it = p.items[ticket];
        const MafatTaskDev tk = p.tasks[it.task];
        const MafatStageDev st = p.stages[tk.stage];
        if (tid == 0) {
            if (p.trace) {
                mafat_dev::trace_put(p.trace, ticket, 0, mafat_dev::globaltimer_ns());
                mafat_dev::trace_put(p.trace, ticket, 4, mafat_dev::smid());
            }
            mafat_dev::wait_item_deps(p.ctr, it, p.timeout_ns);
            if (tk.dep_count > 0) mafat_dev::wait_dep_list(p.ctr, p.deps, tk.dep_first, tk.dep_count, p.timeout_ns);
            if (p.trace) mafat_dev::trace_put(p.trace, ticket, 1, mafat_dev::globaltimer_ns());
        }
        __syncthreads();

        const float* in = buf_ptr(p, tk.in_kind) + tk.in_off;
        float* out = (float*)(tk.out_kind == MAFAT_BUF_USER_OUT ? p.user_out
                              : tk.out_kind == MAFAT_BUF_CUT    ? p.cut
                                                                : p.scratch) + tk.out_off;
        const float* w = p.w_f32 + st.w32_off;
        const int k = st.k, kk = st.k * st.k;
        const int o_end = min((it.nb + 1) * st.n_blk, st.cout);
        for (int blk = 0; blk < it.nbk; ++blk)
        for (int o0 = it.nb * st.n_blk; o0 < o_end; o0 += 8) {
            // pixel of this thread: (r, c) of a 16 x 8 block, or in a flat stage pixel
            // 128 (by + blk) + tid of the region read row after row, cols_box pixels a row
            int Y = tk.cy0 + (it.by + blk) * MAFAT_BLK_ROWS + r, X = tk.cx0 + it.bx * MAFAT_BLK_COLS + c;
            if (st.flat) {
                const int pf = (it.by + blk) * 128 + tid;
                const int yy = pf / st.cols_box;
                Y = tk.cy0 + yy;
                X = tk.cx0 + (pf - yy * st.cols_box);
            }
            const bool valid = (Y < tk.cy0 + tk.ch) && (X < tk.cx0 + tk.cw);
            float acc[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) acc[q] = 0.f;
            // the caller's input is NHWC; every other buffer is octet-planar
            const bool nhwc_in = tk.in_kind == MAFAT_BUF_USER_IN;
            const int pix_stride = nhwc_in ? st.cin : 8;
            for (int ci = 0; ci < st.cin; ++ci) {
                const float* in_c = nhwc_in ? in + ci : in + (size_t)(ci >> 3) * tk.in_h * tk.in_w * 8 + (ci & 7);
                for (int ky = 0; ky < k; ++ky) {
                    const int ly = Y + ky - st.pad - tk.in_y0;
                    for (int kx = 0; kx < k; ++kx) {
                        const int lx = X + kx - st.pad - tk.in_x0;
                        float v = 0.f;
                        if (ly >= 0 && ly < tk.in_h && lx >= 0 && lx < tk.in_w)
                            v = in_c[((size_t)ly * tk.in_w + lx) * pix_stride];
                        const float* wp = w + ((size_t)o0 * st.cin + ci) * kk + ky * k + kx;
#pragma unroll
                        for (int q = 0; q < 8; ++q) acc[q] = fmaf(__ldg(wp + (size_t)q * st.cin * kk), v, acc[q]);
                    }
                }
            }
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                float z = __ldg(p.scale + st.sb_off + o0 + q) * acc[q] + __ldg(p.bias + st.sb_off + o0 + q);
                acc[q] = z > 0.f ? z : 0.1f * z;
            }
            int oy = Y, ox = X;
            bool store = valid;
            if (st.pool) {
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    acc[q] = fmaxf(acc[q], __shfl_xor_sync(0xffffffffu, acc[q], 1));
                    acc[q] = fmaxf(acc[q], __shfl_xor_sync(0xffffffffu, acc[q], 8));
                }
                store = valid && ((r & 1) == 0) && ((c & 1) == 0);
                oy = Y >> 1;
                ox = X >> 1;
            }
            if (store) {
                const int ly = oy - tk.out_y0, lx = ox - tk.out_x0;
                float* dst;
                if (tk.out_nhwc)
                    dst = out + ((size_t)ly * tk.out_w + lx) * st.cout + o0;
                else
                    dst = out + (((size_t)(o0 >> 3) * tk.out_h + ly) * tk.out_w + lx) * 8;
                reinterpret_cast<float4*>(dst)[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
                reinterpret_cast<float4*>(dst)[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
            }
        }
        __threadfence();
        __syncthreads();
        if (tid == 0) {
            mafat_dev::publish_item(p.ctr, it, tk.done_ctr);
            if (p.trace) {
                const uint64_t t = mafat_dev::globaltimer_ns();
                mafat_dev::trace_put(p.trace, ticket, 2, t);
                mafat_dev::trace_put(p.trace, ticket, 3, t);
            }
        }
    }
    mafat_dev::finish_cta(p.ctr, p.n_ctr);
}

}  // namespace

namespace {
// One thread per (frame, octet, y, x), x fastest, so that the 8-element writes of a
// warp are contiguous; channels at or above c are written as zero.
template <typename T>
__global__ void __launch_bounds__(256) to_planar_kernel(const T* __restrict__ in, T* __restrict__ out, int frames,
                                                        int h, int w, int c, int c8) {
    const int64_t total = (int64_t)frames * c8 * h * w;
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= total) return;
    const int x = (int)(idx % w);
    int64_t r = idx / w;
    const int y = (int)(r % h);
    r /= h;
    const int o = (int)(r % c8);
    const int f = (int)(r / c8);
    const T* src = in + (((int64_t)f * h + y) * w + x) * c;
    T v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const int ch = o * 8 + k;
        v[k] = ch < c ? src[ch] : T(0);
    }
    T* dst = out + idx * 8;  // [f][o][y][x][8] in idx order, 16-byte aligned
    if constexpr (sizeof(T) == 2) {
        uint4 q;
        q.x = (uint32_t)v[0] | ((uint32_t)v[1] << 16);
        q.y = (uint32_t)v[2] | ((uint32_t)v[3] << 16);
        q.z = (uint32_t)v[4] | ((uint32_t)v[5] << 16);
        q.w = (uint32_t)v[6] | ((uint32_t)v[7] << 16);
        *reinterpret_cast<uint4*>(dst) = q;
    } else {
        reinterpret_cast<float4*>(dst)[0] = make_float4(v[0], v[1], v[2], v[3]);
        reinterpret_cast<float4*>(dst)[1] = make_float4(v[4], v[5], v[6], v[7]);
    }
}
}  // namespace

cudaError_t mafat_launch_to_planar(const void* nhwc, void* planar, int frames, int h, int w, int c, int c8,
                                   int elem_bytes, cudaStream_t s) {
    const int64_t total = (int64_t)frames * c8 * h * w;
    if (total <= 0) return cudaSuccess;
    const unsigned grid = (unsigned)((total + 255) / 256);
    if (elem_bytes == 2)
        to_planar_kernel<uint16_t><<<grid, 256, 0, s>>>((const uint16_t*)nhwc, (uint16_t*)planar, frames, h, w, c, c8);
    else
        to_planar_kernel<float><<<grid, 256, 0, s>>>((const float*)nhwc, (float*)planar, frames, h, w, c, c8);
    return cudaGetLastError();
}

cudaError_t mafat_launch_fp32(const MafatKParams& p, int grid, cudaStream_t s) {
    mafat_fp32_kernel<<<grid, 128, 0, s>>>(p);
    return cudaGetLastError();
}

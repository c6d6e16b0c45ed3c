// Host-side planner of fused-tile execution (MAFAT, Sec. 4).  See planner.h.
#include "planner.h"

#include <algorithm>
#include <cstring>
#include <string>

namespace mafat {

static int ceil_div(int a, int b) { return (a + b - 1) / b; }

std::string build_net(const int32_t* d, int n, int in_h, int in_w, int in_c, Net& net) {
    if (n <= 0) return "network needs at least one layer";
    if (in_h <= 0 || in_w <= 0 || in_c <= 0) return "input size must be positive";
    net.layers.clear();
    net.in_h = in_h;
    net.in_w = in_w;
    net.in_c = in_c;
    int h = in_h, w = in_w, c = in_c;
    for (int l = 0; l < n; ++l) {
        Layer L{};
        L.type = d[5 * l + 0];
        L.k = d[5 * l + 1];
        L.stride = d[5 * l + 2];
        L.pad = d[5 * l + 3];
        L.filters = d[5 * l + 4];
        L.h_in = h;
        L.w_in = w;
        L.c_in = c;
        if (L.type == L_CONV) {
            if (!((L.k == 3 && L.pad == 1) || (L.k == 1 && L.pad == 0)) || L.stride != 1)
                return "layer " + std::to_string(l) + ": only 3x3/s1/p1 and 1x1/s1/p0 convolutions are supported";
            if (L.filters <= 0 || L.filters % 8 != 0)
                return "layer " + std::to_string(l) + ": output channels must be a positive multiple of 8";
            if (L.k == 1 && c <= 8)
                return "layer " + std::to_string(l) + ": a 1x1 convolution needs more than 8 input channels";
            L.c_out = L.filters;
        } else if (L.type == L_MAXPOOL) {
            if (L.k != 2 || L.stride != 2 || L.pad != 0)
                return "layer " + std::to_string(l) + ": only 2x2/s2 max-pool is supported";
            if (h % 2 != 0 || w % 2 != 0)
                return "layer " + std::to_string(l) + ": max-pool input must have even height and width";
            L.c_out = c;
        } else {
            return "layer " + std::to_string(l) + ": unknown layer type";
        }
        L.h_out = (h + 2 * L.pad - L.k) / L.stride + 1;
        L.w_out = (w + 2 * L.pad - L.k) / L.stride + 1;
        if (L.h_out <= 0 || L.w_out <= 0) return "layer " + std::to_string(l) + ": empty output";
        h = L.h_out;
        w = L.w_out;
        c = L.c_out;
        net.layers.push_back(L);
    }
    net.w.assign(n, {});
    net.scale.assign(n, {});
    net.bias.assign(n, {});
    net.has_w.assign(n, 0);
    return "";
}

void back_interval(int a, int b, int k, int s, int p, int size_in, int* lo, int* hi) {
    if (b <= a) {
        *lo = 0;
        *hi = 0;
        return;
    }
    // The window of output a starts at a*s - p; that of output b-1 ends at (b-1)*s - p + k - 1.
    *lo = std::max(a * s - p, 0);
    *hi = std::min((b - 1) * s - p + k, size_in);
}

void tile_regions(const Net& net, int first, int last, int n, int m, int i, int j,
                  std::vector<Rect>& out_rects, std::vector<Rect>& in_rects) {
    const Layer& Ll = net.layers[last];
    Rect r;
    r.y0 = grid_bound(Ll.h_out, n, i);
    r.y1 = grid_bound(Ll.h_out, n, i + 1);
    r.x0 = grid_bound(Ll.w_out, m, j);
    r.x1 = grid_bound(Ll.w_out, m, j + 1);
    rect_regions(net, first, last, r, out_rects, in_rects);
}

std::vector<int> axis_bounds(int len, int n, const std::vector<int>& given) {
    if (!given.empty()) return given;
    std::vector<int> b(n + 1);
    for (int i = 0; i <= n; ++i) b[i] = grid_bound(len, n, i);
    return b;
}

std::string check_bounds(const std::vector<int>& b, int len, int n) {
    if ((int)b.size() != n + 1) return "tile bounds: need n + 1 values per axis";
    if (b[0] != 0 || b[n] != len) return "tile bounds must start at 0 and end at the map size";
    for (int i = 0; i < n; ++i)
        if (b[i + 1] <= b[i]) return "tile bounds must increase strictly";
    return "";
}

std::vector<int> balanced_bounds(const Net& net, int first, int last, int n, int axis) {
    const Layer& Ll = net.layers[last];
    const int len = axis == 0 ? Ll.h_out : Ll.w_out;
    n = std::max(1, std::min(n, len));
    // work[a][b]: MACs of the part [a, b) with the other axis whole
    std::vector<double> work((size_t)(len + 1) * (len + 1), 0.0);
    for (int a = 0; a < len; ++a)
        for (int b = a + 1; b <= len; ++b) {
            int lo = a, hi = b;
            double w = 0.0;
            for (int l = last; l >= first; --l) {
                const Layer& L = net.layers[l];
                int ilo, ihi;
                back_interval(lo, hi, L.k, L.stride, L.pad, axis == 0 ? L.h_in : L.w_in, &ilo, &ihi);
                if (L.type == L_CONV)
                    w += (double)(hi - lo) * (axis == 0 ? L.w_out : L.h_out) * L.c_out * (double)L.c_in * L.k * L.k;
                lo = ilo;
                hi = ihi;
            }
            work[(size_t)a * (len + 1) + b] = w;
        }
    // best[k][b]: smallest possible largest part when [0, b) is cut into k parts
    const double inf = 1e300;
    std::vector<double> best((size_t)(n + 1) * (len + 1), inf);
    std::vector<int> from((size_t)(n + 1) * (len + 1), -1);
    best[0] = 0.0;
    for (int k = 1; k <= n; ++k)
        for (int b = k; b <= len; ++b)
            for (int a = k - 1; a < b; ++a) {
                const double prev = best[(size_t)(k - 1) * (len + 1) + a];
                if (prev >= inf) continue;
                const double v = std::max(prev, work[(size_t)a * (len + 1) + b]);
                if (v < best[(size_t)k * (len + 1) + b]) {
                    best[(size_t)k * (len + 1) + b] = v;
                    from[(size_t)k * (len + 1) + b] = a;
                }
            }
    std::vector<int> bounds(n + 1);
    bounds[n] = len;
    for (int k = n; k > 0; --k) bounds[k - 1] = from[(size_t)k * (len + 1) + bounds[k]];
    return bounds;
}

// Halo reuse: the part of every layer's output a tile owns (its group-output rectangle
// scaled through the max-pools, never grown by a convolution's halo: stride-1 convs keep
// the map size), and the input region each layer reads for it (halo included, computed
// by the neighbours that own it).
void owned_regions(const Net& net, int first, int last, const Rect& out_last, std::vector<Rect>& out_rects,
                   std::vector<Rect>& in_rects) {
    Rect r = out_last;
    if ((int)out_rects.size() < (int)net.layers.size()) out_rects.resize(net.layers.size());
    if ((int)in_rects.size() < (int)net.layers.size()) in_rects.resize(net.layers.size());
    for (int l = last; l >= first; --l) {
        const Layer& L = net.layers[l];
        Rect in;
        back_interval(r.y0, r.y1, L.k, L.stride, L.pad, L.h_in, &in.y0, &in.y1);
        back_interval(r.x0, r.x1, L.k, L.stride, L.pad, L.w_in, &in.x0, &in.x1);
        if (r.empty()) in = Rect{};
        out_rects[l] = r;
        in_rects[l] = in;
        if (L.type == L_MAXPOOL) r = Rect{2 * r.y0, 2 * r.y1, 2 * r.x0, 2 * r.x1};
    }
}

void rect_regions(const Net& net, int first, int last, const Rect& out_last, std::vector<Rect>& out_rects,
                  std::vector<Rect>& in_rects) {
    Rect r = out_last;
    if ((int)out_rects.size() < (int)net.layers.size()) out_rects.resize(net.layers.size());
    if ((int)in_rects.size() < (int)net.layers.size()) in_rects.resize(net.layers.size());
    for (int l = last; l >= first; --l) {
        const Layer& L = net.layers[l];
        Rect in;
        back_interval(r.y0, r.y1, L.k, L.stride, L.pad, L.h_in, &in.y0, &in.y1);
        back_interval(r.x0, r.x1, L.k, L.stride, L.pad, L.w_in, &in.x0, &in.x1);
        if (r.empty()) in = Rect{};
        out_rects[l] = r;
        in_rects[l] = in;
        r = in;
    }
}

double predict_layer_group(const Net& net, int first, int last, int n, int m, double bias_mib,
                           int input_factor) {
    double best = 0.0;
    std::vector<Rect> outs, ins;
    for (int i = 0; i < n; ++i)
        for (int j = 0; j < m; ++j) {
            tile_regions(net, first, last, n, m, i, j, outs, ins);
            for (int l = first; l <= last; ++l) {
                const Layer& L = net.layers[l];
                double w_out = outs[l].w(), h_out = outs[l].h();
                double w_in = ins[l].w(), h_in = ins[l].h();
                double scratch = w_out * h_out * (double)L.c_in * (double)(L.k * L.k) / (double)L.stride;
                double input = w_in * h_in * (double)L.c_in;
                double output = w_out * h_out * (double)L.c_out;
                double mem = scratch + output + input * (double)input_factor;
                if (mem > best) best = mem;
            }
        }
    return best * 4.0 / (double)(1 << 20) + bias_mib;
}

double predict_mem(const Net& net, int cut, int n1, int m1, int n2, int m2, double bias_mib) {
    int n = (int)net.layers.size();
    if (cut <= 0 || cut >= n) return predict_layer_group(net, 0, n - 1, n1, m1, bias_mib, 2);
    double a = predict_layer_group(net, 0, cut - 1, n1, m1, bias_mib, 2);
    double b = predict_layer_group(net, cut, n - 1, n2, m2, bias_mib, 2);
    return std::max(a, b);
}

void search(const Net& net, double limit_mib, double bias_mib, int* top, int* cut, int* bottom) {
    const int n = (int)net.layers.size();
    const int cuts[3] = {n, 12, 8};
    const int bottom_tile = 2;
    int lg1 = 0, c = 0;
    for (int ci = 0; ci < 3; ++ci) {
        c = cuts[ci];
        for (int tile = 1; tile <= 5; ++tile) {
            lg1 = tile;
            double p = predict_mem(net, c, tile, tile, bottom_tile, bottom_tile, bias_mib);
            if (p < limit_mib) {
                *top = lg1;
                *cut = c;
                *bottom = bottom_tile;
                return;
            }
        }
    }
    *top = lg1;
    *cut = c;
    *bottom = bottom_tile;
}

uint16_t f32_to_bf16_rne(float f) {
    uint32_t u;
    std::memcpy(&u, &f, 4);
    if ((u & 0x7f800000u) == 0x7f800000u && (u & 0x007fffffu)) return (uint16_t)((u >> 16) | 0x40);  // quiet NaN
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

namespace {

struct TileInfo {
    int i, j;
    std::vector<Rect> outs, ins;
};

int largest_nblk(int cout) {
    for (int d = MAFAT_MAX_NBLK; d >= 16; d -= 16)
        if (cout % d == 0) return d;
    return 16;
}

}  // namespace

std::string build_plan(const Net& net, const PlanConfig& cfg, PlanTables& t, bool* unsupported) {
    *unsupported = false;
    const int n = (int)net.layers.size();
    t = PlanTables{};
    t.cfg = cfg;
    if (cfg.n_groups < 1 || cfg.n_groups > MAFAT_MAX_GROUPS) return "n_groups must be 1..4";
    for (int c = 0; c + 1 < cfg.n_groups; ++c) {
        if (cfg.cuts[c] <= 0 || cfg.cuts[c] >= n) return "cuts must be in 1..n-1";
        if (c > 0 && cfg.cuts[c] <= cfg.cuts[c - 1]) return "cuts must increase";
    }
    if (cfg.batch <= 0) return "batch must be positive";
    if (cfg.dtype != 0 && cfg.dtype != 1) return "unknown dtype";
    for (int g = 0; g < cfg.n_groups; ++g)
        if (cfg.grid_n[g] <= 0 || cfg.grid_m[g] <= 0) return "grid sizes must be positive";
    const int G = cfg.n_groups;
    for (int g = 0; g < G; ++g) {
        t.groups[g][0] = g == 0 ? 0 : cfg.cuts[g - 1];
        t.groups[g][1] = g == G - 1 ? n - 1 : cfg.cuts[g] - 1;
    }

    // ---- tiles of every group (non-empty only), on the even grid or the given bounds
    std::vector<std::vector<TileInfo>> tiles(G);
    int max_tiles = 1;
    for (int g = 0; g < G; ++g) {
        const Layer& Lg = net.layers[t.groups[g][1]];
        if (!cfg.row_bounds[g].empty() || !cfg.col_bounds[g].empty()) {
            std::string e = check_bounds(cfg.row_bounds[g], Lg.h_out, cfg.grid_n[g]);
            if (e.empty()) e = check_bounds(cfg.col_bounds[g], Lg.w_out, cfg.grid_m[g]);
            if (!e.empty()) return "group " + std::to_string(g + 1) + ": " + e;
        }
        t.rows[g] = axis_bounds(Lg.h_out, cfg.grid_n[g], cfg.row_bounds[g]);
        t.cols[g] = axis_bounds(Lg.w_out, cfg.grid_m[g], cfg.col_bounds[g]);
        for (int i = 0; i < cfg.grid_n[g]; ++i)
            for (int j = 0; j < cfg.grid_m[g]; ++j) {
                TileInfo ti;
                ti.i = i;
                ti.j = j;
                Rect r;
                r.y0 = t.rows[g][i];
                r.y1 = t.rows[g][i + 1];
                r.x0 = t.cols[g][j];
                r.x1 = t.cols[g][j + 1];
                if (cfg.halo_reuse)
                    owned_regions(net, t.groups[g][0], t.groups[g][1], r, ti.outs, ti.ins);
                else
                    rect_regions(net, t.groups[g][0], t.groups[g][1], r, ti.outs, ti.ins);
                if (ti.outs[t.groups[g][1]].empty()) continue;
                tiles[g].push_back(std::move(ti));
            }
        max_tiles = std::max(max_tiles, (int)tiles[g].size());
    }

    // ---- fused stages: a conv, plus the max-pool that directly follows it in the same group
    const int n_ctas = cfg.n_ctas > 0 ? cfg.n_ctas : 152;
    std::vector<int> stage_pool_layer;
    for (int g = 0; g < G; ++g) {
        int first = t.groups[g][0], last = t.groups[g][1];
        t.stage_first[g] = (int)t.stages.size();
        for (int l = first; l <= last; ++l) {
            const Layer& L = net.layers[l];
            if (L.type == L_MAXPOOL) {
                *unsupported = true;
                return "layer " + std::to_string(l) + ": a max-pool must directly follow a convolution of its group";
            }
            if (!net.has_w[l]) return "layer " + std::to_string(l) + ": weights not set";
            MafatStageDev s{};
            s.layer = l;
            s.k = L.k;
            s.pad = L.pad;
            s.cin = L.c_in;
            s.cin8 = ceil_div(L.c_in, 8);
            s.cout = L.c_out;
            s.pool = (l + 1 <= last && net.layers[l + 1].type == L_MAXPOOL) ? 1 : 0;
            if (s.cin8 != 1 && s.cin8 % 2 != 0) {
                *unsupported = true;
                return "layer " + std::to_string(l) + ": input channels above 8 must be a multiple of 16";
            }
            // M blocks of this stage over the tiles of one frame: frames go through a stage one
            // after another (or overlapped with another group), never all side by side, so
            // a stage's parallelism is one frame's
            int64_t blocks = 0;
            for (const TileInfo& ti : tiles[g]) {
                const Rect& cr = ti.outs[l];
                blocks += (int64_t)ceil_div(cr.h(), MAFAT_BLK_ROWS) * ceil_div(cr.w(), MAFAT_BLK_COLS);
            }
            // Output-channel block (MMA N, a multiple of 16 dividing the padded cout; zero
            // weights pad it, only cout channels are stored): the narrowest block of at least
            // 64 channels whose items fit one wave of CTAs, else the widest.  A stage with few
            // M blocks (the small maps after the cut) then spreads over the SMs without a
            // second wave, which its successor would wait for; below N = 64 the MMA's A read
            // dominates.  Stages with more blocks than CTAs keep the widest block, which
            // reuses every A operand for the most output channels.
            const int cout_pad = (L.c_out + 15) / 16 * 16;
            // On-chip chaining (option; tensor-core plans, halo recompute): a 3x3 convolution
            // without a fused pool whose next layer is a 1x1 convolution of the same group runs
            // both in one item when the 3x3's accumulator, its bf16 result and the 1x1's
            // accumulator fit one 256-column TMEM buffer for a block of 128 pixels; the 1x1's
            // stage has no tasks.
            const bool prev_chain = !t.stages.empty() && t.stage_first[g] < (int)t.stages.size() &&
                                    t.stages.back().chain;
            bool chain_here = false;
            if (cfg.dtype == 0 && !cfg.halo_reuse && cfg.chain && !prev_chain && L.k == 3 && l + 1 <= last &&
                net.layers[l + 1].type == L_CONV && net.layers[l + 1].k == 1) {
                const int next_pad = (net.layers[l + 1].c_out + 15) / 16 * 16;
                chain_here = cout_pad % 64 == 0 && cout_pad + cout_pad / 2 + next_pad <= 256;
            }
            // Flattened M blocks (MafatStageDev::flat) where they take fewer blocks than 16 x 8
            // rectangles: convolutions without a fused pool (a pool window's four pixels are
            // lanes of one warp only in a rectangle), of more than 8 input channels (the
            // paired-tap form of one-octet inputs keeps rectangles) and outside a chained pair,
            // whose widest region needs a pitch of at most 32 pixels (a tensor-map box row
            // holds at most 256 elements, 8 per pixel).
            int flat_pitch = 0;
            if (!cfg.rect_blocks && !s.pool && s.cin8 > 1 && !chain_here && !prev_chain) {
                int pitch = 0;
                for (const TileInfo& ti : tiles[g])
                    if (!ti.outs[l].empty()) pitch = std::max(pitch, (ti.outs[l].w() + L.k - 1 + 7) / 8 * 8);
                int64_t flat_blocks = 0;
                for (const TileInfo& ti : tiles[g]) flat_blocks += ((int64_t)ti.outs[l].h() * pitch + 127) / 128;
                if (pitch > 0 && pitch <= 32 && flat_blocks < blocks) {
                    flat_pitch = pitch;
                    blocks = flat_blocks;
                }
            }
            s.flat = flat_pitch > 0 ? 1 : 0;
            // With several frames in flight the SMs are kept busy by the next frame anyway, and an
            // item reads its whole K = c_in * k * k halo for n_blk channels: there the narrowest
            // block considered is 128 (608x608, 16 frames: 1x1 layers at N = 64 -> 128, 83.0 ->
            // 81.3 us per frame; then the flat 3x3 layers after the cut too, 83.5 -> 79.7 us; at
            // one frame the extra parallelism of N = 64 wins, 117.4 against 121.5 us).
            const int min_nb = cfg.batch > 1 ? 128 : 64;
            if (chain_here || prev_chain) {
                s.n_blk = cout_pad;  // every channel of the pixels in one item
            } else if (cfg.fixed_nblk > 0 && cout_pad % cfg.fixed_nblk == 0) {
                s.n_blk = cfg.fixed_nblk;
            } else {
                s.n_blk = largest_nblk(cout_pad);
                for (int nb = std::min(min_nb, cout_pad); nb <= std::min(cout_pad, MAFAT_MAX_NBLK); nb += 16) {
                    if (cout_pad % nb != 0) continue;
                    if (blocks * (cout_pad / nb) <= n_ctas) {
                        s.n_blk = nb;
                        break;
                    }
                }
            }
            s.n_nblk = cout_pad / s.n_blk;
            // Blocks per item (stacked along rows, one accumulator each, sharing every
            // weight blob): grow while the stage keeps at least one item per CTA.
            s.mb = 1;
            if (chain_here || prev_chain) {
                // one 128-pixel block per item: the chained pair's three TMEM regions fill a buffer
            } else if (cfg.fixed_mb > 0) {
                s.mb = cfg.fixed_mb;
            } else {
                while (s.mb * 2 * s.n_blk <= 256 && blocks * s.n_nblk / (s.mb * 2) >= n_ctas) s.mb *= 2;
            }
            if (s.mb * s.n_blk > 256) s.mb = std::max(1, 256 / s.n_blk);
            // the kernel has MMA code for 1..4 blocks per item, and 1..8 for the paired-tap
            // form of 8-input-channel layers (narrow N, many small items: their epilogue's
            // fixed cost per item dominates)
            s.mb = std::min(s.mb, s.cin8 == 1 ? MAFAT_MAX_MB_PAIRED : MAFAT_MAX_MB);
            s.cols_box = s.flat ? flat_pitch : MAFAT_BLK_COLS + L.k - 1;
            // How the caller's NHWC input reaches the first stage's A halo (tensor-core plans; the
            // fp32 kernel reads NHWC directly).  An image of fewer than 8 channels is read in place
            // as raw rows, which a TMA box needs to be a multiple of 16 bytes; 8 channels are one
            // octet plane already.  Other inputs (rows of another size, or more than 8 channels,
            // i.e. not an image) are converted to octet-planar by a small kernel before the launch.
            s.in_mode = MAFAT_IN_PLANAR;
            s.raw_e = 0;
            s.pix_pair = 0;
            s.blk_halo = 0;
            if (l == 0 && cfg.dtype == 0) {
                if (L.c_in < 8 && ((int64_t)L.w_in * L.c_in) % 8 == 0) {
                    s.in_mode = MAFAT_IN_GATHER;
                    // up to 7 leading elements of alignment; pixel pairs read one pixel more
                    s.pix_pair = (L.c_in <= 4 && L.k == 3) ? 1 : 0;
                    s.blk_halo = 1;
                    s.raw_e = (L.c_in * (s.cols_box + s.pix_pair) + 7 + 7) / 8 * 8;
                } else if (L.c_in != 8) {
                    t.in_convert = 1;
                }
            }
            // input octets per A chunk: the largest that fits the A stage with mb blocks
            for (;;) {
                s.rows_box = s.flat       ? mafat_flat_rows(s.mb, s.cols_box, L.k)
                             : s.blk_halo ? (MAFAT_BLK_ROWS + L.k - 1) * s.mb
                                          : MAFAT_BLK_ROWS * s.mb + L.k - 1;
                const int row_bytes = s.cols_box * 16 * s.rows_box;
                if (s.in_mode == MAFAT_IN_GATHER) {
                    // the expanded halos plus the raw rows they are built from share the stage
                    s.chunk8 = 1;
                    if (mafat_raw_offset(s.rows_box, s.cols_box) + s.mb * mafat_raw_blk_stride(L.k, s.raw_e) <=
                            MAFAT_A_STAGE_BYTES ||
                        s.mb == 1)
                        break;
                    s.mb /= 2;
                    continue;
                }
                if (s.cin8 == 1) {
                    s.chunk8 = 1;
                } else {
                    s.chunk8 = 0;
                    for (int d = 8; d >= 2; d /= 2)  // 8, 4 or 2 octets: 4, 2 or 1 K steps per blob
                        if (s.cin8 % d == 0 && d * row_bytes <= MAFAT_A_STAGE_BYTES) {
                            s.chunk8 = d;
                            break;
                        }
                }
                if ((s.chunk8 > 0 && s.chunk8 * row_bytes <= MAFAT_A_STAGE_BYTES) || s.mb == 1) break;
                s.mb /= 2;
            }
            if (s.chunk8 == 0) return "internal: no A chunk fits the shared-memory stage";
            if (s.cin8 == 1) {
                s.paired = 1;
                s.n_chunks = 1;
                s.n_bsteps = s.pix_pair ? L.k : ceil_div(L.k * L.k, 2);  // a kernel row, or two taps, per K step
                s.kst = 1;
            } else {
                s.paired = 0;
                s.n_chunks = s.cin8 / s.chunk8;
                s.n_bsteps = L.k * L.k;
                s.kst = s.chunk8 / 2;
            }
            // 64-channel blobs use the 128-byte swizzled layout: one 128-byte row per
            // output channel, 8-row atoms of 1024 bytes (the MMA streams them faster
            // than no-swizzle core matrices); narrower blobs stay unswizzled.
            s.b_swz = s.kst == 4 ? 1 : 0;
            s.blob_elems = s.n_blk * 16 * s.kst;
            s.set_bytes = s.n_chunks * s.n_bsteps * s.blob_elems * 2;
            // Weights travel in pieces of whole blobs that fill one shared-memory buffer:
            // a set that fits one piece stays resident across items, larger sets stream
            // through the two buffers (every copy has a fixed cost, so pieces are large).
            s.bpp = std::max(1, MAFAT_B_PIECE_BYTES / (s.blob_elems * 2));
            s.bpp = std::min(s.bpp, s.n_chunks * s.n_bsteps);
            s.n_pieces = ceil_div(s.n_chunks * s.n_bsteps, s.bpp);
            if (s.blob_elems * 2 > MAFAT_B_PIECE_BYTES) {
                *unsupported = true;
                return "layer " + std::to_string(l) + ": one weight blob exceeds a shared-memory buffer";
            }
            s.w_off = t.weight_elems;
            t.weight_elems += (int64_t)s.n_nblk * s.n_chunks * s.n_bsteps * s.blob_elems;
            s.w32_off = t.weight32_elems;
            t.weight32_elems += (int64_t)L.c_out * L.c_in * L.k * L.k;
            s.sb_off = (int)t.sb_elems;
            t.sb_elems += cout_pad;
            s.chain = chain_here ? 1 : 0;
            s.chained = prev_chain ? 1 : 0;
            if (chain_here) {
                s.chain_a_col = cout_pad;
                s.chain_out_col = cout_pad + cout_pad / 2;
            }
            t.stages.push_back(s);
            stage_pool_layer.push_back(s.pool ? l + 1 : -1);
            if (s.pool) ++l;
        }
        t.stage_last[g] = (int)t.stages.size() - 1;
    }
    // a chain stage carries the fields of its chained 1x1 that the kernel reads
    for (size_t si = 0; si + 1 < t.stages.size(); ++si) {
        MafatStageDev& a = t.stages[si];
        if (!a.chain) continue;
        const MafatStageDev& b = t.stages[si + 1];
        a.c2_n_blk = b.n_blk;
        a.c2_cout = b.cout;
        a.c2_pool = b.pool;
        a.c2_n_chunks = b.n_chunks;
        a.c2_kst = b.kst;
        a.c2_b_swz = b.b_swz;
        a.c2_bpp = b.bpp;
        a.c2_n_pieces = b.n_pieces;
        a.c2_blob_elems = b.blob_elems;
        a.c2_sb_off = b.sb_off;
        a.c2_w_off = b.w_off;
    }

    // ---- geometry of the group inputs / outputs
    const Layer& L0 = net.layers[0];
    t.in_c8 = ceil_div(L0.c_in, 8);
    const MafatStageDev& s_in = t.stages[t.stage_first[0]];
    t.in_rows_box = s_in.rows_box;
    t.in_cols_box = s_in.cols_box;
    t.in_chunk8 = s_in.chunk8;
    if (G >= 2) {
        const Layer& Lc = net.layers[t.groups[0][1]];
        t.cut_h = Lc.h_out;
        t.cut_w = Lc.w_out;
        t.cut_c8 = ceil_div(Lc.c_out, 8);
        const MafatStageDev& s2 = t.stages[t.stage_first[1]];
        t.cut_rows_box = s2.rows_box;
        t.cut_cols_box = s2.cols_box;
        t.cut_chunk8 = s2.chunk8;
    }
    const Layer& Ln = net.layers[n - 1];
    t.out_h = Ln.h_out;
    t.out_w = Ln.w_out;
    t.out_c = Ln.c_out;
    const int64_t in_frame = (int64_t)L0.c_in * L0.h_in * L0.w_in;  // the caller's NHWC input
    const int64_t cut_frame = (int64_t)t.cut_c8 * 8 * t.cut_h * t.cut_w;
    const int64_t out_frame = (int64_t)t.out_h * t.out_w * t.out_c;

    // The ring holds one frame's tiles of every group when several frames go through it, so
    // that a tile's slot predecessor is the same tile of the previous frame (the frames'
    // groups may then overlap in the hand-out order below)
    int tiles_per_frame = 0;
    for (int g = 0; g < G; ++g) tiles_per_frame += (int)tiles[g].size();
    int S = cfg.ring_slots > 0 ? cfg.ring_slots
            : cfg.batch > 1    ? std::min(std::max(max_tiles, tiles_per_frame), 256)
                               : std::min(max_tiles, 64);
    int W = cfg.wave_tiles > 0 ? std::min(cfg.wave_tiles, S) : S;
    if (cfg.halo_reuse) {
        // a layer's tasks read their neighbours' previous layer, so every tile of a group
        // goes out stage by stage in one wave; there is no ring
        S = W = max_tiles;
    }
    t.ring_slots = cfg.halo_reuse ? 0 : S;
    t.wave_tiles = W;

    // ---- scratch buffer size: largest non-final stage output of any tile
    int64_t buf = 0;
    for (int g = 0; g < G; ++g)
        for (const TileInfo& ti : tiles[g])
            for (int s = t.stage_first[g]; s < t.stage_last[g]; ++s) {
                const MafatStageDev& st = t.stages[s];
                int ol = stage_pool_layer[s] >= 0 ? stage_pool_layer[s] : st.layer;
                const Rect& r = ti.outs[ol];
                buf = std::max(buf, (int64_t)r.h() * r.w() * ceil_div(st.cout, 8) * 8);
            }
    t.slot_buf_elems = (buf + 127) / 128 * 128;  // 256-byte aligned for bf16, 512 for fp32
    t.scratch_elems = (int64_t)S * 2 * t.slot_buf_elems;
    // halo reuse: one whole output map per non-final stage, every frame, instead of the ring
    std::vector<int64_t> map_off(t.stages.size(), -1), map_frame(t.stages.size(), 0);
    std::vector<int> map_h(t.stages.size(), 0), map_w(t.stages.size(), 0), stage_tmap(t.stages.size(), -1);
    if (cfg.halo_reuse) {
        int64_t off = 0;
        for (int g = 0; g < G; ++g)
            for (int s = t.stage_first[g]; s < t.stage_last[g]; ++s) {
                const MafatStageDev& st = t.stages[s];
                const Layer& Lo = net.layers[stage_pool_layer[s] >= 0 ? stage_pool_layer[s] : st.layer];
                map_h[s] = Lo.h_out;
                map_w[s] = Lo.w_out;
                map_frame[s] = (int64_t)ceil_div(st.cout, 8) * 8 * Lo.h_out * Lo.w_out;
                map_off[s] = off;
                off += (map_frame[s] * cfg.batch + 127) / 128 * 128;
            }
        t.scratch_elems = std::max<int64_t>(off, 128);
        t.slot_buf_elems = 0;
        for (int g = 0; g < G; ++g)
            for (int s = t.stage_first[g] + 1; s <= t.stage_last[g]; ++s) {
                const MafatStageDev& st = t.stages[s];
                TmapReq req{};
                req.task = -1;
                req.elem_off = map_off[s - 1];
                req.h = map_h[s - 1];
                req.w = map_w[s - 1];
                req.c8 = st.cin8;
                req.frames = cfg.batch;
                req.rows_box = st.rows_box;
                req.cols_box = st.cols_box;
                req.chunk8 = st.chunk8;
                stage_tmap[s] = (int)t.tmaps.size();
                t.tmaps.push_back(req);
            }
    }

    // ---- outputs of groups 2 .. G-1 (group 1's is the cut tensor): whole maps of every
    // frame after the ring or the layer maps, read by the next group's first stage through
    // a tensor map of its own
    std::vector<int64_t> bmap_off(G, -1), bmap_frame(G, 0);
    for (int g = 1; g + 1 < G; ++g) {
        const int s_last = t.stage_last[g];
        const MafatStageDev& st = t.stages[s_last];
        const Layer& Lo = net.layers[t.groups[g][1]];
        bmap_frame[g] = (int64_t)ceil_div(st.cout, 8) * 8 * Lo.h_out * Lo.w_out;
        bmap_off[g] = (t.scratch_elems + 127) / 128 * 128;
        t.scratch_elems = bmap_off[g] + bmap_frame[g] * cfg.batch;
        const int s_next = t.stage_first[g + 1];
        const MafatStageDev& sn = t.stages[s_next];
        TmapReq req{};
        req.task = -1;
        req.elem_off = bmap_off[g];
        req.h = Lo.h_out;
        req.w = Lo.w_out;
        req.c8 = sn.cin8;
        req.frames = cfg.batch;
        req.rows_box = sn.rows_box;
        req.cols_box = sn.cols_box;
        req.chunk8 = sn.chunk8;
        stage_tmap[s_next] = (int)t.tmaps.size();
        t.tmaps.push_back(req);
    }

    // ---- tasks in hand-out order, with their dependencies expressed as task indices
    struct TaskDep {
        int prev_task = -1;    // previous stage of the same tile, or the ring predecessor's last stage
        int group_ctr = -1;    // (frame, group) counter whose group must be complete (first stages)
        int bump_ctr = -1;     // (frame, group) counter this last stage of a group bumps
    };
    std::vector<TaskDep> deps;
    std::vector<int> last_task_of_seq;
    int seq = 0;
    for (int f = 0; f < cfg.batch; ++f) {
        for (int g = 0; g < G; ++g) {
            const auto& tl = tiles[g];
            for (size_t w0 = 0; w0 < tl.size(); w0 += W) {
                size_t w1 = std::min(tl.size(), w0 + (size_t)W);
                std::vector<int> prev_of_tile(w1 - w0, -1);
                int rel = -1;  // index of the stage among the group's stages that have tasks
                for (int s = t.stage_first[g]; s <= t.stage_last[g]; ++s) {
                    const MafatStageDev& st = t.stages[s];
                    if (st.chained) continue;  // runs inside the items of the chain stage before it
                    ++rel;
                    // the stage whose output this task writes: its own, or the chained 1x1's
                    const int s_out = st.chain ? s + 1 : s;
                    const Layer& Lc = net.layers[st.layer];
                    const std::vector<int> prev_stage_task = prev_of_tile;  // previous task stage of each tile
                    for (size_t q = w0; q < w1; ++q) {
                        const TileInfo& ti = tl[q];
                        int tseq = seq + (int)(q - w0);
                        int slot = tseq % S;
                        MafatTaskDev tk{};
                        tk.stage = s;
                        tk.frame = f;
                        const Rect& cr = ti.outs[st.layer];
                        const Rect& ir = ti.ins[st.layer];
                        int ol = stage_pool_layer[s_out] >= 0 ? stage_pool_layer[s_out] : t.stages[s_out].layer;
                        const Rect& orr = ti.outs[ol];
                        if (st.chain && !(ti.outs[t.stages[s_out].layer] == cr))
                            return "internal: chained 1x1 region differs from its 3x3";
                        if (t.stages[s_out].pool) {
                            // the conv region of a pooled stage is exactly twice the pooled region
                            if (!(cr.y0 == 2 * orr.y0 && cr.y1 == 2 * orr.y1 && cr.x0 == 2 * orr.x0 &&
                                  cr.x1 == 2 * orr.x1))
                                return "internal: pooled region mismatch";
                        }
                        tk.cy0 = cr.y0;
                        tk.cx0 = cr.x0;
                        tk.ch = cr.h();
                        tk.cw = cr.w();
                        tk.nby = st.flat ? ceil_div(tk.ch * st.cols_box, 128) : ceil_div(tk.ch, MAFAT_BLK_ROWS);
                        tk.nbx = st.flat ? 1 : ceil_div(tk.cw, MAFAT_BLK_COLS);
                        if (s == t.stage_first[g]) {
                            tk.in_kind = g == 0 ? MAFAT_BUF_USER_IN : g == 1 ? MAFAT_BUF_CUT : MAFAT_BUF_MAP;
                            tk.in_tmap = g >= 2 ? stage_tmap[s] : -1;
                            tk.in_off = g == 0 ? f * in_frame : g == 1 ? f * cut_frame : bmap_off[g - 1] + f * bmap_frame[g - 1];
                            tk.in_h = Lc.h_in;
                            tk.in_w = Lc.w_in;
                            tk.in_y0 = 0;
                            tk.in_x0 = 0;
                        } else if (cfg.halo_reuse) {
                            tk.in_kind = MAFAT_BUF_MAP;
                            tk.in_off = map_off[s - 1] + f * map_frame[s - 1];
                            tk.in_h = map_h[s - 1];
                            tk.in_w = map_w[s - 1];
                            tk.in_y0 = 0;
                            tk.in_x0 = 0;
                            tk.in_tmap = stage_tmap[s];
                        } else {
                            int b = (slot * 2) + ((rel - 1) & 1);
                            tk.in_kind = MAFAT_BUF_SCRATCH;
                            tk.in_off = (int64_t)b * t.slot_buf_elems;
                            tk.in_h = ir.h();
                            tk.in_w = ir.w();
                            tk.in_y0 = ir.y0;
                            tk.in_x0 = ir.x0;
                            TmapReq req{};
                            req.task = (int)t.tasks.size();
                            req.elem_off = (int64_t)b * t.slot_buf_elems;
                            req.frames = 1;
                            req.h = ir.h();
                            req.w = ir.w();
                            req.c8 = st.cin8;
                            req.rows_box = st.rows_box;
                            req.cols_box = st.cols_box;
                            req.chunk8 = st.chunk8;
                            tk.in_tmap = (int)t.tmaps.size();
                            t.tmaps.push_back(req);
                        }
                        if (s_out == t.stage_last[g]) {
                            if (g == G - 1) {
                                tk.out_kind = MAFAT_BUF_USER_OUT;
                                tk.out_nhwc = 1;
                                tk.out_off = f * out_frame;
                                tk.out_h = t.out_h;
                                tk.out_w = t.out_w;
                            } else if (g == 0) {
                                tk.out_kind = MAFAT_BUF_CUT;
                                tk.out_nhwc = 0;
                                tk.out_off = f * cut_frame;
                                tk.out_h = t.cut_h;
                                tk.out_w = t.cut_w;
                            } else {
                                tk.out_kind = MAFAT_BUF_MAP;
                                tk.out_nhwc = 0;
                                tk.out_off = bmap_off[g] + f * bmap_frame[g];
                                tk.out_h = net.layers[t.groups[g][1]].h_out;
                                tk.out_w = net.layers[t.groups[g][1]].w_out;
                            }
                            tk.out_y0 = 0;
                            tk.out_x0 = 0;
                        } else if (cfg.halo_reuse) {
                            tk.out_kind = MAFAT_BUF_MAP;
                            tk.out_nhwc = 0;
                            tk.out_off = map_off[s] + f * map_frame[s];
                            tk.out_h = map_h[s];
                            tk.out_w = map_w[s];
                            tk.out_y0 = 0;
                            tk.out_x0 = 0;
                        } else {
                            int b = (slot * 2) + (rel & 1);
                            tk.out_kind = MAFAT_BUF_SCRATCH;
                            tk.out_nhwc = 0;
                            tk.out_off = (int64_t)b * t.slot_buf_elems;
                            tk.out_h = orr.h();
                            tk.out_w = orr.w();
                            tk.out_y0 = orr.y0;
                            tk.out_x0 = orr.x0;
                        }
                        tk.n_items = (st.blk_halo ? ceil_div(tk.nby * tk.nbx, st.mb) : ceil_div(tk.nby, st.mb) * tk.nbx) *
                                     st.n_nblk;
                        TaskDep d;
                        int qi = (int)(q - w0);
                        if (s == t.stage_first[g]) {
                            if (!cfg.halo_reuse && tseq >= S) d.prev_task = last_task_of_seq[tseq - S];
                            if (g >= 1) d.group_ctr = f * (G - 1) + (g - 1);
                        } else if (cfg.halo_reuse) {
                            // every previous-stage task whose owned output meets this task's input
                            // region (halo included): itself and the neighbours around it
                            const int ps = s - 1;
                            const int pol = stage_pool_layer[ps] >= 0 ? stage_pool_layer[ps] : t.stages[ps].layer;
                            const Rect& need = ti.ins[st.layer];
                            tk.dep_first = (int)t.deps.size();
                            for (size_t q2 = w0; q2 < w1; ++q2) {
                                const Rect& own = tl[q2].outs[pol];
                                if (own.empty() || need.empty() || own.y1 <= need.y0 || need.y1 <= own.y0 ||
                                    own.x1 <= need.x0 || need.x1 <= own.x0)
                                    continue;
                                const int pt = prev_stage_task[q2 - w0];
                                t.deps.push_back(MafatDepDev{MAFAT_CTR_BASE + pt, t.tasks[pt].n_items});
                            }
                            tk.dep_count = (int)t.deps.size() - tk.dep_first;
                        } else {
                            d.prev_task = prev_of_tile[qi];
                        }
                        if (g + 1 < G && s_out == t.stage_last[g]) d.bump_ctr = f * (G - 1) + g;
                        prev_of_tile[qi] = (int)t.tasks.size();
                        t.tasks.push_back(tk);
                        deps.push_back(d);
                        // statistics (a chain task does the work of both of its stages)
                        for (int sx = s; sx <= s_out; ++sx) {
                            const MafatStageDev& sw = t.stages[sx];
                            const double kk = (double)sw.k * sw.k;
                            t.executed_flops += 2.0 * cr.h() * cr.w() * (double)sw.cout * sw.cin * kk;
                            t.issued_flops += 2.0 * tk.nby * tk.nbx * (double)(MAFAT_BLK_ROWS * MAFAT_BLK_COLS) *
                                              (double)sw.n_nblk * sw.n_blk * sw.n_chunks * sw.n_bsteps * sw.kst * 16.0;
                        }
                    }
                }
                for (size_t q = w0; q < w1; ++q) last_task_of_seq.push_back(prev_of_tile[q - w0]);
                seq += (int)(w1 - w0);
            }
        }
    }
    t.n_tiles = seq;

    // ---- frames in flight (batch > 1, two groups): the second group of a frame is a chain of
    // stages over a few small tiles that leaves most SMs idle, so the next frame's first-group
    // tasks are handed out between its stages (shares below).  Every
    // dependency still points to an earlier task: a first-group task depends on its own frame's
    // earlier tasks and on the same tile of the previous frame (its ring slot); a second-group
    // task on its own frame's first group, all of which was handed out before.
    if (cfg.batch > 1 && G == 2 && !cfg.halo_reuse && !cfg.frame_major && S >= tiles_per_frame && W >= max_tiles) {
        const int n_t = (int)t.tasks.size();
        std::vector<std::vector<int>> fill(cfg.batch), chain(cfg.batch);
        for (int i = 0; i < n_t; ++i)
            (t.tasks[i].stage <= t.stage_last[0] ? fill : chain)[t.tasks[i].frame].push_back(i);
        std::vector<int> order;
        order.reserve(n_t);
        order.insert(order.end(), fill[0].begin(), fill[0].end());
        for (int f = 0; f < cfg.batch; ++f) {
            const std::vector<int>& cf = chain[f];
            std::vector<size_t> cuts_at;  // starts of the runs of one stage
            for (size_t i = 0; i < cf.size(); ++i)
                if (i == 0 || t.tasks[cf[i]].stage != t.tasks[cf[i - 1]].stage) cuts_at.push_back(i);
            cuts_at.push_back(cf.size());
            static const std::vector<int> none;
            const std::vector<int>& nx = f + 1 < cfg.batch ? fill[f + 1] : none;
            int64_t nx_items = 0;
            for (int i : nx) nx_items += t.tasks[i].n_items;
            // Share of the next frame's first group handed out behind each second-group stage:
            // in proportion to the stage's estimated duration, in units of one 128x128x16 MMA
            // (a fixed part for the halo load, epilogue and completion round trip, plus the
            // MMAs of one item), and a share ahead of the first stage, whose CTAs would
            // otherwise wait for the whole first group of their own frame (measured on the
            // 608x608 network, 16 frames: 83 us per frame against 88 with an even split).
            const size_t n_runs = cuts_at.size() - 1;
            const double kFixedMma = 72.0, kAheadMma = 288.0;
            std::vector<double> share(n_runs + 1, 0.0);
            share[0] = kAheadMma;
            double total = kAheadMma;
            for (size_t r = 0; r < n_runs; ++r) {
                const MafatStageDev& st = t.stages[t.tasks[cf[cuts_at[r]]].stage];
                share[r + 1] = kFixedMma + (double)st.n_blk / 128.0 * st.n_chunks * st.n_bsteps * st.kst * st.mb;
                total += share[r + 1];
            }
            size_t pos = 0;
            int64_t taken = 0;
            double acc = 0.0;
            for (size_t r = 0; r <= n_runs; ++r) {
                if (r > 0)
                    for (size_t i = cuts_at[r - 1]; i < cuts_at[r]; ++i) order.push_back(cf[i]);
                acc += share[r];
                const int64_t target = (int64_t)((double)nx_items * acc / total + 0.5);
                while (pos < nx.size() && taken < target) {
                    taken += t.tasks[nx[pos]].n_items;
                    order.push_back(nx[pos++]);
                }
            }
            while (pos < nx.size()) order.push_back(nx[pos++]);
        }
        if ((int)order.size() != n_t) return "internal: frame interleave lost a task";
        std::vector<int> new_of(n_t);
        for (int k = 0; k < n_t; ++k) new_of[order[k]] = k;
        std::vector<MafatTaskDev> tasks2(n_t);
        std::vector<TaskDep> deps2(n_t);
        for (int k = 0; k < n_t; ++k) {
            tasks2[k] = t.tasks[order[k]];
            deps2[k] = deps[order[k]];
            if (deps2[k].prev_task >= 0) deps2[k].prev_task = new_of[deps2[k].prev_task];
        }
        t.tasks.swap(tasks2);
        deps.swap(deps2);
        for (TmapReq& r : t.tmaps)
            if (r.task >= 0) r.task = new_of[r.task];
        t.frames_overlapped = 1;
    }

    // ---- counters: one per task, then one per frame (group-1 completion)
    const int n_tasks = (int)t.tasks.size();
    t.frame_ctr_base = MAFAT_CTR_BASE + n_tasks;
    t.n_counters = n_tasks + cfg.batch * (G - 1);
    std::vector<int> group_items((size_t)cfg.batch * std::max(G - 1, 1), 0);
    for (int ti = 0; ti < n_tasks; ++ti) {
        t.tasks[ti].done_ctr = MAFAT_CTR_BASE + ti;
        if (deps[ti].bump_ctr >= 0) group_items[deps[ti].bump_ctr] += t.tasks[ti].n_items;
    }
    // ---- items
    for (int ti = 0; ti < n_tasks; ++ti) {
        const MafatTaskDev& tk = t.tasks[ti];
        const MafatStageDev& st = t.stages[tk.stage];
        const TaskDep& d = deps[ti];
        // channel-block major: consecutive items share a resident weight set; a task's block
        // rows are split evenly over ceil(nby / mb) items (9 rows at mb = 8 give 5 + 4, not
        // 8 + 1, whose 1-block item would pay a whole item's fixed cost for little work)
        // Per-block-halo stages pack the task's blocks, in column-major order, evenly into
        // ceil(blocks / mb) items whatever the block columns (`by` = first block, `bx` = 0).
        const int n_blocks = tk.nby * tk.nbx;
        const int n_rows = st.blk_halo ? ceil_div(n_blocks, st.mb) : ceil_div(tk.nby, st.mb);
        const int n_cols = st.blk_halo ? 1 : tk.nbx;
        const int n_span = st.blk_halo ? n_blocks : tk.nby;
        for (int nb = 0; nb < st.n_nblk; ++nb)
            for (int ri = 0; ri < n_rows; ++ri)
                for (int bx = 0; bx < n_cols; ++bx) {
                    const int by = ri * n_span / n_rows, by_end = (ri + 1) * n_span / n_rows;
                    MafatItemDev it{};
                    it.task = ti;
                    it.stage = (int16_t)tk.stage;
                    it.by = (int16_t)by;
                    it.nbk = (int16_t)(by_end - by);
                    it.bx = (int16_t)bx;
                    it.nb = (int16_t)nb;
                    it.flags = (ti == cfg.unpublished_task) ? 1 : 0;
                    it.dep0 = -1;
                    it.dep1 = -1;
                    it.extra_ctr = -1;
                    if (d.prev_task >= 0) {
                        it.dep0 = MAFAT_CTR_BASE + d.prev_task;
                        it.dep0_target = t.tasks[d.prev_task].n_items;
                    }
                    if (d.group_ctr >= 0) {
                        it.dep1 = t.frame_ctr_base + d.group_ctr;
                        it.dep1_target = group_items[d.group_ctr];
                    }
                    if (d.bump_ctr >= 0) it.extra_ctr = t.frame_ctr_base + d.bump_ctr;
                    t.items.push_back(it);
                }
    }
    if (t.items.size() > (size_t)0x7fffffff) return "too many work items";
    // Stages with many items (all tiles of one frame) keep every CTA busy whatever it holds,
    // so their CTAs take the next ticket early; stages with about a wave of items or fewer
    // take it only when the CTA can start it, so that no idle CTA waits for a busy one.
    // With frames overlapped the next frame keeps every CTA busy in any stage (608x608, 16
    // frames: 80.4 against 80.9 us per frame).
    {
        const int n_ctas = cfg.n_ctas > 0 ? cfg.n_ctas : 152;
        const int64_t thr = cfg.lookahead_items > 0 ? cfg.lookahead_items
                            : t.frames_overlapped  ? 1
                                                   : (int64_t)n_ctas * 5 / 4;
        std::vector<int64_t> stage_items(t.stages.size(), 0);
        for (const MafatTaskDev& tk : t.tasks)
            if (tk.frame == 0) stage_items[tk.stage] += tk.n_items;
        for (size_t s = 0; s < t.stages.size(); ++s)
            t.stages[s].lookahead = (cfg.lookahead_items >= 0 && stage_items[s] >= thr) ? 1 : 0;
    }

    // ---- statistics
    for (int l = 0; l < n; ++l) {
        const Layer& L = net.layers[l];
        if (L.type == L_CONV)
            t.useful_flops += 2.0 * L.h_out * L.w_out * (double)L.c_out * L.c_in * L.k * L.k * cfg.batch;
    }
    int64_t io = in_frame + out_frame + (G >= 2 ? 2 * cut_frame : 0);
    for (int g = 1; g + 1 < G; ++g) io += 2 * bmap_frame[g];
    t.group_io_elems = io * cfg.batch;
    if (G <= 2) {
        t.predicted_mib = predict_mem(net, G == 2 ? cfg.cuts[0] : 0, cfg.grid_n[0], cfg.grid_m[0],
                                      G == 2 ? cfg.grid_n[1] : 1, G == 2 ? cfg.grid_m[1] : 1, 31.0);
    } else {  // predictMem's maximum over the groups, for any number of them
        t.predicted_mib = 0.0;
        for (int g = 0; g < G; ++g)
            t.predicted_mib = std::max(t.predicted_mib, predict_layer_group(net, t.groups[g][0], t.groups[g][1],
                                                                            cfg.grid_n[g], cfg.grid_m[g], 31.0, 2));
    }
    return validate_plan(net, t);
}

std::string validate_plan(const Net& net, const PlanTables& t) {
    const int n_tasks = (int)t.tasks.size();
    const Layer& L0 = net.layers[0];
    const int64_t in_total = (int64_t)t.cfg.batch * L0.c_in * L0.h_in * L0.w_in;
    const int64_t cut_total = (int64_t)t.cfg.batch * t.cut_c8 * 8 * t.cut_h * t.cut_w;
    const int64_t out_total = (int64_t)t.cfg.batch * t.out_h * t.out_w * t.out_c;
    const int64_t scratch_total = t.scratch_elems;
    if (!t.cfg.halo_reuse && scratch_total < (int64_t)t.ring_slots * 2 * t.slot_buf_elems) return "scratch below the ring";
    auto buf_total = [&](int kind) {
        return kind == MAFAT_BUF_USER_IN ? in_total
               : kind == MAFAT_BUF_CUT   ? cut_total
               : kind == MAFAT_BUF_USER_OUT ? out_total
                                          : scratch_total;
    };
    for (const MafatStageDev& s : t.stages) {
        if ((int64_t)s.chunk8 * s.rows_box * s.cols_box * 16 > MAFAT_A_STAGE_BYTES) return "A box exceeds its stage";
        if (s.set_bytes != s.n_chunks * s.n_bsteps * s.blob_elems * 2 || s.set_bytes % 16 != 0)
            return "bad weight set size";
        if (s.bpp < 1 || (int64_t)s.bpp * s.blob_elems * 2 > MAFAT_B_PIECE_BYTES) return "weight piece exceeds its buffer";
        if (s.n_pieces != ceil_div(s.n_chunks * s.n_bsteps, s.bpp)) return "bad weight piece count";
        if (s.cols_box * 8 > 256 || s.rows_box > 256 || s.chunk8 > 256) return "TMA box dimension above 256";
        if ((s.cols_box * 16) % 16 != 0) return "TMA inner box not a multiple of 16 bytes";
        if (s.n_blk % 16 != 0 || s.n_blk < 16 || s.n_blk > MAFAT_MAX_NBLK) return "bad MMA N";
        if (s.mb < 1 || s.mb * s.n_blk > 256) return "blocks of an item exceed one TMEM accumulator buffer";
        if (s.rows_box != (s.flat       ? mafat_flat_rows(s.mb, s.cols_box, s.k)
                           : s.blk_halo ? (MAFAT_BLK_ROWS + s.k - 1) * s.mb
                                        : MAFAT_BLK_ROWS * s.mb + s.k - 1))
            return "A box rows do not cover the item";
        if (s.blk_halo && (s.in_mode != MAFAT_IN_GATHER || s.flat)) return "per-block halos on a stage that is not gathered";
        if (s.flat) {
            if (s.pool || s.chain || s.chained || s.paired || s.cin8 < 2 || s.in_mode != MAFAT_IN_PLANAR)
                return "flat blocks on a pooled, chained, paired-tap or gathered stage";
            if (s.cols_box % 8 != 0 || s.cols_box < 8) return "flat pitch not a multiple of 8 pixels";
        } else if (s.cols_box != MAFAT_BLK_COLS + s.k - 1) {
            return "A box columns do not cover a 16x8 block's taps";
        }
        if (s.w_off + (int64_t)s.n_nblk * s.n_chunks * s.n_bsteps * s.blob_elems > t.weight_elems)
            return "weight blobs outside the packed weights";
        if (s.n_chunks * s.chunk8 != s.cin8) return "chunks do not cover the input channels";
        if (s.mb < 1 || s.mb > (s.paired ? MAFAT_MAX_MB_PAIRED : MAFAT_MAX_MB)) return "blocks per item out of range";
        if (!(s.kst == 1 || s.kst == 2 || s.kst == 4) || (s.paired && s.kst != 1))
            return "K steps per blob must be 1, 2 or 4 (1 when taps are paired)";
        if (s.b_swz && (s.kst != 4 || s.paired || (s.blob_elems * 2) % 1024 != 0))
            return "swizzled blobs need 64 channels and whole 1024-byte atoms";
        if (s.chain) {
            const size_t si = (size_t)(&s - t.stages.data());
            if (si + 1 >= t.stages.size() || !t.stages[si + 1].chained || t.stages[si + 1].k != 1 || s.k != 3 ||
                s.pool)
                return "a chain stage must be a 3x3 convolution followed by its chained 1x1";
            const MafatStageDev& s2 = t.stages[si + 1];
            if (s.n_nblk != 1 || s2.n_nblk != 1 || s.mb != 1 || s2.cin != s.cout || s.n_blk % 64 != 0)
                return "chained stages need every channel of one 128-pixel block in one item";
            if (s.chain_a_col != s.n_blk || s.chain_out_col != s.n_blk + s.n_blk / 2 ||
                s.chain_out_col + s2.n_blk > 256)
                return "chained stages exceed one TMEM accumulator buffer";
            if (s.c2_n_blk != s2.n_blk || s.c2_cout != s2.cout || s.c2_pool != s2.pool || s.c2_n_chunks != s2.n_chunks ||
                s.c2_kst != s2.kst || s.c2_b_swz != s2.b_swz || s.c2_bpp != s2.bpp || s.c2_n_pieces != s2.n_pieces ||
                s.c2_blob_elems != s2.blob_elems || s.c2_sb_off != s2.sb_off || s.c2_w_off != s2.w_off ||
                s2.n_bsteps != 1)
                return "chain stage's copy of its 1x1 differs";
        }
        if (s.chained && (&s == t.stages.data() || !(&s - 1)->chain)) return "a chained stage without its chain stage";
        if (s.pix_pair && s.in_mode != MAFAT_IN_GATHER) return "pixel pairs on a stage that is not gathered";
        if (s.in_mode == MAFAT_IN_GATHER) {
            const Layer& L = net.layers[s.layer];
            if (s.layer != 0 || !s.paired || L.c_in >= 8 || (int64_t)L.w_in * L.c_in % 8 != 0)
                return "raw-row gather on a stage that does not read a narrow NHWC input";
            if (s.raw_e % 8 != 0 || s.raw_e > 256 || s.raw_e < 7 + L.c_in * (s.cols_box + s.pix_pair))
                return "raw row does not hold the halo's elements";
            if (s.pix_pair && (L.c_in > 4 || s.k != 3 || s.n_bsteps != 3 || s.cols_box != MAFAT_BLK_COLS + 2))
                return "pixel pairs on a stage that is not a 3x3 convolution of at most 4 gathered channels";
            if (!s.blk_halo) return "a gathered stage without per-block halos";
            if (mafat_raw_offset(s.rows_box, s.cols_box) + (int64_t)s.mb * mafat_raw_blk_stride(s.k, s.raw_e) >
                MAFAT_A_STAGE_BYTES)
                return "raw rows exceed their A stage";
        }
    }
    std::vector<int> first_item(n_tasks, -1), last_item(n_tasks, -1);
    for (size_t i = 0; i < t.items.size(); ++i) {
        int tk = t.items[i].task;
        if (tk < 0 || tk >= n_tasks) return "item with a bad task";
        if (t.items[i].stage != t.tasks[tk].stage) return "item names another stage than its task";
        if (first_item[tk] < 0) first_item[tk] = (int)i;
        last_item[tk] = (int)i;
    }
    for (int ti = 0; ti < n_tasks; ++ti) {
        const MafatTaskDev& k = t.tasks[ti];
        const MafatStageDev& s = t.stages[k.stage];
        const MafatStageDev& so = s.chain ? t.stages[k.stage + 1] : s;  // the stage whose output it writes
        const Layer& L = net.layers[s.layer];
        if (s.chained) return "a chained stage has a task";
        if (last_item[ti] - first_item[ti] + 1 != k.n_items) return "task items not contiguous";
        if (s.flat ? (k.cw + s.k - 1 > s.cols_box || k.nbx != 1 || k.nby != ceil_div(k.ch * s.cols_box, 128))
                   : (k.nby != ceil_div(k.ch, MAFAT_BLK_ROWS) || k.nbx != ceil_div(k.cw, MAFAT_BLK_COLS)))
            return "task blocks do not tile its conv rectangle";
        // input buffer extent and coverage of every in-map tap of the conv rectangle
        const int64_t in_elems = k.in_kind == MAFAT_BUF_USER_IN ? (int64_t)s.cin * k.in_h * k.in_w
                                                                 : (int64_t)s.cin8 * 8 * k.in_h * k.in_w;
        if (k.in_off < 0 || k.in_off + in_elems > buf_total(k.in_kind)) return "input buffer outside its allocation";
        int ny0 = std::max(k.cy0 - s.pad, 0), ny1 = std::min(k.cy0 + k.ch - 1 - s.pad + s.k, L.h_in);
        int nx0 = std::max(k.cx0 - s.pad, 0), nx1 = std::min(k.cx0 + k.cw - 1 - s.pad + s.k, L.w_in);
        if (k.in_y0 > ny0 || k.in_y0 + k.in_h < ny1 || k.in_x0 > nx0 || k.in_x0 + k.in_w < nx1)
            return "input region does not cover the conv rectangle's taps";
        if (k.in_y0 + k.in_h > L.h_in || k.in_x0 + k.in_w > L.w_in || k.in_y0 < 0 || k.in_x0 < 0)
            return "input region outside the map";
        if (k.in_kind == MAFAT_BUF_SCRATCH && k.in_off % t.slot_buf_elems != 0) return "scratch input misaligned";
        if (k.dep_count < 0 || k.dep_first < 0 || k.dep_first + k.dep_count > (int)t.deps.size()) return "bad dependency list";
        for (int d = k.dep_first; d < k.dep_first + k.dep_count; ++d) {
            const int dt = t.deps[d].ctr - MAFAT_CTR_BASE;
            if (dt < 0 || dt >= n_tasks) return "dependency list names no task";
            if (t.deps[d].target != t.tasks[dt].n_items) return "dependency list target mismatch";
            if (last_item[dt] >= first_item[ti]) return "dependency list names a later task";
        }
        // output extent of the valid pixels
        int oy0 = k.cy0, oy1 = k.cy0 + k.ch, ox0 = k.cx0, ox1 = k.cx0 + k.cw;
        if (so.pool) {
            if (k.cy0 % 2 || k.ch % 2 || k.cx0 % 2 || k.cw % 2) return "pooled rectangle not quad aligned";
            oy0 /= 2; oy1 /= 2; ox0 /= 2; ox1 /= 2;
        }
        if (oy0 < k.out_y0 || ox0 < k.out_x0 || oy1 > k.out_y0 + k.out_h || ox1 > k.out_x0 + k.out_w)
            return "output rectangle outside its buffer";
        int64_t out_elems = k.out_nhwc ? (int64_t)k.out_h * k.out_w * so.cout
                                       : (int64_t)((so.cout + 7) / 8) * 8 * k.out_h * k.out_w;
        if (k.out_off < 0 || k.out_off + out_elems > buf_total(k.out_kind)) return "output buffer outside its allocation";
        if (out_elems >= ((int64_t)1 << 31)) return "an output region exceeds 2^31 elements";
        if (k.out_kind == MAFAT_BUF_SCRATCH && out_elems > t.slot_buf_elems) return "scratch output above buffer size";
        if (k.done_ctr < MAFAT_CTR_BASE || k.done_ctr >= MAFAT_CTR_BASE + t.n_counters) return "bad done counter";
    }
    // dependencies: every counter an item waits on is fed only by items handed out before it
    std::vector<int> frame_last((size_t)t.cfg.batch * std::max(t.cfg.n_groups - 1, 1), -1);
    for (size_t i = 0; i < t.items.size(); ++i) {
        const MafatItemDev& it = t.items[i];
        const MafatTaskDev& k = t.tasks[it.task];
        const MafatStageDev& s = t.stages[k.stage];
        if (s.blk_halo) {
            // a run of the task's blocks in column-major order
            if ((int64_t)k.nby * k.nbx > 32767 || it.bx != 0 || it.by < 0 || it.nb < 0 || it.nb >= s.n_nblk ||
                it.nbk < 1 || it.nbk > s.mb || it.by + it.nbk > k.nby * k.nbx)
                return "per-block-halo item out of range";
        } else {
            if (it.by >= k.nby || it.bx >= k.nbx || it.nb >= s.n_nblk || it.by < 0 || it.bx < 0 || it.nb < 0)
                return "item block out of range";
            if (it.nbk < 1 || it.nbk > s.mb || it.by + it.nbk > k.nby) return "item block count out of range";
        }
        if (s.flat) {
            // every pixel the item's MMAs read (its blocks' 128 pixels at every tap offset) lies
            // inside the A box that starts at the row of its first pixel
            const int64_t p0 = (int64_t)it.by * 128, y_lo = p0 / s.cols_box;
            const int64_t last = p0 - y_lo * s.cols_box + 128 * it.nbk - 1 + (int64_t)(s.k - 1) * (s.cols_box + 1);
            if (last >= (int64_t)s.rows_box * s.cols_box) return "flat item reads past its A box";
            if (it.bx != 0) return "flat item with a block column";
        }
        const int deps[2] = {it.dep0, it.dep1};
        const int tgts[2] = {it.dep0_target, it.dep1_target};
        for (int d = 0; d < 2; ++d) {
            if (deps[d] < 0) continue;
            if (deps[d] < MAFAT_CTR_BASE || deps[d] >= MAFAT_CTR_BASE + t.n_counters) return "bad dependency counter";
            if (deps[d] < t.frame_ctr_base) {
                int dt = deps[d] - MAFAT_CTR_BASE;
                if (last_item[dt] >= (int)i) return "dependency on a later item";
                if (tgts[d] != t.tasks[dt].n_items) return "dependency target mismatch";
            } else {
                int f = deps[d] - t.frame_ctr_base;
                if (frame_last[f] < 0 || frame_last[f] >= (int)i) return "frame dependency on a later item";
            }
        }
        if (it.extra_ctr >= 0) {
            if (it.extra_ctr < t.frame_ctr_base || it.extra_ctr >= MAFAT_CTR_BASE + t.n_counters)
                return "bad extra counter";
            frame_last[it.extra_ctr - t.frame_ctr_base] = (int)i;
        }
    }
    return "";
}

// Packed bf16 weight order, per stage: [n-block][chunk][blob], each blob one B operand of
// kst K=16 steps for n_blk output channels, in one of two shared-memory images:
//  - no swizzle: [K step][K half][N/8][8 rows][8 k]: one K=16 step holds two 8 x 8
//    core-matrix columns (K halves); within a half, the n_blk rows are groups of 8 rows x
//    16 bytes (one core matrix each);
//  - 128-byte swizzle (kst == 4): output channel n owns the 128-byte row (n/8)*1024 +
//    (n%8)*128 of K = 64 channels, whose 16-byte unit u (input octet u of the chunk) sits
//    at unit u ^ (n%8) of the row; the tensor core undoes the XOR from the address bits.
//  - regular stages: blob = tap (ky, kx), K half h of step j = input octet chunk*chunk8 + 2j + h;
//  - paired stages (8 input channels): blob p holds taps (a, b) = (2p, 2p+1), or for an odd
//    tap count the last blob holds (zero weights, last tap); K half 0 = tap a, half 1 = tap b
//    (the kernel points both halves of that last blob at the last tap);
//  - pixel-pair stages (3x3, at most 4 input channels): blob p is kernel row ky = p; K half h
//    holds taps kx = 2h (elements 0-3, its channels) and 2h + 1 (elements 4-7; kx = 3 is a
//    zero tap), matching a halo slot that holds two neighbouring pixels of 4 channels.
void pack_weights_bf16(const Net& net, const PlanTables& t, std::vector<uint16_t>& out) {
    out.assign((size_t)t.weight_elems, 0);
    for (const MafatStageDev& s : t.stages) {
        const Layer& L = net.layers[s.layer];
        const std::vector<float>& w = net.w[s.layer];
        const int k = L.k, cin = L.c_in, taps = k * k;
        for (int nb = 0; nb < s.n_nblk; ++nb)
            for (int c = 0; c < s.n_chunks; ++c)
                for (int b = 0; b < s.n_bsteps; ++b) {
                    size_t blob = (size_t)s.w_off +
                                  ((size_t)(nb * s.n_chunks + c) * s.n_bsteps + b) * (size_t)s.blob_elems;
                    for (int j = 0; j < s.kst; ++j)
                        for (int h = 0; h < 2; ++h)
                            for (int nn = 0; nn < s.n_blk; ++nn)
                                for (int e = 0; e < 8; ++e) {
                                    int o = nb * s.n_blk + nn;
                                    int ci, tap;
                                    if (s.pix_pair) {
                                        const int kx = 2 * h + (e >> 2);
                                        tap = kx < k ? b * k + kx : -1;
                                        ci = e & 3;
                                    } else if (s.paired) {
                                        int a = 2 * b, bb = 2 * b + 1;
                                        if (bb >= taps) {
                                            a = -1;  // zero weights paired with the last tap
                                            bb = taps - 1;
                                        }
                                        tap = h == 0 ? a : bb;
                                        ci = e;
                                    } else {
                                        tap = b;
                                        ci = ((c * s.chunk8) + 2 * j + h) * 8 + e;
                                    }
                                    float v = 0.f;
                                    if (tap >= 0 && ci < cin && o < L.c_out) {
                                        int ky = tap / k, kx = tap % k;
                                        v = w[(((size_t)o * cin + ci) * k + ky) * k + kx];
                                    }
                                    size_t idx;
                                    if (s.b_swz) {
                                        const int u = 2 * j + h;  // 16-byte unit of the 128-byte row
                                        idx = blob + (size_t)(nn / 8) * 512 + (size_t)(nn % 8) * 64 +
                                              (size_t)((u ^ (nn % 8)) * 8) + e;
                                    } else {
                                        idx = blob + (size_t)j * 2 * s.n_blk * 8 + (size_t)h * s.n_blk * 8 +
                                              (size_t)(nn / 8) * 64 + (size_t)(nn % 8) * 8 + e;
                                    }
                                    out[idx] = f32_to_bf16_rne(v);
                                }
                }
    }
}

void pack_weights_fp32(const Net& net, const PlanTables& t, std::vector<float>& w32,
                       std::vector<float>& scale, std::vector<float>& bias) {
    w32.assign((size_t)t.weight32_elems, 0.f);
    scale.assign((size_t)t.sb_elems, 0.f);
    bias.assign((size_t)t.sb_elems, 0.f);
    for (const MafatStageDev& s : t.stages) {
        const std::vector<float>& w = net.w[s.layer];
        std::copy(w.begin(), w.end(), w32.begin() + s.w32_off);
        std::copy(net.scale[s.layer].begin(), net.scale[s.layer].end(), scale.begin() + s.sb_off);
        std::copy(net.bias[s.layer].begin(), net.bias[s.layer].end(), bias.begin() + s.sb_off);
    }
}

}  // namespace mafat

// backward.cu -- row and column kernels of the DiT backward (the training
// pass of the policy update differentiates the loss through v_theta):
//   * gate_backward: through the gated residual x' = x + gate * y, the
//     branch gradient dy = g * gate (bf16 GEMM operand) and per-chunk column
//     sums of g * y (the gate's gradient, per sample) and g * gate (the
//     branch bias's gradient);
//   * ln_modulate_backward: through h = LN(x) (1 + scale) + shift, the
//     residual gradient g += (dn - mean(dn) - n mean(dn n)) / s with
//     dn = dh (1 + scale), and per-chunk column sums of dh and dh n; the
//     affine form h = LN(x) w + b takes dn = dh w (same sums);
//   * qk_norm_rope_backward: through q = rope(RMSNorm(q_raw) w), in place on
//     the q | k gradient columns, with per-CTA partial sums of the scale's
//     gradient;
//   * colsum: column sums of a bf16 or fp32 matrix (bias gradients);
//   * silu_backward: dx = dy SiLU'(pre) (+ a second gradient) for the
//     timestep MLP;
//   * wan_modulation_backward: the WAN model's shared modulation e0 + b_l
//     and final e + b_final, back to d e0, d e and the bias gradients;
//   * reduce_chunks: fixed-order fp64 sums of the partials, so every
//     gradient is deterministic.
#include "internal.h"
#include "ptx.cuh"
#include "reduce_jobs.h"

namespace ff {
namespace {

constexpr float kLnEps = 1e-6f;
constexpr float kRmsEps = 1e-6f;
constexpr int kThreads = 256;

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Sum over the CTA; red holds one slot per warp and is not reused until
// every thread has passed a later __syncthreads.
__device__ __forceinline__ float2 block_sum2(float2 v, float2* red, int lane, int w) {
    v.x = warp_sum(v.x);
    v.y = warp_sum(v.y);
    if (lane == 0) red[w] = v;
    __syncthreads();
    float2 t = make_float2(0.f, 0.f);
#pragma unroll
    for (int i = 0; i < kThreads / 32; ++i) {
        t.x += red[i].x;
        t.y += red[i].y;
    }
    return t;
}

// Chunk c of a segment list -> its segment (copied out with selects, so the
// parameter struct is never indexed dynamically), sample and row range.
__device__ __forceinline__ bool chunk_rows(const BwdSegs& s, int c, BwdSeg& sg, int& b, int& r0, int& r1) {
    const bool second = c >= s.first[1];
    if (second && s.n < 2) return false;
    sg.row0 = second ? s.seg[1].row0 : s.seg[0].row0;
    sg.tokens = second ? s.seg[1].tokens : s.seg[0].tokens;
    sg.col_a = second ? s.seg[1].col_a : s.seg[0].col_a;
    sg.col_b = second ? s.seg[1].col_b : s.seg[0].col_b;
    const int local = c - (second ? s.first[1] : s.first[0]);
    const int cps = bwd_chunks(sg.tokens);
    b = local / cps;
    if (b >= s.B) return false;
    const int k = local - b * cps;
    const int start = sg.row0 + b * sg.tokens;
    r0 = start + k * kBwdChunk;
    r1 = min(r0 + kBwdChunk, start + sg.tokens);
    return true;
}

// ---------------------------------------------------------------- gate

// CTA = (chunk, 1024-column slab); thread t owns columns 4 (slab 256 + t) ..+3.
// Rows go in groups of four whose g and y loads are all issued before the
// group's arithmetic and dy stores (the loop is bound by load latency); the
// sums still add the rows in order.
constexpr int kGateRows = 4;
__global__ void __launch_bounds__(kThreads, 5) gate_backward_kernel(const float* g, const __nv_bfloat16* y, int64_t ld,
                                                                  const float* mods, int64_t ld_mods, BwdSegs s, int H,
                                                                  __nv_bfloat16* dy, float* part) {
    BwdSeg sg;
    int b, r0, r1;
    if (!chunk_rows(s, blockIdx.x, sg, b, r0, r1)) return;
    const int j = 4 * (blockIdx.y * kThreads + threadIdx.x);
    if (j >= H) return;
    const float4 gt = *reinterpret_cast<const float4*>(mods + static_cast<int64_t>(b) * ld_mods + sg.col_a + j);
    float4 sy = make_float4(0.f, 0.f, 0.f, 0.f), sb = sy;
    for (int r = r0; r < r1; r += kGateRows) {
        float4 gv[kGateRows];
        uint2 yu[kGateRows];
#pragma unroll
        for (int k = 0; k < kGateRows; ++k) {
            if (r + k >= r1) break;
            const int64_t o = static_cast<int64_t>(r + k) * ld + j;
            gv[k] = __ldcs(reinterpret_cast<const float4*>(g + o));
            yu[k] = *reinterpret_cast<const uint2*>(y + o);
        }
#pragma unroll
        for (int k = 0; k < kGateRows; ++k) {
            if (r + k >= r1) break;
            const int64_t o = static_cast<int64_t>(r + k) * ld + j;
            const float2 y01 = unpack_bf16x2(yu[k].x), y23 = unpack_bf16x2(yu[k].y);
            sy.x = fmaf(gv[k].x, y01.x, sy.x);
            sy.y = fmaf(gv[k].y, y01.y, sy.y);
            sy.z = fmaf(gv[k].z, y23.x, sy.z);
            sy.w = fmaf(gv[k].w, y23.y, sy.w);
            const float d0 = gv[k].x * gt.x, d1 = gv[k].y * gt.y, d2 = gv[k].z * gt.z, d3 = gv[k].w * gt.w;
            sb.x += d0;
            sb.y += d1;
            sb.z += d2;
            sb.w += d3;
            *reinterpret_cast<uint2*>(dy + o) = make_uint2(pack_bf16x2(d0, d1), pack_bf16x2(d2, d3));
        }
    }
    float* p = part + static_cast<int64_t>(blockIdx.x) * 2 * H + j;
    *reinterpret_cast<float4*>(p) = sy;
    *reinterpret_cast<float4*>(p + H) = sb;
}

// ---------------------------------------------------------------- LN-modulate

// Sum of three values over the CTA (same slot discipline as block_sum2).
__device__ __forceinline__ float3 block_sum3(float3 v, float3* red, int lane, int w) {
    v.x = warp_sum(v.x);
    v.y = warp_sum(v.y);
    v.z = warp_sum(v.z);
    if (lane == 0) red[w] = v;
    __syncthreads();
    float3 t = make_float3(0.f, 0.f, 0.f);
#pragma unroll
    for (int i = 0; i < kThreads / 32; ++i) {
        t.x += red[i].x;
        t.y += red[i].y;
        t.z += red[i].z;
    }
    return t;
}

// CTA = one chunk of rows, all H columns: thread t holds float4s t, t + 256,
// ... of a row (PER of them).  Per row, with d = dh (1 + scale) (or dh w):
// one reduction of (sum x, sum d, sum d x), one of the centred variance (as
// in the forward); mean(d n) = (sum d x - mean sum d) rstd / H.  The next
// row's x, dh and g are loaded before this row's reductions.
template <int PER>
__global__ void __launch_bounds__(kThreads, (PER <= 3 ? 2 : 1)) ln_modulate_backward_kernel(const float* x, const float* dh, float* gx,
                                                                         int64_t ld, const float* mods,
                                                                         int64_t ld_mods, BwdSegs s, int H,
                                                                         const __nv_bfloat16* aff_w, float* part) {
    __shared__ float3 red3[2][kThreads / 32];
    __shared__ float2 red2[2][kThreads / 32];
    BwdSeg sg;
    int b, r0, r1;
    if (!chunk_rows(s, blockIdx.x, sg, b, r0, r1)) return;
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    const int nv = H >> 2;
    // the multiplier of n: 1 + scale of this sample, or the affine weight
    float4 sc1[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        const int k = t + kThreads * i;
        if (aff_w) {
            const uint2 u = k < nv ? *reinterpret_cast<const uint2*>(aff_w + 4 * k) : make_uint2(0u, 0u);
            const float2 lo = unpack_bf16x2(u.x), hi = unpack_bf16x2(u.y);
            sc1[i] = make_float4(lo.x, lo.y, hi.x, hi.y);
        } else {
            const float4* scale = reinterpret_cast<const float4*>(mods + static_cast<int64_t>(b) * ld_mods + sg.col_b);
            const float4 c = k < nv ? scale[k] : make_float4(0.f, 0.f, 0.f, 0.f);
            sc1[i] = make_float4(1.f + c.x, 1.f + c.y, 1.f + c.z, 1.f + c.w);
        }
    }
    float4 acc_sh[PER], acc_sc[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) acc_sh[i] = acc_sc[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
    float4 xr[PER], dr[PER], gr[PER];
    {
        const float4* xp = reinterpret_cast<const float4*>(x + static_cast<int64_t>(r0) * ld);
        const float4* dp = reinterpret_cast<const float4*>(dh + static_cast<int64_t>(r0) * ld);
        const float4* gp = reinterpret_cast<const float4*>(gx + static_cast<int64_t>(r0) * ld);
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const int k = t + kThreads * i;
            xr[i] = k < nv ? __ldcs(xp + k) : z;
            dr[i] = k < nv ? __ldcs(dp + k) : z;
            gr[i] = k < nv ? gp[k] : z;
        }
    }
    const float invH = 1.f / H;
    int par = 0;
    for (int r = r0; r < r1; ++r, par ^= 1) {
        float4 xn[PER], dn[PER], gn[PER];
        {
            const bool more = r + 1 < r1;
            const float4* xp = reinterpret_cast<const float4*>(x + static_cast<int64_t>(r + 1) * ld);
            const float4* dp = reinterpret_cast<const float4*>(dh + static_cast<int64_t>(r + 1) * ld);
            const float4* gp = reinterpret_cast<const float4*>(gx + static_cast<int64_t>(r + 1) * ld);
#pragma unroll
            for (int i = 0; i < PER; ++i) {
                const int k = t + kThreads * i;
                xn[i] = more && k < nv ? __ldcs(xp + k) : z;
                dn[i] = more && k < nv ? __ldcs(dp + k) : z;
                gn[i] = more && k < nv ? gp[k] : z;
            }
        }
        // d = dh (1 + scale); sums of x, d and d x
        float sx = 0.f, sd = 0.f, sdx = 0.f;
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const float4 d = make_float4(dr[i].x * sc1[i].x, dr[i].y * sc1[i].y, dr[i].z * sc1[i].z,
                                         dr[i].w * sc1[i].w);
            sx += (xr[i].x + xr[i].y) + (xr[i].z + xr[i].w);
            sd += (d.x + d.y) + (d.z + d.w);
            sdx += (d.x * xr[i].x + d.y * xr[i].y) + (d.z * xr[i].z + d.w * xr[i].w);
        }
        const float3 s3 = block_sum3(make_float3(sx, sd, sdx), red3[par], lane, w);
        const float mean = s3.x * invH;
        float q = 0.f;
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            if (t + kThreads * i < nv) {
                const float d0 = xr[i].x - mean, d1 = xr[i].y - mean, d2 = xr[i].z - mean, d3 = xr[i].w - mean;
                q += (d0 * d0 + d1 * d1) + (d2 * d2 + d3 * d3);
            }
        }
        const float rstd = rsqrtf(block_sum2(make_float2(q, 0.f), red2[par], lane, w).x * invH + kLnEps);
        const float m1 = s3.y * invH, m2 = (s3.z - mean * s3.y) * rstd * invH;
        float4* gp = reinterpret_cast<float4*>(gx + static_cast<int64_t>(r) * ld);
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const int k = t + kThreads * i;
            if (k >= nv) continue;
            const float4 n = make_float4((xr[i].x - mean) * rstd, (xr[i].y - mean) * rstd, (xr[i].z - mean) * rstd,
                                         (xr[i].w - mean) * rstd);
            acc_sh[i].x += dr[i].x; acc_sh[i].y += dr[i].y; acc_sh[i].z += dr[i].z; acc_sh[i].w += dr[i].w;
            acc_sc[i].x = fmaf(dr[i].x, n.x, acc_sc[i].x);
            acc_sc[i].y = fmaf(dr[i].y, n.y, acc_sc[i].y);
            acc_sc[i].z = fmaf(dr[i].z, n.z, acc_sc[i].z);
            acc_sc[i].w = fmaf(dr[i].w, n.w, acc_sc[i].w);
            float4 o = gr[i];
            o.x += rstd * (dr[i].x * sc1[i].x - m1 - n.x * m2);
            o.y += rstd * (dr[i].y * sc1[i].y - m1 - n.y * m2);
            o.z += rstd * (dr[i].z * sc1[i].z - m1 - n.z * m2);
            o.w += rstd * (dr[i].w * sc1[i].w - m1 - n.w * m2);
            gp[k] = o;
        }
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            xr[i] = xn[i];
            dr[i] = dn[i];
            gr[i] = gn[i];
        }
    }
    float4* p = reinterpret_cast<float4*>(part + static_cast<int64_t>(blockIdx.x) * 2 * H);
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        const int k = t + kThreads * i;
        if (k >= nv) continue;
        p[k] = acc_sh[i];
        p[nv + k] = acc_sc[i];
    }
}

// ---------------------------------------------------------------- QK norm + RoPE

// A warp takes whole rows (rows r_begin + w, r_begin + w + 8, ...) and, per
// row, every head in order; lane owns E = d / 32 consecutive elements of a
// head (whole rotation pairs).  The rotation of a lane's pairs depends on
// the row only, so it is looked up once per row and serves every head of q
// and k.  The q and k gradient and raw loads of the next head are issued
// before the current head's arithmetic (the loop is bound by load latency).  A CTA covers kQkRows rows of one segment; its warps add
// their lanes' scale-gradient terms, summed over the CTA at the end into
// part[cta][q: 0..d | k: d..2d].
constexpr int kQkRows = kQkBwdRows;
constexpr int kQkWarps = kThreads / 32;

template <int E>
__global__ void __launch_bounds__(kThreads) qk_norm_rope_backward_kernel(QkBwdArgs a, int ctas_txt) {
    __shared__ float red[kQkWarps][2][128];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const bool img = static_cast<int>(blockIdx.x) >= ctas_txt;
    const int r_begin = img ? a.rows_txt + (blockIdx.x - ctas_txt) * kQkRows : blockIdx.x * kQkRows;
    const int r_end = min(r_begin + kQkRows, img ? a.rows : a.rows_txt);
    const int c0 = lane * E;
    const int d = a.head_dim;
    const __nv_bfloat16* qs = img ? a.q_scale_img : a.q_scale_txt;
    const __nv_bfloat16* ks = img ? a.k_scale_img : a.k_scale_txt;
    float wq[E], wk[E], gq[E], gk[E];
#pragma unroll
    for (int i = 0; i < E; ++i) {
        wq[i] = __bfloat162float(qs[c0 + i]);
        wk[i] = __bfloat162float(ks[c0 + i]);
        gq[i] = gk[i] = 0.f;
    }
    const int h0 = a.axes0 >> 1, h1 = a.axes1 >> 1;
    for (int row = r_begin + w; row < r_end; row += kQkWarps) {
        // rotation of this lane's pairs (identity for text tokens)
        float cs[E / 2], sn[E / 2];
        if (img && a.rope_cs) {
            const int n = (row - a.rows_txt) % a.n_img;
            const int hw = a.grid_h * a.grid_w;
            const int base0 = (n / hw) * h0;
            const int base1 = a.grid_f * h0 + ((n / a.grid_w) % a.grid_h) * h1 - h0;
            const int base2 = a.grid_f * h0 + a.grid_h * h1 + (n % a.grid_w) * (a.axes2 >> 1) - h0 - h1;
#pragma unroll
            for (int p = 0; p < E / 2; ++p) {
                const int pair = c0 / 2 + p;
                const float2 t = a.rope_cs[pair < h0 ? base0 + pair : (pair < h0 + h1 ? base1 + pair : base2 + pair)];
                cs[p] = t.x;
                sn[p] = t.y;
            }
        } else {
#pragma unroll
            for (int p = 0; p < E / 2; ++p) { cs[p] = 1.f; sn[p] = 0.f; }
        }
        __nv_bfloat16* grow = a.d + static_cast<int64_t>(row) * a.ldd + c0;
        const __nv_bfloat16* xrow = a.raw + static_cast<int64_t>(row) * a.ldr + c0;
        // packed bf16 pairs of head h (cur) and of head h + 1 (nxt, loaded
        // before head h's arithmetic and stores)
        uint32_t cur_g[2][E / 2], cur_x[2][E / 2], nxt_g[2][E / 2], nxt_x[2][E / 2];
        auto load_head = [&](int head, uint32_t (&g)[2][E / 2], uint32_t (&x)[2][E / 2]) {
#pragma unroll
            for (int which = 0; which < 2; ++which) {
                if (which >= a.sets) break;
                const int col = (which * a.heads + head) * d;
#pragma unroll
                for (int i = 0; i < E / 2; ++i) {
                    g[which][i] = *reinterpret_cast<const uint32_t*>(grow + col + 2 * i);
                    x[which][i] = *reinterpret_cast<const uint32_t*>(xrow + col + 2 * i);
                }
            }
        };
        load_head(0, cur_g, cur_x);
        for (int head = 0; head < a.heads; ++head) {
            if (head + 1 < a.heads) load_head(head + 1, nxt_g, nxt_x);
            float gv[2][E], xv[2][E];
#pragma unroll
            for (int which = 0; which < 2; ++which) {
#pragma unroll
                for (int i = 0; i < E / 2; ++i) {
                    const float2 g2 = unpack_bf16x2(cur_g[which][i]);
                    const float2 x2 = unpack_bf16x2(cur_x[which][i]);
                    gv[which][2 * i] = g2.x; gv[which][2 * i + 1] = g2.y;
                    xv[which][2 * i] = x2.x; xv[which][2 * i + 1] = x2.y;
                }
            }
#pragma unroll
            for (int which = 0; which < 2; ++which) {
                if (which >= a.sets) break;
                // transposed rotation: gradient w.r.t. the normalised, scaled values
                float gy[E];
#pragma unroll
                for (int p = 0; p < E / 2; ++p) {
                    gy[2 * p] = gv[which][2 * p] * cs[p] + gv[which][2 * p + 1] * sn[p];
                    gy[2 * p + 1] = -gv[which][2 * p] * sn[p] + gv[which][2 * p + 1] * cs[p];
                }
                float ss = 0.f;
#pragma unroll
                for (int i = 0; i < E; ++i) ss = fmaf(xv[which][i], xv[which][i], ss);
                const float r = rsqrtf(warp_sum(ss) / d + kRmsEps);
                const float* wv = which ? wk : wq;
                float* acc = which ? gk : gq;
                float dot = 0.f;
                float xn[E], gg[E];
#pragma unroll
                for (int i = 0; i < E; ++i) {
                    xn[i] = xv[which][i] * r;
                    gg[i] = gy[i] * wv[i];
                    acc[i] = fmaf(gy[i], xn[i], acc[i]);
                    dot = fmaf(gg[i], xn[i], dot);
                }
                const float m = warp_sum(dot) / d;
                __nv_bfloat16* gp = grow + (which * a.heads + head) * d;
#pragma unroll
                for (int i = 0; i < E; i += 2)
                    *reinterpret_cast<uint32_t*>(gp + i) =
                        pack_bf16x2(r * (gg[i] - xn[i] * m), r * (gg[i + 1] - xn[i + 1] * m));
            }
#pragma unroll
            for (int which = 0; which < 2; ++which)
#pragma unroll
                for (int i = 0; i < E / 2; ++i) {
                    cur_g[which][i] = nxt_g[which][i];
                    cur_x[which][i] = nxt_x[which][i];
                }
        }
    }
#pragma unroll
    for (int i = 0; i < E; ++i) {
        red[w][0][c0 + i] = gq[i];
        red[w][1][c0 + i] = gk[i];
    }
    __syncthreads();
    for (int k = threadIdx.x; k < 2 * d; k += kThreads) {
        const int which = k / d, j = k - which * d;
        float s = 0.f;
#pragma unroll
        for (int ww = 0; ww < kQkWarps; ++ww) s += red[ww][which][j];
        a.part[static_cast<int64_t>(blockIdx.x) * 2 * d + k] = s;
    }
}

// ---------------------------------------------------------------- column sums

// CTA = (chunk of kBwdChunk rows, 1024-column slab).
template <typename T>
__global__ void __launch_bounds__(kThreads) colsum_partial_kernel(const T* in, int64_t ld, int rows, int ncols,
                                                                   float* part) {
    const int j = 4 * (blockIdx.y * kThreads + threadIdx.x);
    if (j >= ncols) return;
    const int r0 = blockIdx.x * kBwdChunk, r1 = min(r0 + kBwdChunk, rows);
    float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int r = r0; r < r1; ++r) {
        float4 v;
        if constexpr (sizeof(T) == 4) {
            v = *reinterpret_cast<const float4*>(in + static_cast<int64_t>(r) * ld + j);
        } else {
            const uint2 u = *reinterpret_cast<const uint2*>(in + static_cast<int64_t>(r) * ld + j);
            const float2 a = unpack_bf16x2(u.x), b = unpack_bf16x2(u.y);
            v = make_float4(a.x, a.y, b.x, b.y);
        }
        s.x += v.x; s.y += v.y; s.z += v.z; s.w += v.w;
    }
    *reinterpret_cast<float4*>(part + static_cast<int64_t>(blockIdx.x) * ncols + j) = s;
}

// ---------------------------------------------------------------- chunk reduction

// A batch of fixed-order sums: column block x of the grid belongs to job k
// (blk0[k] <= x < blk0[k + 1]), blockIdx.y is the sample of a per-sample job.
// out[b * ld_out + j] = sum over sample b's chunks of every span
// (per_sample), or out[j] = sum over all chunks of every span.  A CTA takes 32
// columns (lane = column, so a chunk row is one 128-byte load per warp); warp
// w takes the chunks w, w + 8, ... in four interleaved fp64 chains, and the
// eight warp sums are added in warp order: a fixed order for a given shape,
// the same whichever jobs share the launch.
struct ReduceBatch {
    ReduceJob job[kMaxReduceJobs];
    int blk0[kMaxReduceJobs + 1];
    int n;
};

__global__ void __launch_bounds__(256) reduce_chunks_kernel(ReduceBatch rb) {
    __shared__ double red[8][32];
    // the job of this column block, picked by selects (no dynamic indexing
    // of the parameter struct)
    const int x = blockIdx.x;
    ReduceJob jb = rb.job[0];
    int blk0 = 0;
#pragma unroll
    for (int k = 1; k < kMaxReduceJobs; ++k)
        if (k < rb.n && x >= rb.blk0[k]) {
            jb = rb.job[k];
            blk0 = rb.blk0[k];
        }
    const int b = blockIdx.y;
    if (!jb.per_sample && b > 0) return;   // uniform over the CTA
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int j = (x - blk0) * 32 + lane;
    double acc[4] = {0.0, 0.0, 0.0, 0.0};
    if (j < jb.ncols) {
        for (int i = 0; i < jb.sp.n; ++i) {
            const int cnt = i ? jb.sp.count[1] : jb.sp.count[0];
            const int first = (i ? jb.sp.first[1] : jb.sp.first[0]) + (jb.per_sample ? b * cnt : 0);
            const float* base = jb.part + static_cast<int64_t>(first) * jb.ld_part + j;
            const int64_t ld = jb.ld_part;
            int c = w;
            for (; c + 24 < cnt; c += 32) {
                acc[0] += base[static_cast<int64_t>(c) * ld];
                acc[1] += base[static_cast<int64_t>(c + 8) * ld];
                acc[2] += base[static_cast<int64_t>(c + 16) * ld];
                acc[3] += base[static_cast<int64_t>(c + 24) * ld];
            }
            for (; c < cnt; c += 8) acc[0] += base[static_cast<int64_t>(c) * ld];
        }
    }
    red[w][lane] = (acc[0] + acc[1]) + (acc[2] + acc[3]);
    __syncthreads();
    if (w == 0 && j < jb.ncols) {
        double s = 0.0;
#pragma unroll
        for (int k = 0; k < 8; ++k) s += red[k][lane];
        jb.out[static_cast<int64_t>(b) * jb.ld_out + j] = static_cast<float>(s);
    }
}

// ---------------------------------------------------------------- SiLU

// dx = dy SiLU'(pre) for rows < B, written fp32 [B, n] and bf16 [rows_pad, n]
// (rows B.. rows_pad - 1 zero: the padded operand of the weight gradient).
__global__ void silu_backward_kernel(const float* dy, int64_t ld_dy, const __nv_bfloat16* pre, int B, int rows_pad,
                                     int n, const float* add, float* dx, __nv_bfloat16* dxb) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= rows_pad * n) return;
    const int b = i / n, j = i - b * n;
    float v = 0.f;
    if (b < B) {
        const float p = __bfloat162float(pre[i]);
        const float s = 1.f / (1.f + __expf(-p));
        v = dy[static_cast<int64_t>(b) * ld_dy + j] * s * (1.f + p * (1.f - s));
        if (add) v += add[i];
        dx[i] = v;
    }
    dxb[i] = __float2bfloat16_rn(v);
}

// Items, flat: [0, nb) the bias gradients (column j of dm summed over the
// batch in order; block l's 6H at gbias0 + l stride, the final 2H at
// gfinal); then rows_pad x 6H of d e0 = sum over blocks in order (bf16 copy
// zero past B); then B x H of the final layer's d e = d shift + d scale.
__global__ void wan_modulation_backward_kernel(const float* dm, int64_t ld, int B, int rows_pad, int H, int L,
                                               float* gbias0, int64_t stride, float* gfinal, float* de0,
                                               __nv_bfloat16* de0b, float* de_fin) {
    const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    const int64_t H6 = 6 * static_cast<int64_t>(H), nb = L * H6 + 2 * H, ne0 = rows_pad * H6;
    if (i < nb) {
        float acc = 0.f;
        for (int b = 0; b < B; ++b) acc += dm[b * ld + i];
        const int64_t l = i / H6;
        if (l < L) gbias0[l * stride + (i - l * H6)] = acc;
        else gfinal[i - L * H6] = acc;
    } else if (i < nb + ne0) {
        const int64_t k = i - nb;
        const int64_t b = k / H6, j = k - b * H6;
        float acc = 0.f;
        if (b < B) {
            for (int l = 0; l < L; ++l) acc += dm[b * ld + l * H6 + j];
            de0[k] = acc;
        }
        de0b[k] = __float2bfloat16_rn(acc);
    } else if (i < nb + ne0 + static_cast<int64_t>(B) * H) {
        const int64_t k = i - nb - ne0;
        const int64_t b = k / H, j = k - b * H;
        de_fin[k] = dm[b * ld + L * H6 + j] + dm[b * ld + L * H6 + H + j];
    }
}

int reduce(const float* part, int64_t ld_part, int ncols, const ChunkSpans& sp, int B, float* out, int64_t ld_out,
           cudaStream_t stream) {
    const ReduceJob j{part, ld_part, ncols, sp, B > 0 ? 1 : 0, out, ld_out};
    return reduce_chunks_batch(&j, 1, B, stream);
}

}  // namespace

BwdSegs bwd_segs(const BwdSeg* segs, int n, int B) {
    BwdSegs s{};
    s.n = n;
    s.B = B;
    int c = 0;
    for (int i = 0; i < 2; ++i) {
        s.first[i] = c;
        if (i < n) {
            s.seg[i] = segs[i];
            c += B * bwd_chunks(segs[i].tokens);
        }
    }
    s.chunks = c;
    s.rows = 0;
    for (int i = 0; i < n; ++i) s.rows += static_cast<int64_t>(B) * segs[i].tokens;
    return s;
}

int gate_backward(const float* g, const __nv_bfloat16* y, int64_t ld, const float* mods, int64_t ld_mods,
                  const BwdSegs& s, int H, __nv_bfloat16* dy, float* part, cudaStream_t stream) {
    if (H % 4 || ld % 4) return set_error(FF_ERR_UNSUPPORTED, "gate_backward: H and ld must be multiples of 4");
    if (s.chunks == 0) return FF_OK;
    ProfScope prof(stream, "gate_backward", 0.0, 8.0 * s.rows * H);
    dim3 grid(s.chunks, (H / 4 + kThreads - 1) / kThreads);
    gate_backward_kernel<<<grid, kThreads, 0, stream>>>(g, y, ld, mods, ld_mods, s, H, dy, part);
    return check_launch("gate_backward_kernel");
}

int ln_modulate_backward(const float* x, const float* dh, float* gx, int64_t ld, const float* mods, int64_t ld_mods,
                         const BwdSegs& s, int H, float* part, cudaStream_t stream, const __nv_bfloat16* aff_w) {
    if (H % 4 || ld % 4) return set_error(FF_ERR_UNSUPPORTED, "ln_modulate_backward: H and ld must be multiples of 4");
    const int per = (H / 4 + kThreads - 1) / kThreads;
    if (per > 8) return set_error(FF_ERR_UNSUPPORTED, "ln_modulate_backward: H=%d > 8192", H);
    if (s.chunks == 0) return FF_OK;
    ProfScope prof(stream, "ln_modulate_backward", 0.0, 16.0 * s.rows * H);
#define FF_LNB(P)                                                                                                   \
    case P:                                                                                                          \
        ln_modulate_backward_kernel<P><<<s.chunks, kThreads, 0, stream>>>(x, dh, gx, ld, mods, ld_mods, s, H, aff_w, \
                                                                           part);                                     \
        break;
    switch (per) {
        FF_LNB(1) FF_LNB(2) FF_LNB(3) FF_LNB(4) FF_LNB(5) FF_LNB(6) FF_LNB(7) FF_LNB(8)
    }
#undef FF_LNB
    return check_launch("ln_modulate_backward_kernel");
}

int qk_norm_rope_backward(const QkBwdArgs& a, int* ctas_txt, int* ctas_img, cudaStream_t stream) {
    if ((a.head_dim != 64 && a.head_dim != 128) || a.rows_txt < 0 || a.rows < a.rows_txt)
        return set_error(FF_ERR_UNSUPPORTED, "qk_norm_rope_backward: head_dim %d", a.head_dim);
    const int ct = (a.rows_txt + kQkRows - 1) / kQkRows;
    const int ci = (a.rows - a.rows_txt + kQkRows - 1) / kQkRows;
    *ctas_txt = ct;
    *ctas_img = ci;
    if (ct + ci == 0) return FF_OK;
    ProfScope prof(stream, "qk_norm_rope_backward", 0.0, 12.0 * a.rows * a.heads * a.head_dim);
    if (a.head_dim == 128) qk_norm_rope_backward_kernel<4><<<ct + ci, kThreads, 0, stream>>>(a, ct);
    else qk_norm_rope_backward_kernel<2><<<ct + ci, kThreads, 0, stream>>>(a, ct);
    return check_launch("qk_norm_rope_backward_kernel");
}

size_t colsum_ws_floats(int rows, int ncols) { return static_cast<size_t>((rows + kBwdChunk - 1) / kBwdChunk) * ncols; }

int colsum(const void* in, bool f32, int64_t ld, int rows, int ncols, float* out, float* ws, cudaStream_t stream) {
    if (ncols % 4 || ld % 4) return set_error(FF_ERR_UNSUPPORTED, "colsum: ncols and ld must be multiples of 4");
    if (rows <= 0) return set_error(FF_ERR_INVALID_ARG, "colsum: rows=%d", rows);
    const int chunks = (rows + kBwdChunk - 1) / kBwdChunk;
    {
        ProfScope prof(stream, "colsum", 0.0, static_cast<double>(rows) * ncols * (f32 ? 4 : 2));
        dim3 grid(chunks, (ncols / 4 + kThreads - 1) / kThreads);
        if (f32) colsum_partial_kernel<float><<<grid, kThreads, 0, stream>>>(static_cast<const float*>(in), ld, rows, ncols, ws);
        else colsum_partial_kernel<__nv_bfloat16><<<grid, kThreads, 0, stream>>>(static_cast<const __nv_bfloat16*>(in), ld, rows, ncols, ws);
        FF_TRY(check_launch("colsum_partial_kernel"));
    }
    ChunkSpans sp{};
    sp.n = 1;
    sp.first[0] = 0;
    sp.count[0] = chunks;
    return reduce(ws, ncols, ncols, sp, 0, out, 0, stream);
}

int reduce_chunks(const float* part, int64_t ld_part, int ncols, const ChunkSpans& sp, int B, float* out,
                  int64_t ld_out, cudaStream_t stream) {
    return reduce(part, ld_part, ncols, sp, B, out, ld_out, stream);
}

int reduce_chunks_batch(const ReduceJob* jobs, int n, int B, cudaStream_t stream) {
    for (int i = 0; i < n; ++i) {   // every job checked before the first launch
        const ReduceJob& j = jobs[i];
        if (j.ncols <= 0 || j.sp.n < 1 || j.sp.n > 2 || (j.per_sample && B <= 0))
            return set_error(FF_ERR_INVALID_ARG, "reduce_chunks: job %d: ncols=%d spans=%d B=%d", i, j.ncols, j.sp.n, B);
    }
    for (int at = 0; at < n; at += kMaxReduceJobs) {
        ReduceBatch rb{};
        rb.n = n - at < kMaxReduceJobs ? n - at : kMaxReduceJobs;
        bool any_per_sample = false;
        double bytes = 0.0;
        int blocks = 0;
        for (int k = 0; k < rb.n; ++k) {
            const ReduceJob& j = jobs[at + k];
            rb.job[k] = j;
            rb.blk0[k] = blocks;
            blocks += (j.ncols + 31) / 32;
            any_per_sample = any_per_sample || j.per_sample;
            double chunks = 0.0;
            for (int i = 0; i < j.sp.n; ++i) chunks += static_cast<double>(j.sp.count[i]) * (j.per_sample ? B : 1);
            bytes += chunks * j.ncols * 4.0;
        }
        rb.blk0[rb.n] = blocks;
        ProfScope prof(stream, "reduce_chunks", 0.0, bytes);
        reduce_chunks_kernel<<<dim3(blocks, any_per_sample ? B : 1), 256, 0, stream>>>(rb);
        FF_TRY(check_launch("reduce_chunks_kernel"));
    }
    return FF_OK;
}

int silu_backward(const float* dy, int64_t ld_dy, const __nv_bfloat16* pre, int B, int rows_pad, int n, float* dx,
                  __nv_bfloat16* dxb, cudaStream_t stream, const float* add) {
    const int total = rows_pad * n;
    silu_backward_kernel<<<(total + 255) / 256, 256, 0, stream>>>(dy, ld_dy, pre, B, rows_pad, n, add, dx, dxb);
    return check_launch("silu_backward_kernel");
}

namespace {

// dW[m, n] = sum_{b < B} dy[b, m] x[b, n], b in order: the weight gradient of
// a Linear applied to B rows (the adaLN modulation, the time MLP).  A thread
// writes four consecutive columns of kRowsW rows; x's slice stays in L1.
constexpr int kRowsW = 8;
__global__ void __launch_bounds__(256) rows_wgrad_kernel(int B, int M, int N, const float* __restrict__ dy,
                                                         int64_t ldy, const __nv_bfloat16* __restrict__ x,
                                                         int64_t ldx, float* __restrict__ dw, int64_t ldw) {
    const int n = (blockIdx.y * 256 + threadIdx.x) * 4;
    if (n >= N) return;
    const int m0 = blockIdx.x * kRowsW;   // row groups on x: M reaches millions of rows
    for (int m = m0; m < m0 + kRowsW && m < M; ++m) {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int b = 0; b < B; ++b) {
            const float g = dy[static_cast<int64_t>(b) * ldy + m];
            const uint2 u = *reinterpret_cast<const uint2*>(x + static_cast<int64_t>(b) * ldx + n);
            const float2 x01 = unpack_bf16x2(u.x), x23 = unpack_bf16x2(u.y);
            acc.x = fmaf(g, x01.x, acc.x);
            acc.y = fmaf(g, x01.y, acc.y);
            acc.z = fmaf(g, x23.x, acc.z);
            acc.w = fmaf(g, x23.y, acc.w);
        }
        *reinterpret_cast<float4*>(dw + static_cast<int64_t>(m) * ldw + n) = acc;
    }
}

// dx[b, n] = sum_{m < M} dy[b, m] w[m, n]: the input gradient of a Linear
// applied to B <= kRowsDgrad rows.  Stage 1: a block takes a chunk of rows of
// w (a multiple of 8 rows) for 512 columns; a thread issues the loads of 8
// rows (a warp reads 256 contiguous bytes of each) before their arithmetic,
// and writes the chunk's partial sums; stage 2 sums the chunks in order.
constexpr int kRowsDgrad = 16;
// BMAX: accumulators for up to BMAX batch rows (4, 8 or 16), so a small batch
// keeps the registers low and more rows' loads in flight per SM
template <int BMAX>
__global__ void __launch_bounds__(128) rows_dgrad_partial_kernel(int B, int M, int N, int rows_per_chunk,
                                                                 const float* __restrict__ dy, int64_t ldy,
                                                                 const __nv_bfloat16* __restrict__ w, int64_t ldw,
                                                                 float* __restrict__ part) {
    const int n = (blockIdx.x * 128 + threadIdx.x) * 4;
    const int c = blockIdx.y;
    const int m0 = c * rows_per_chunk;
    const int m1 = min(M, m0 + rows_per_chunk);
    if (n >= N) return;
    float4 acc[BMAX];
#pragma unroll
    for (int b = 0; b < BMAX; ++b) acc[b] = make_float4(0.f, 0.f, 0.f, 0.f);
    // rows m0 .. m1 in groups of 8 (m1 - m0 a multiple of 8): group g + 1's
    // loads are in flight while group g is used
    auto load8 = [&](int m, uint2 (&u)[8]) {
#pragma unroll
        for (int r = 0; r < 8; ++r) u[r] = *reinterpret_cast<const uint2*>(w + static_cast<int64_t>(m + r) * ldw + n);
    };
    uint2 cur[8], nxt[8];
    if (m0 < m1) load8(m0, cur);
    for (int m = m0; m < m1; m += 8) {
        if (m + 8 < m1) load8(m + 8, nxt);
        float2 wv[8][2];
#pragma unroll
        for (int r = 0; r < 8; ++r) {
            wv[r][0] = unpack_bf16x2(cur[r].x);
            wv[r][1] = unpack_bf16x2(cur[r].y);
        }
#pragma unroll
        for (int b = 0; b < BMAX; ++b) {
            if (b < B) {
                // dy[b, m .. m + 7] (m and ldy multiples of 4)
                const float* g = dy + static_cast<int64_t>(b) * ldy + m;
                const float4 g0 = *reinterpret_cast<const float4*>(g);
                const float4 g1 = *reinterpret_cast<const float4*>(g + 4);
                const float gv[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
#pragma unroll
                for (int r = 0; r < 8; ++r) {
                    acc[b].x = fmaf(gv[r], wv[r][0].x, acc[b].x);
                    acc[b].y = fmaf(gv[r], wv[r][0].y, acc[b].y);
                    acc[b].z = fmaf(gv[r], wv[r][1].x, acc[b].z);
                    acc[b].w = fmaf(gv[r], wv[r][1].y, acc[b].w);
                }
            }
        }
#pragma unroll
        for (int r = 0; r < 8; ++r) cur[r] = nxt[r];
    }
#pragma unroll
    for (int b = 0; b < BMAX; ++b)
        if (b < B) *reinterpret_cast<float4*>(part + (static_cast<int64_t>(c) * B + b) * N + n) = acc[b];
}

__global__ void __launch_bounds__(256) rows_dgrad_sum_kernel(int B, int N, int chunks, const float* __restrict__ part,
                                                             float* __restrict__ dx, int64_t ldx) {
    const int n = (blockIdx.x * 256 + threadIdx.x) * 4;
    const int b = blockIdx.y;
    if (n >= N) return;
    float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int c = 0; c < chunks; ++c) {
        const float4 v = *reinterpret_cast<const float4*>(part + (static_cast<int64_t>(c) * B + b) * N + n);
        s.x += v.x;
        s.y += v.y;
        s.z += v.z;
        s.w += v.w;
    }
    *reinterpret_cast<float4*>(dx + static_cast<int64_t>(b) * ldx + n) = s;
}

}  // namespace

int rows_wgrad(int B, int M, int N, const float* dy, int64_t ldy, const __nv_bfloat16* x, int64_t ldx, float* dw,
               int64_t ldw, cudaStream_t stream) {
    if (B <= 0 || M <= 0 || N <= 0 || N % 4 || ldx % 4 || ldw % 4 || ldy < M || ldx < N || ldw < N)
        return set_error(FF_ERR_INVALID_ARG, "rows_wgrad: B=%d M=%d N=%d", B, M, N);
    ProfScope prof(stream, "rows_wgrad", 2.0 * B * M * N, 4.0 * M * N + 2.0 * B * N + 4.0 * B * M);
    if (N / 4 > 255 * 65535) return set_error(FF_ERR_INVALID_ARG, "rows_wgrad: N=%d", N);
    const dim3 grid((M + kRowsW - 1) / kRowsW, (N / 4 + 255) / 256);
    rows_wgrad_kernel<<<grid, 256, 0, stream>>>(B, M, N, dy, ldy, x, ldx, dw, ldw);
    return check_launch("rows_wgrad_kernel");
}

int rows_dgrad_chunks(int M) {
    const int by_rows = (M + 31) / 32;              // at least 32 rows per chunk
    return by_rows < kRowsDgradMaxChunks ? by_rows : kRowsDgradMaxChunks;
}

int rows_dgrad(int B, int M, int N, const float* dy, int64_t ldy, const __nv_bfloat16* w, int64_t ldw, float* dx,
               int64_t ldx, float* part, size_t part_floats, cudaStream_t stream) {
    const int chunks = rows_dgrad_chunks(M);
    if (B <= 0 || B > kRowsDgrad || M <= 0 || M % 8 || N <= 0 || N % 4 || ldw % 4 || ldx % 4 || ldy % 4 ||
        ldy < M || ldw < N || ldx < N)
        return set_error(FF_ERR_INVALID_ARG, "rows_dgrad: B=%d M=%d N=%d", B, M, N);
    if (part_floats < static_cast<size_t>(chunks) * B * N)
        return set_error(FF_ERR_WORKSPACE, "rows_dgrad: %zu partial floats < %zu", part_floats,
                         static_cast<size_t>(chunks) * B * N);
    const int rows_per_chunk = ((M + chunks - 1) / chunks + 7) / 8 * 8;   // chunks start on 8-row boundaries
    {
        ProfScope prof(stream, "rows_dgrad", 2.0 * B * M * N, 2.0 * M * N + 4.0 * B * M + 4.0 * chunks * B * N);
        const dim3 grid((N / 4 + 127) / 128, chunks);
        if (B <= 4) rows_dgrad_partial_kernel<4><<<grid, 128, 0, stream>>>(B, M, N, rows_per_chunk, dy, ldy, w, ldw, part);
        else if (B <= 8) rows_dgrad_partial_kernel<8><<<grid, 128, 0, stream>>>(B, M, N, rows_per_chunk, dy, ldy, w, ldw, part);
        else rows_dgrad_partial_kernel<16><<<grid, 128, 0, stream>>>(B, M, N, rows_per_chunk, dy, ldy, w, ldw, part);
        FF_TRY(check_launch("rows_dgrad_partial_kernel"));
    }
    rows_dgrad_sum_kernel<<<dim3((N / 4 + 255) / 256, B), 256, 0, stream>>>(B, N, chunks, part, dx, ldx);
    return check_launch("rows_dgrad_sum_kernel");
}

int wan_modulation_backward(const float* dmods, int64_t ld, int B, int rows_pad, int H, int L, float* gbias0,
                            int64_t stride, float* gfinal, float* de0, __nv_bfloat16* de0b, float* de_fin,
                            cudaStream_t stream) {
    if (B <= 0 || rows_pad < B || H <= 0 || L <= 0) return set_error(FF_ERR_INVALID_ARG, "wan_modulation_backward: bad shape");
    const int64_t total = static_cast<int64_t>(L) * 6 * H + 2 * H + static_cast<int64_t>(rows_pad) * 6 * H +
                          static_cast<int64_t>(B) * H;
    ProfScope prof(stream, "wan_modulation_backward", 0.0, 8.0 * B * (static_cast<double>(L) * 6 * H + 2 * H));
    wan_modulation_backward_kernel<<<static_cast<unsigned>((total + 255) / 256), 256, 0, stream>>>(
        dmods, ld, B, rows_pad, H, L, gbias0, stride, gfinal, de0, de0b, de_fin);
    return check_launch("wan_modulation_backward_kernel");
}

}  // namespace ff

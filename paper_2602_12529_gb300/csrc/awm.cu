// awm.cu -- the flow-matching objectives of Sec. 3.2: Advantage Weighted
// Matching (Eq. 3) and DiffusionNFT (Eq. 2).  AWM:
//   * training times t_b from the caller's random draws (uniform,
//     logit-normal or discrete);
//   * the forward process x_t = (1 - t_b) x0 + t_b eps;
//   * the loss (1/B) sum_b A_b e_b, e_b = ||v_b - (eps_b - x0_b)||^2 (or its
//     per-element mean), with dL/dv and the per-sample e_b;
//   * DiffusionNFT: (1/B) sum_b r_b e+_b + (1 - r_b) e-_b with e+-_b the
//     squared error of the implicit policies v+- (read from the cited
//     method: v+ = (1 - beta) v_old + beta v, v- = (1 + beta) v_old - beta v)
//     against eps - x0, with dL/dv.
// The elementwise kernels stream 128-bit loads over a (chunk, sample) grid
// with the per-sample scalars formed once per block.  The loss is reduced
// deterministically: one fp64 partial per (sample, block); then one block per
// sample adds its partials in a fixed order; then one block forms the
// advantage-weighted batch mean.
#include "internal.h"
#include "ptx.cuh"

namespace ff {
namespace {

constexpr int kThreads = 256;
constexpr int kVecPerThread = 4;                          // float4 per thread per chunk
constexpr int kChunk = kThreads * kVecPerThread * 4;      // 4096 elements
constexpr int kMaxBlocksPerSample = 1024;

int nchunks(int64_t D) {
    const int64_t c = (D + kChunk - 1) / kChunk;
    return static_cast<int>(c < kMaxBlocksPerSample ? c : kMaxBlocksPerSample);
}

__global__ void sample_timesteps_kernel(int mode, int B, const float* draw, float p0, float p1, const float* grid,
                                        int n_grid, float* t) {
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= B) return;
    const float d = draw[b];
    float r;
    if (mode == FF_TSAMPLE_UNIFORM) {
        r = fmaf(p1 - p0, d, p0);
    } else if (mode == FF_TSAMPLE_LOGIT_NORMAL) {
        r = 1.0f / (1.0f + expf(-fmaf(p1, d, p0)));
    } else {
        int k = static_cast<int>(floorf(d * static_cast<float>(n_grid)));
        k = k < 0 ? 0 : (k > n_grid - 1 ? n_grid - 1 : k);
        r = grid[k];
    }
    t[b] = r;
}

// x_t = (1 - t_b) x0 + t_b eps over a (chunk, sample) grid.
__global__ void __launch_bounds__(kThreads) forward_process_kernel(int64_t D, int nblk, const float* x0,
                                                                   const float* eps, const float* t, float* xt) {
    const int b = blockIdx.y;
    const float tb = t[b];
    const float sb = 1.0f - tb;
    const int64_t row = static_cast<int64_t>(b) * D;
    const float4* a4 = reinterpret_cast<const float4*>(x0 + row);
    const float4* e4 = reinterpret_cast<const float4*>(eps + row);
    float4* o4 = reinterpret_cast<float4*>(xt + row);
    const int64_t nvec = D >> 2;
    for (int64_t base = static_cast<int64_t>(blockIdx.x) * (kChunk / 4); base < nvec;
         base += static_cast<int64_t>(nblk) * (kChunk / 4)) {
        float4 av[kVecPerThread], ev[kVecPerThread];
#pragma unroll
        for (int j = 0; j < kVecPerThread; ++j) {
            const int64_t i = base + threadIdx.x + j * kThreads;
            if (i < nvec) {
                av[j] = __ldcs(a4 + i);
                ev[j] = __ldcs(e4 + i);
            }
        }
#pragma unroll
        for (int j = 0; j < kVecPerThread; ++j) {
            const int64_t i = base + threadIdx.x + j * kThreads;
            if (i < nvec)
                __stcs(o4 + i, make_float4(fmaf(tb, ev[j].x, sb * av[j].x), fmaf(tb, ev[j].y, sb * av[j].y),
                                           fmaf(tb, ev[j].z, sb * av[j].z), fmaf(tb, ev[j].w, sb * av[j].w)));
        }
    }
}

__device__ __forceinline__ double block_sum(double v, double* red) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int w = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) red[w] = v;
    __syncthreads();
    double s = 0.0;
    if (threadIdx.x == 0) {
        for (int i = 0; i < (int)(blockDim.x >> 5); ++i) s += red[i];
    }
    return s;   // valid in thread 0
}

// Pass 1: residual r = v - (eps - x0); one fp64 partial of sum r^2 per
// (sample, block); with GRAD, dL/dv = gscale_b r, gscale_b = 2 A_b scale / B.
template <bool GRAD>
__global__ void __launch_bounds__(kThreads) awm_partial_kernel(int64_t D, int nblk, const float* v, const float* eps,
                                                               const float* x0, const float* adv, double gcoef,
                                                               float* grad, double* partial) {
    __shared__ double red[kThreads / 32];
    const int b = blockIdx.y;
    const float gs = GRAD ? static_cast<float>(gcoef * static_cast<double>(adv[b])) : 0.0f;
    const int64_t row = static_cast<int64_t>(b) * D;
    const float4* v4 = reinterpret_cast<const float4*>(v + row);
    const float4* e4 = reinterpret_cast<const float4*>(eps + row);
    const float4* a4 = reinterpret_cast<const float4*>(x0 + row);
    float4* g4 = reinterpret_cast<float4*>(grad + (GRAD ? row : 0));
    const int64_t nvec = D >> 2;
    float ss = 0.f;
    for (int64_t base = static_cast<int64_t>(blockIdx.x) * (kChunk / 4); base < nvec;
         base += static_cast<int64_t>(nblk) * (kChunk / 4)) {
        float4 vv[kVecPerThread], ev[kVecPerThread], av[kVecPerThread];
#pragma unroll
        for (int j = 0; j < kVecPerThread; ++j) {
            const int64_t i = base + threadIdx.x + j * kThreads;
            if (i < nvec) {
                vv[j] = __ldcs(v4 + i);
                ev[j] = __ldcs(e4 + i);
                av[j] = __ldcs(a4 + i);
            }
        }
#pragma unroll
        for (int j = 0; j < kVecPerThread; ++j) {
            const int64_t i = base + threadIdx.x + j * kThreads;
            if (i < nvec) {
                const float r0 = vv[j].x - (ev[j].x - av[j].x), r1 = vv[j].y - (ev[j].y - av[j].y);
                const float r2 = vv[j].z - (ev[j].z - av[j].z), r3 = vv[j].w - (ev[j].w - av[j].w);
                ss = fmaf(r0, r0, ss);
                ss = fmaf(r1, r1, ss);
                ss = fmaf(r2, r2, ss);
                ss = fmaf(r3, r3, ss);
                if (GRAD) __stcs(g4 + i, make_float4(gs * r0, gs * r1, gs * r2, gs * r3));
            }
        }
    }
    const double s = block_sum(static_cast<double>(ss), red);
    if (threadIdx.x == 0) partial[static_cast<int64_t>(b) * nblk + blockIdx.x] = s;
}

// Pass 2 (one block per sample): e_b = scale * the sum of its partials,
// thread i taking partials i, i + 256, ... and the block sum in a fixed tree.
__global__ void __launch_bounds__(kThreads) awm_sample_kernel(int nblk, const double* partial, double scale,
                                                              double* e_ws, float* err) {
    __shared__ double red[kThreads / 32];
    const int b = blockIdx.x;
    double s = 0.0;
    for (int k = threadIdx.x; k < nblk; k += kThreads) s += partial[static_cast<int64_t>(b) * nblk + k];
    s = block_sum(s, red) * scale;
    if (threadIdx.x == 0) {
        e_ws[b] = s;
        if (err) err[b] = static_cast<float>(s);
    }
}

// Pass 3 (one block): loss = (1/B) sum_b A_b e_b, thread i taking samples
// i, i + 256, ... in order, then the fixed tree.
__global__ void __launch_bounds__(kThreads) awm_batch_kernel(int B, const double* e_ws, const float* adv,
                                                             float* loss) {
    __shared__ double red[kThreads / 32];
    double acc = 0.0;
    for (int b = threadIdx.x; b < B; b += kThreads) acc += static_cast<double>(adv[b]) * e_ws[b];
    const double s = block_sum(acc, red);
    if (threadIdx.x == 0) *loss = static_cast<float>(s / B);
}

// DiffusionNFT (Eq. 2), pass 1: with target = eps - x0,
// v+ = (1 - beta) v_old + beta v, v- = (1 + beta) v_old - beta v, one fp64
// partial of sum (v+ - target)^2 and one of sum (v- - target)^2 per
// (sample, block); with GRAD, dL/dv = gs (r_b (v+ - target) - (1 - r_b)
// (v- - target)), gs = 2 beta scale / B.
template <bool GRAD>
__global__ void __launch_bounds__(kThreads) nft_partial_kernel(int64_t D, int nblk, const float* v, const float* v_old,
                                                               const float* eps, const float* x0, const float* r,
                                                               float beta, float gs, float* grad, double* partial) {
    __shared__ double red[2][kThreads / 32];
    const int b = blockIdx.y;
    const float rb = GRAD ? r[b] : 0.0f;
    const float wp = gs * rb, wn = gs * (1.0f - rb);
    const float cp = 1.0f - beta, cn = 1.0f + beta;
    const int64_t row = static_cast<int64_t>(b) * D;
    const float4* v4 = reinterpret_cast<const float4*>(v + row);
    const float4* o4 = reinterpret_cast<const float4*>(v_old + row);
    const float4* e4 = reinterpret_cast<const float4*>(eps + row);
    const float4* a4 = reinterpret_cast<const float4*>(x0 + row);
    float4* g4 = reinterpret_cast<float4*>(grad + (GRAD ? row : 0));
    const int64_t nvec = D >> 2;
    float sp = 0.f, sn = 0.f;
    for (int64_t base = static_cast<int64_t>(blockIdx.x) * (kChunk / 4); base < nvec;
         base += static_cast<int64_t>(nblk) * (kChunk / 4)) {
        float4 vv[kVecPerThread], ov[kVecPerThread], ev[kVecPerThread], av[kVecPerThread];
#pragma unroll
        for (int j = 0; j < kVecPerThread; ++j) {
            const int64_t i = base + threadIdx.x + j * kThreads;
            if (i < nvec) {
                vv[j] = __ldcs(v4 + i);
                ov[j] = __ldcs(o4 + i);
                ev[j] = __ldcs(e4 + i);
                av[j] = __ldcs(a4 + i);
            }
        }
#pragma unroll
        for (int j = 0; j < kVecPerThread; ++j) {
            const int64_t i = base + threadIdx.x + j * kThreads;
            if (i < nvec) {
                const float vx[4] = {vv[j].x, vv[j].y, vv[j].z, vv[j].w};
                const float ox[4] = {ov[j].x, ov[j].y, ov[j].z, ov[j].w};
                const float tx[4] = {ev[j].x - av[j].x, ev[j].y - av[j].y, ev[j].z - av[j].z, ev[j].w - av[j].w};
                float g[4];
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const float rp = fmaf(cp, ox[k], beta * vx[k]) - tx[k];
                    const float rn = fmaf(cn, ox[k], -beta * vx[k]) - tx[k];
                    sp = fmaf(rp, rp, sp);
                    sn = fmaf(rn, rn, sn);
                    g[k] = wp * rp - wn * rn;
                }
                if (GRAD) __stcs(g4 + i, make_float4(g[0], g[1], g[2], g[3]));
            }
        }
    }
    const double a = block_sum(static_cast<double>(sp), red[0]);
    const double c = block_sum(static_cast<double>(sn), red[1]);
    if (threadIdx.x == 0) {
        partial[(static_cast<int64_t>(b) * nblk + blockIdx.x) * 2] = a;
        partial[(static_cast<int64_t>(b) * nblk + blockIdx.x) * 2 + 1] = c;
    }
}

// Pass 2 (one block per sample): e+_b, e-_b in a fixed order; pass 3 (one
// block): loss = (1/B) sum_b r_b e+_b + (1 - r_b) e-_b.
__global__ void __launch_bounds__(kThreads) nft_sample_kernel(int nblk, const double* partial, double scale,
                                                              double* e_ws, float* err) {
    __shared__ double red[2][kThreads / 32];
    const int b = blockIdx.x;
    double sp = 0.0, sn = 0.0;
    for (int k = threadIdx.x; k < nblk; k += kThreads) {
        sp += partial[(static_cast<int64_t>(b) * nblk + k) * 2];
        sn += partial[(static_cast<int64_t>(b) * nblk + k) * 2 + 1];
    }
    sp = block_sum(sp, red[0]) * scale;
    sn = block_sum(sn, red[1]) * scale;
    if (threadIdx.x == 0) {
        e_ws[2 * b] = sp;
        e_ws[2 * b + 1] = sn;
        if (err) {
            err[2 * b] = static_cast<float>(sp);
            err[2 * b + 1] = static_cast<float>(sn);
        }
    }
}

__global__ void __launch_bounds__(kThreads) nft_batch_kernel(int B, const double* e_ws, const float* r, float* loss) {
    __shared__ double red[kThreads / 32];
    double acc = 0.0;
    for (int b = threadIdx.x; b < B; b += kThreads) {
        const double rb = r[b];
        acc += rb * e_ws[2 * b] + (1.0 - rb) * e_ws[2 * b + 1];
    }
    const double s = block_sum(acc, red);
    if (threadIdx.x == 0) *loss = static_cast<float>(s / B);
}

}  // namespace
}  // namespace ff

extern "C" {

int ff_nft_loss_workspace_size(int B, int64_t D, size_t* bytes) {
    if (!bytes) return ff::set_error(FF_ERR_INVALID_ARG, "bytes is null");
    if (B <= 0 || D <= 0) return ff::set_error(FF_ERR_INVALID_ARG, "B and D must be positive");
    *bytes = static_cast<size_t>(B) * static_cast<size_t>(ff::nchunks(D) + 1) * 2 * sizeof(double);
    return FF_OK;
}

int ff_nft_loss(int B, int64_t D, const float* v, const float* v_old, const float* eps, const float* x0,
                const float* r, float beta, int reduce, float* loss, float* grad_v, float* err_out, void* ws,
                size_t ws_bytes, cudaStream_t stream) {
    using namespace ff;
    if (B <= 0 || D <= 0) return set_error(FF_ERR_INVALID_ARG, "nft: B=%d D=%lld must be positive", B, (long long)D);
    if (D % 4) return set_error(FF_ERR_UNSUPPORTED, "nft: D=%lld not a multiple of 4", (long long)D);
    if (B > 65535) return set_error(FF_ERR_UNSUPPORTED, "nft: B=%d > 65535", B);
    if (reduce != FF_AWM_SUM && reduce != FF_AWM_MEAN) return set_error(FF_ERR_INVALID_ARG, "nft: bad reduce %d", reduce);
    if (!(beta > 0.0f)) return set_error(FF_ERR_INVALID_ARG, "nft: beta must be > 0");
    if (!v || !v_old || !eps || !x0 || !r || !loss) return set_error(FF_ERR_INVALID_ARG, "nft: null pointer");
    if (!aligned16(v) || !aligned16(v_old) || !aligned16(eps) || !aligned16(x0) || (grad_v && !aligned16(grad_v)))
        return set_error(FF_ERR_INVALID_ARG, "nft: arrays must be 16-byte aligned");
    const int nb = nchunks(D);
    const size_t need = static_cast<size_t>(B) * (nb + 1) * 2 * sizeof(double);   // partials, then e+-_b
    if (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 7))
        return set_error(FF_ERR_WORKSPACE, "nft: workspace %zu B < %zu B needed (or misaligned)", ws_bytes, need);
    double* partial = static_cast<double*>(ws);
    const double scale = reduce == FF_AWM_MEAN ? 1.0 / static_cast<double>(D) : 1.0;
    const float gs = static_cast<float>(2.0 * beta * scale / B);
    {
    ProfScope prof(stream, "nft_loss", 0.0, static_cast<double>(B) * D * (grad_v ? 20.0 : 16.0));
    if (grad_v)
        nft_partial_kernel<true><<<dim3(nb, B), kThreads, 0, stream>>>(D, nb, v, v_old, eps, x0, r, beta, gs, grad_v,
                                                                       partial);
    else
        nft_partial_kernel<false><<<dim3(nb, B), kThreads, 0, stream>>>(D, nb, v, v_old, eps, x0, r, beta, 0.f,
                                                                        nullptr, partial);
    }
    int rc = check_launch("nft_partial_kernel");
    if (rc) return rc;
    double* e_ws = partial + static_cast<size_t>(B) * nb * 2;
    {
    ProfScope prof(stream, "nft_finalize", 0.0, static_cast<double>(B) * nb * 16.0 + 20.0 * B);
    nft_sample_kernel<<<B, kThreads, 0, stream>>>(nb, partial, scale, e_ws, err_out);
    rc = check_launch("nft_sample_kernel");
    if (rc) return rc;
    nft_batch_kernel<<<1, kThreads, 0, stream>>>(B, e_ws, r, loss);
    }
    return check_launch("nft_batch_kernel");
}

int ff_sample_timesteps(int mode, int B, const float* draw, float p0, float p1, const float* grid, int n_grid,
                        float* t_out, cudaStream_t stream) {
    using namespace ff;
    if (B <= 0 || !draw || !t_out) return set_error(FF_ERR_INVALID_ARG, "timesteps: bad arguments");
    if (mode != FF_TSAMPLE_UNIFORM && mode != FF_TSAMPLE_LOGIT_NORMAL && mode != FF_TSAMPLE_DISCRETE)
        return set_error(FF_ERR_INVALID_ARG, "timesteps: bad mode %d", mode);
    if (mode == FF_TSAMPLE_DISCRETE && (!grid || n_grid <= 0))
        return set_error(FF_ERR_INVALID_ARG, "timesteps: the discrete sampler needs a grid");
    if (mode == FF_TSAMPLE_LOGIT_NORMAL && !(p1 >= 0.0f))
        return set_error(FF_ERR_INVALID_ARG, "timesteps: the logit-normal scale must be >= 0");
    ProfScope prof(stream, "sample_timesteps", 0.0, 8.0 * B);
    sample_timesteps_kernel<<<(B + 255) / 256, 256, 0, stream>>>(mode, B, draw, p0, p1, grid, n_grid, t_out);
    return check_launch("sample_timesteps_kernel");
}

int ff_forward_process(int B, int64_t D, const float* x0, const float* eps, const float* t, float* x_t,
                       cudaStream_t stream) {
    using namespace ff;
    if (B <= 0 || D <= 0) return set_error(FF_ERR_INVALID_ARG, "forward process: B=%d D=%lld", B, (long long)D);
    if (D % 4) return set_error(FF_ERR_UNSUPPORTED, "forward process: D=%lld not a multiple of 4", (long long)D);
    if (B > 65535) return set_error(FF_ERR_UNSUPPORTED, "forward process: B=%d > 65535", B);
    if (!x0 || !eps || !t || !x_t) return set_error(FF_ERR_INVALID_ARG, "forward process: null pointer");
    if (!aligned16(x0) || !aligned16(eps) || !aligned16(x_t))
        return set_error(FF_ERR_INVALID_ARG, "forward process: arrays must be 16-byte aligned");
    const int nb = nchunks(D);
    ProfScope prof(stream, "forward_process", 0.0, 12.0 * static_cast<double>(B) * D);
    forward_process_kernel<<<dim3(nb, B), kThreads, 0, stream>>>(D, nb, x0, eps, t, x_t);
    return check_launch("forward_process_kernel");
}

int ff_awm_loss_workspace_size(int B, int64_t D, size_t* bytes) {
    if (!bytes) return ff::set_error(FF_ERR_INVALID_ARG, "bytes is null");
    if (B <= 0 || D <= 0) return ff::set_error(FF_ERR_INVALID_ARG, "B and D must be positive");
    *bytes = static_cast<size_t>(B) * static_cast<size_t>(ff::nchunks(D) + 1) * sizeof(double);
    return FF_OK;
}

int ff_awm_loss(int B, int64_t D, const float* v, const float* eps, const float* x0, const float* adv, int reduce,
                float* loss, float* grad_v, float* err_out, void* ws, size_t ws_bytes, cudaStream_t stream) {
    using namespace ff;
    if (B <= 0 || D <= 0) return set_error(FF_ERR_INVALID_ARG, "awm: B=%d D=%lld must be positive", B, (long long)D);
    if (D % 4) return set_error(FF_ERR_UNSUPPORTED, "awm: D=%lld not a multiple of 4", (long long)D);
    if (B > 65535) return set_error(FF_ERR_UNSUPPORTED, "awm: B=%d > 65535", B);
    if (reduce != FF_AWM_SUM && reduce != FF_AWM_MEAN) return set_error(FF_ERR_INVALID_ARG, "awm: bad reduce %d", reduce);
    if (!v || !eps || !x0 || !adv || !loss) return set_error(FF_ERR_INVALID_ARG, "awm: null pointer");
    if (!aligned16(v) || !aligned16(eps) || !aligned16(x0) || (grad_v && !aligned16(grad_v)))
        return set_error(FF_ERR_INVALID_ARG, "awm: arrays must be 16-byte aligned");
    const int nb = nchunks(D);
    const size_t need = static_cast<size_t>(B) * (nb + 1) * sizeof(double);   // partials, then e_b
    if (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 7))
        return set_error(FF_ERR_WORKSPACE, "awm: workspace %zu B < %zu B needed (or misaligned)", ws_bytes, need);
    double* partial = static_cast<double*>(ws);
    const double scale = reduce == FF_AWM_MEAN ? 1.0 / static_cast<double>(D) : 1.0;
    {
    ProfScope prof(stream, "awm_loss", 0.0, static_cast<double>(B) * D * (grad_v ? 16.0 : 12.0));
    if (grad_v)
        awm_partial_kernel<true><<<dim3(nb, B), kThreads, 0, stream>>>(D, nb, v, eps, x0, adv, 2.0 * scale / B,
                                                                       grad_v, partial);
    else
        awm_partial_kernel<false><<<dim3(nb, B), kThreads, 0, stream>>>(D, nb, v, eps, x0, adv, 0.0, nullptr,
                                                                        partial);
    }
    int rc = check_launch("awm_partial_kernel");
    if (rc) return rc;
    double* e_ws = partial + static_cast<size_t>(B) * nb;
    {
    ProfScope prof(stream, "awm_finalize", 0.0, static_cast<double>(B) * nb * 8.0 + 12.0 * B);
    awm_sample_kernel<<<B, kThreads, 0, stream>>>(nb, partial, scale, e_ws, err_out);
    rc = check_launch("awm_sample_kernel");
    if (rc) return rc;
    awm_batch_kernel<<<1, kThreads, 0, stream>>>(B, e_ws, adv, loss);
    }
    return check_launch("awm_batch_kernel");
}

}  // extern "C"

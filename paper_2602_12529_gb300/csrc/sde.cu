// sde.cu -- fused Flow-SDE step and Gaussian transition log-probability
// (paper Eq. 1 and Table 1).
//
// Per sample b (Delta = t - t_next > 0, a = sigma^2 / (2 t)):
//   mean = x - Delta (v + a (x + (1 - t) v)) = cx x + cv v,
//          cx = 1 - Delta a,  cv = -Delta (1 + a (1 - t))
//   std  = sigma sqrt(Delta)
//   SAMPLE: x_next = mean + std eps;  EVAL: x_next given; SAMPLE with eps
//   drawn in the kernel from the counter-based generator of rng.cuh
//   logp = -sum (x_next - mean)^2 / (2 std^2) - D ln std - D/2 ln 2 pi
// Everything is fp32: fp64 arithmetic runs on very few units of this part,
// and a handful of dependent fp64 operations (a log, a square root, a
// shuffle reduction) cost microseconds.  The per-sample coefficients are
// formed by every thread; the elementwise work is FMAs over 128-bit loads.
// One launch: every block writes one partial sum of squared residuals, then
// takes a ticket; the block that draws the sample's last ticket adds that
// sample's partials in a fixed order (so the result does not depend on which
// block finished last), writes logp and puts the ticket word back to zero.
// The partials of up to 1024 blocks are added pairwise-ish (four per thread,
// then shuffles, then eight warps in order): relative error about 1e-6.
#include "internal.h"
#include "ptx.cuh"
#include "rng.cuh"

namespace ff {
namespace {

constexpr int kThreads = 256;
constexpr int kModePhilox = 2;                                // SAMPLE, eps from rng.cuh (internal mode)
constexpr int kVecPerThread = 4;                              // float4 per thread per chunk
constexpr int kChunk = kThreads * kVecPerThread * 4;          // 4096 elements

struct StepCoef {
    float cx, cv, std;
};

// Per-sample coefficients in fp32 (every thread forms its own: no barrier,
// and fp64 arithmetic is slow on this part).  Relative error a few ulp.
__device__ __forceinline__ StepCoef step_coef(const float* t, const float* t_next, const float* sigma, int b) {
    const float tt = __ldg(t + b);
    const float tn = __ldg(t_next + b);
    const float sg = __ldg(sigma + b);
    const float delta = tt - tn;
    const float a = sg * sg / (2.0f * tt);
    StepCoef c;
    c.cx = fmaf(-delta, a, 1.0f);
    c.cv = -delta * fmaf(a, 1.0f - tt, 1.0f);
    c.std = sg * sqrtf(delta);
    return c;
}

// Sum over the block in fp32 (shuffles, then the warps' sums in order by
// thread 0); valid in thread 0.
__device__ __forceinline__ float block_sum_f32(float v, float* red) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    float s = 0.f;
    if (threadIdx.x == 0) {
        for (int i = 0; i < (int)(blockDim.x >> 5); ++i) s += red[i];
    }
    return s;
}

// The log-probability of sample b from its summed squared residual ss:
// -ss / (2 std^2) - D ln std - D/2 ln 2 pi (divided by D for FF_LP_MEAN);
// 0 when std == 0 (no density).  The three terms are each about D in size
// and do not cancel, so fp32 keeps about 1e-6 of relative accuracy.
__device__ __forceinline__ float logprob_of(float ss, int64_t D, const float* t, const float* t_next,
                                            const float* sigma, int b, int reduce) {
    const float delta = t[b] - t_next[b];
    const float sd = sigma[b] * sqrtf(delta);
    if (!(sd > 0.f)) return 0.f;
    const float dd = static_cast<float>(D);
    const float kHalfLog2Pi = 0.91893853320467274f;   // ln(2 pi) / 2
    float lp = -(0.5f * ss / (sd * sd) + dd * (logf(sd) + kHalfLog2Pi));
    if (reduce == FF_LP_MEAN) lp /= dd;
    return lp;
}

// Grid (blocks_per_sample, B); block k of sample b handles chunks
// k, k + blocks_per_sample, ... and writes one fp32 partial.  The number of
// blocks per sample depends only on D (see nchunks), so the summation order
// is fixed.
// ticket[b] counts the blocks of sample b that have stored their partial; it
// is zero on entry and the last block of the sample sets it back to zero.
template <int MODE>
__global__ void __launch_bounds__(kThreads) sde_step_partial_kernel(int64_t D, int nblk, const float* x,
                                                                    const float* v, const float* eps, float* x_next,
                                                                    const float* t, const float* t_next,
                                                                    const float* sigma, float* partial,
                                                                    unsigned* ticket, int reduce, float* logp, int ld,
                                                                    PhiloxKey key, uint32_t rng_stream) {
    __shared__ float redf[kThreads / 32];
    const int b = blockIdx.y;
    const StepCoef c = step_coef(t, t_next, sigma, b);
    const int64_t row = static_cast<int64_t>(b) * D;
    const float4* x4 = reinterpret_cast<const float4*>(x + row);
    const float4* v4 = reinterpret_cast<const float4*>(v + row);
    const float4* e4 = reinterpret_cast<const float4*>(eps + (MODE == FF_SDE_SAMPLE ? row : 0));
    float4* n4 = reinterpret_cast<float4*>(x_next + row);
    const int64_t nvec = D >> 2;
    float ss = 0.f;
    for (int64_t base = static_cast<int64_t>(blockIdx.x) * (kChunk / 4); base < nvec;
         base += static_cast<int64_t>(nblk) * (kChunk / 4)) {
        // every load of the chunk is issued before any arithmetic; the
        // inputs keep the default cache policy (a rollout's v and x_t are
        // often still in L2) and so does x_next (the next step reads it)
        float4 xv[kVecPerThread], vv[kVecPerThread], ev[kVecPerThread];
#pragma unroll
        for (int j = 0; j < kVecPerThread; ++j) {
            const int64_t i = base + threadIdx.x + j * kThreads;
            if (i < nvec) {
                xv[j] = __ldg(x4 + i);
                vv[j] = __ldg(v4 + i);
                if (MODE == FF_SDE_SAMPLE) ev[j] = __ldg(e4 + i);
                else if (MODE == FF_SDE_EVAL) ev[j] = *(reinterpret_cast<const float4*>(n4) + i);
            }
        }
        if (MODE == kModePhilox) {
#pragma unroll
            for (int j = 0; j < kVecPerThread; ++j) {
                const int64_t i = base + threadIdx.x + j * kThreads;
                if (i < nvec) ev[j] = philox_normal4(static_cast<uint32_t>(i), b, rng_stream, key);
            }
        }
#pragma unroll
        for (int j = 0; j < kVecPerThread; ++j) {
            const int64_t i = base + threadIdx.x + j * kThreads;
            if (i < nvec) {
                float m[4] = {fmaf(c.cx, xv[j].x, c.cv * vv[j].x), fmaf(c.cx, xv[j].y, c.cv * vv[j].y),
                              fmaf(c.cx, xv[j].z, c.cv * vv[j].z), fmaf(c.cx, xv[j].w, c.cv * vv[j].w)};
                float o[4];
                if (MODE != FF_SDE_EVAL) {
                    o[0] = fmaf(c.std, ev[j].x, m[0]);
                    o[1] = fmaf(c.std, ev[j].y, m[1]);
                    o[2] = fmaf(c.std, ev[j].z, m[2]);
                    o[3] = fmaf(c.std, ev[j].w, m[3]);
                    n4[i] = make_float4(o[0], o[1], o[2], o[3]);
                } else {
                    o[0] = ev[j].x; o[1] = ev[j].y; o[2] = ev[j].z; o[3] = ev[j].w;
                }
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const float r = o[k] - m[k];
                    ss = fmaf(r, r, ss);
                }
            }
        }
    }
    const float s = block_sum_f32(ss, redf);
    __shared__ bool last;
    if (threadIdx.x == 0) {
        partial[static_cast<int64_t>(b) * nblk + blockIdx.x] = s;
        last = ticket_add_acq_rel(ticket + b, 1u) == static_cast<unsigned>(nblk - 1);
    }
    __syncthreads();
    if (!last) return;
    // every partial of sample b is stored (the last ticket acquired them);
    // add them in index order
    const float* pb = partial + static_cast<int64_t>(b) * nblk;
    float acc = 0.f;
    for (int i = threadIdx.x; i < nblk; i += kThreads) acc += __ldcg(pb + i);
    acc = block_sum_f32(acc, redf);
    if (threadIdx.x == 0) {
        ticket[b] = 0u;
        logp[static_cast<int64_t>(b) * ld] = logprob_of(acc, D, t, t_next, sigma, b, reduce);
    }
}

// out[b, 4g .. 4g + 3] = the normals of element group g of sample b (rng.cuh).
__global__ void __launch_bounds__(kThreads) philox_normal_kernel(int B, int64_t nvec, PhiloxKey key,
                                                                 uint32_t rng_stream, float4* out) {
    const int64_t total = static_cast<int64_t>(B) * nvec;
    for (int64_t k = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; k < total;
         k += static_cast<int64_t>(gridDim.x) * kThreads) {
        const int64_t b = k / nvec, g = k - b * nvec;
        __stcs(out + k, philox_normal4(static_cast<uint32_t>(g), static_cast<uint32_t>(b), rng_stream, key));
    }
}

// Backward of the log-probability in v with x_next held fixed:
// d logp / d v_j = (x_next_j - mean_j) / std^2 * cv (divided by D for the
// mean reduction), times the upstream gradient g[b * ldg].  Zero where
// std = 0 (no density, logp reported as 0).  Same mean arithmetic as the
// forward kernel.
__global__ void __launch_bounds__(kThreads) sde_logprob_backward_kernel(int64_t D, int nblk, const float* x,
                                                                        const float* v, const float* x_next,
                                                                        const float* t, const float* t_next,
                                                                        const float* sigma, const float* g, int ldg,
                                                                        int reduce, float* dv) {
    const int b = blockIdx.y;
    const StepCoef sc = step_coef(t, t_next, sigma, b);
    float k = 0.f;
    if (sc.std > 0.f) {
        const float delta = t[b] - t_next[b];
        const float sg = sigma[b];
        k = g[static_cast<int64_t>(b) * ldg] * sc.cv / (sg * sg * delta);
        if (reduce == FF_LP_MEAN) k /= static_cast<float>(D);
    }
    const float3 c = make_float3(sc.cx, sc.cv, k);
    const int64_t row = static_cast<int64_t>(b) * D;
    const float4* x4 = reinterpret_cast<const float4*>(x + row);
    const float4* v4 = reinterpret_cast<const float4*>(v + row);
    const float4* n4 = reinterpret_cast<const float4*>(x_next + row);
    float4* d4 = reinterpret_cast<float4*>(dv + row);
    const int64_t nvec = D >> 2;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; i < nvec;
         i += static_cast<int64_t>(nblk) * kThreads) {
        const float4 xv = __ldcs(x4 + i), vv = __ldcs(v4 + i), nv = __ldcs(n4 + i);
        float4 o;
        o.x = c.z * (nv.x - fmaf(c.x, xv.x, c.y * vv.x));
        o.y = c.z * (nv.y - fmaf(c.x, xv.y, c.y * vv.y));
        o.z = c.z * (nv.z - fmaf(c.x, xv.z, c.y * vv.z));
        o.w = c.z * (nv.w - fmaf(c.x, xv.w, c.y * vv.w));
        __stcs(d4 + i, o);
    }
}

constexpr int kMaxBlocksPerSample = 1024;
constexpr int kMaxSamples = 65535;

// Workspace layout: the ticket words of up to kMaxSamples samples at a fixed
// place (offset 0), then the fp64 partials.  Keeping the tickets at the same
// offset whatever B and D are means a workspace zeroed once stays valid for
// calls of any shape: no call ever stores a partial over a ticket word.
constexpr size_t kTicketBytes = 256 * 1024;
static_assert(kTicketBytes >= sizeof(unsigned) * kMaxSamples, "ticket region too small");

// partial sums (blocks) per sample: one per 4096-element chunk up to 1024,
// then every block loops over several chunks
int nchunks(int64_t D) {
    const int64_t c = (D + kChunk - 1) / kChunk;
    return static_cast<int>(c < kMaxBlocksPerSample ? c : kMaxBlocksPerSample);
}

}  // namespace
}  // namespace ff

extern "C" {

int ff_sde_workspace_size(int B, int64_t D, size_t* bytes) {
    if (!bytes) return ff::set_error(FF_ERR_INVALID_ARG, "bytes is null");
    if (B <= 0 || D <= 0) return ff::set_error(FF_ERR_INVALID_ARG, "B and D must be positive");
    *bytes = ff::kTicketBytes + static_cast<size_t>(B) * static_cast<size_t>(ff::nchunks(D)) * sizeof(float);
    return FF_OK;
}

}  // extern "C"

namespace ff {
namespace {

// One launch of the SDE step (mode FF_SDE_SAMPLE, FF_SDE_EVAL or
// kModePhilox) over caller scratch: tickets (zero on entry, zero again on
// exit) and B * nchunks(D) fp64 partials.
int launch_sde_step(int B, int64_t D, int nc, const float* x_t, const float* v, const float* eps, float* x_next,
                    const float* t, const float* t_next, const float* sigma, int mode, int reduce, float* logp,
                    int ld, unsigned* ticket, float* partial, PhiloxKey key, uint32_t rng_stream,
                    cudaStream_t stream) {
    const dim3 grid(nc, B);
    ProfScope prof(stream, "sde_step", 0.0, static_cast<double>(B) * D * (mode == FF_SDE_SAMPLE ? 16.0 : 12.0));
    if (mode == FF_SDE_SAMPLE)
        sde_step_partial_kernel<FF_SDE_SAMPLE><<<grid, kThreads, 0, stream>>>(
            D, nc, x_t, v, eps, x_next, t, t_next, sigma, partial, ticket, reduce, logp, ld, key, rng_stream);
    else if (mode == kModePhilox)
        sde_step_partial_kernel<kModePhilox><<<grid, kThreads, 0, stream>>>(
            D, nc, x_t, v, eps, x_next, t, t_next, sigma, partial, ticket, reduce, logp, ld, key, rng_stream);
    else
        sde_step_partial_kernel<FF_SDE_EVAL><<<grid, kThreads, 0, stream>>>(
            D, nc, x_t, v, eps, x_next, t, t_next, sigma, partial, ticket, reduce, logp, ld, key, rng_stream);
    return check_launch("sde_step_kernel");
}

// Argument checks of one SDE step, then its launch.
int sde_step(int B, int64_t D, const float* x_t, const float* v, const float* eps, float* x_next, const float* t,
             const float* t_next, const float* sigma, int mode, int reduce, float* logp, int ld, void* ws,
             size_t ws_bytes, PhiloxKey key, uint32_t rng_stream, cudaStream_t stream) {
    if (B <= 0 || D <= 0) return set_error(FF_ERR_INVALID_ARG, "sde: B=%d D=%lld must be positive", B, (long long)D);
    if (D % 4) return set_error(FF_ERR_UNSUPPORTED, "sde: D=%lld not a multiple of 4", (long long)D);
    if (reduce != FF_LP_SUM && reduce != FF_LP_MEAN) return set_error(FF_ERR_INVALID_ARG, "sde: bad reduce %d", reduce);
    if (!x_t || !v || !x_next || !t || !t_next || !sigma || !logp || (mode == FF_SDE_SAMPLE && !eps))
        return set_error(FF_ERR_INVALID_ARG, "sde: null pointer");
    if (!aligned16(x_t) || !aligned16(v) || !aligned16(x_next) || (mode == FF_SDE_SAMPLE && !aligned16(eps)))
        return set_error(FF_ERR_INVALID_ARG, "sde: arrays must be 16-byte aligned");
    if (ld < 1) return set_error(FF_ERR_INVALID_ARG, "sde: ld=%d < 1", ld);
    if (B > kMaxSamples) return set_error(FF_ERR_UNSUPPORTED, "sde: B=%d > %d", B, kMaxSamples);
    if (mode == kModePhilox && D / 4 > 0xFFFFFFFFll)
        return set_error(FF_ERR_UNSUPPORTED, "sde: D=%lld too large for the generator's counter", (long long)D);
    const int nc = nchunks(D);
    const size_t need = kTicketBytes + static_cast<size_t>(B) * nc * sizeof(float);
    if (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 15))
        return set_error(FF_ERR_WORKSPACE, "sde: workspace %zu B < %zu B needed (or not 16-byte aligned)", ws_bytes,
                         need);
    unsigned* ticket = static_cast<unsigned*>(ws);
    float* partial = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) + kTicketBytes);
    return launch_sde_step(B, D, nc, x_t, v, eps, x_next, t, t_next, sigma, mode, reduce, logp, ld, ticket, partial,
                           key, rng_stream, stream);
}

}  // namespace
}  // namespace ff

extern "C" {

int ff_sde_step_logprob(int B, int64_t D, const float* x_t, const float* v, const float* eps, float* x_next,
                        const float* t, const float* t_next, const float* sigma, int mode, int reduce, float* logp,
                        int ld, void* ws, size_t ws_bytes, cudaStream_t stream) {
    using namespace ff;
    if (mode != FF_SDE_SAMPLE && mode != FF_SDE_EVAL) return set_error(FF_ERR_INVALID_ARG, "sde: bad mode %d", mode);
    return sde_step(B, D, x_t, v, eps, x_next, t, t_next, sigma, mode, reduce, logp, ld, ws, ws_bytes, PhiloxKey{0, 0},
                    0u, stream);
}

int ff_sde_step_logprob_philox(int B, int64_t D, const float* x_t, const float* v, float* x_next, const float* t,
                               const float* t_next, const float* sigma, uint64_t seed, uint32_t rng_stream, int reduce,
                               float* logp, int ld, void* ws, size_t ws_bytes, cudaStream_t stream) {
    using namespace ff;
    return sde_step(B, D, x_t, v, nullptr, x_next, t, t_next, sigma, kModePhilox, reduce, logp, ld, ws, ws_bytes,
                    philox_key(seed), rng_stream, stream);
}

int ff_philox_normal(int B, int64_t D, uint64_t seed, uint32_t rng_stream, float* out, cudaStream_t stream) {
    using namespace ff;
    if (B <= 0 || D <= 0 || !out) return set_error(FF_ERR_INVALID_ARG, "philox: B=%d D=%lld out=%p", B, (long long)D, out);
    if (D % 4) return set_error(FF_ERR_UNSUPPORTED, "philox: D=%lld not a multiple of 4", (long long)D);
    if (D / 4 > 0xFFFFFFFFll) return set_error(FF_ERR_UNSUPPORTED, "philox: D=%lld too large", (long long)D);
    if (!aligned16(out)) return set_error(FF_ERR_INVALID_ARG, "philox: out must be 16-byte aligned");
    const int64_t nvec = D / 4, total = static_cast<int64_t>(B) * nvec;
    int64_t blocks = (total + kThreads - 1) / kThreads;
    const int64_t cap = 8 * static_cast<int64_t>(num_sms());
    if (blocks > cap) blocks = cap;
    ProfScope prof(stream, "philox_normal", 0.0, static_cast<double>(B) * D * 4.0);
    philox_normal_kernel<<<static_cast<unsigned>(blocks), kThreads, 0, stream>>>(B, nvec, philox_key(seed), rng_stream,
                                                                                 reinterpret_cast<float4*>(out));
    return check_launch("philox_normal_kernel");
}

}  // extern "C"

extern "C" int ff_sde_logprob_backward(int B, int64_t D, const float* x_t, const float* v, const float* x_next,
                                       const float* t, const float* t_next, const float* sigma, int reduce,
                                       const float* grad_logp, int ld, float* grad_v, cudaStream_t stream) {
    using namespace ff;
    if (B <= 0 || D <= 0) return set_error(FF_ERR_INVALID_ARG, "sde backward: B=%d D=%lld must be positive", B, (long long)D);
    if (D % 4) return set_error(FF_ERR_UNSUPPORTED, "sde backward: D=%lld not a multiple of 4", (long long)D);
    if (reduce != FF_LP_SUM && reduce != FF_LP_MEAN) return set_error(FF_ERR_INVALID_ARG, "sde backward: bad reduce %d", reduce);
    if (!x_t || !v || !x_next || !t || !t_next || !sigma || !grad_logp || !grad_v)
        return set_error(FF_ERR_INVALID_ARG, "sde backward: null pointer");
    if (!aligned16(x_t) || !aligned16(v) || !aligned16(x_next) || !aligned16(grad_v))
        return set_error(FF_ERR_INVALID_ARG, "sde backward: arrays must be 16-byte aligned");
    if (ld < 1) return set_error(FF_ERR_INVALID_ARG, "sde backward: ld=%d < 1", ld);
    if (B > 65535) return set_error(FF_ERR_UNSUPPORTED, "sde backward: B=%d > 65535", B);
    const int64_t nvec = D / 4;
    int64_t nb = (nvec + kThreads * 4 - 1) / (kThreads * 4);   // about four float4 per thread
    const int64_t cap = (4 * static_cast<int64_t>(num_sms()) + B - 1) / B;
    if (nb > cap) nb = cap;
    if (nb < 1) nb = 1;
    ProfScope prof(stream, "sde_logprob_backward", 0.0, static_cast<double>(B) * D * 16.0);
    sde_logprob_backward_kernel<<<dim3(static_cast<unsigned>(nb), B), kThreads, 0, stream>>>(
        D, static_cast<int>(nb), x_t, v, x_next, t, t_next, sigma, grad_logp, ld, reduce, grad_v);
    return check_launch("sde_logprob_backward_kernel");
}

extern "C" int ff_sde_schedule(int kind, int n_steps, double shift, double eta, double t_clamp, double* t_out,
                               double* sigma_out) {
    using namespace ff;
    if (n_steps <= 0 || !t_out || !sigma_out) return set_error(FF_ERR_INVALID_ARG, "schedule: bad arguments");
    if (!(shift > 0.0)) return set_error(FF_ERR_INVALID_ARG, "schedule: shift must be > 0");
    if (kind != FF_SCHED_FLOW_SDE && kind != FF_SCHED_DANCE_SDE && kind != FF_SCHED_ODE)
        return set_error(FF_ERR_INVALID_ARG, "schedule: bad kind %d", kind);
    if (kind == FF_SCHED_FLOW_SDE && !(t_clamp > 0.0 && t_clamp < 1.0))
        return set_error(FF_ERR_INVALID_ARG, "schedule: t_clamp must lie in (0, 1)");
    for (int k = 0; k <= n_steps; ++k) {
        const double t = 1.0 - static_cast<double>(k) / n_steps;
        t_out[k] = shift == 1.0 ? t : shift * t / (1.0 + (shift - 1.0) * t);
    }
    for (int k = 0; k < n_steps; ++k) {
        const double t = t_out[k] < t_clamp ? t_out[k] : t_clamp;
        if (kind == FF_SCHED_FLOW_SDE)
            sigma_out[k] = eta * sqrt(t / (1.0 - t));
        else if (kind == FF_SCHED_DANCE_SDE)
            sigma_out[k] = eta;
        else
            sigma_out[k] = 0.0;
    }
    return FF_OK;
}

extern "C" int ff_sde_schedule_window(int kind, int n_steps, double shift, double eta, double t_clamp,
                                      int window_start, int window_len, double* t_out, double* sigma_out) {
    using namespace ff;
    if (window_start < 0 || window_len < 0 || window_start + window_len > n_steps)
        return set_error(FF_ERR_INVALID_ARG, "schedule: window [%d, %d) outside the %d steps", window_start,
                         window_start + window_len, n_steps);
    const int rc = ff_sde_schedule(kind, n_steps, shift, eta, t_clamp, t_out, sigma_out);
    if (rc) return rc;
    for (int k = 0; k < n_steps; ++k)
        if (k < window_start || k >= window_start + window_len) sigma_out[k] = 0.0;
    return FF_OK;
}

// ---------------------------------------------------------------------------
// ff_sde_step_logprob_noalloc: the same step for callers that cannot hand the
// library any device memory of their own (see include/ff.h).  The tickets and
// the per-chunk partial sums live in a fixed array in the library's device
// image instead of a caller workspace.
// ---------------------------------------------------------------------------
#include <atomic>
#include <mutex>

namespace ff {
namespace {

constexpr int kNoAllocMaxSamples = 4096;      // ticket words, at the front of the array
constexpr int kNoAllocMaxPartials = 65536;    // fp32 partial sums after them

// Shared by every call on a device (272 KiB).  The ticket words start at
// zero (device globals are zero-initialised when the module loads) and every
// call leaves them at zero; the partial slots are rewritten before they are
// read, so nothing else has to be cleared.
static __device__ __align__(256) float g_sde_scratch[kNoAllocMaxSamples + kNoAllocMaxPartials];

constexpr int kNoAllocMaxDevices = 64;
std::atomic<float*> g_sde_scratch_addr[kNoAllocMaxDevices] = {};
std::mutex g_sde_scratch_mu;

// Device address of g_sde_scratch on the current device, looked up once per
// device with that device current (host code cannot use the symbol itself).
// The cache is keyed by device ordinal and holds the primary context's
// address: it is wrong for a caller that runs the library in another context
// on that device, and stale after cudaDeviceReset.
int sde_scratch_address(float** out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kNoAllocMaxDevices)
        return set_error(FF_ERR_CUDA, "sde (no-alloc): no usable current device");
    float* p = g_sde_scratch_addr[dev].load(std::memory_order_acquire);
    if (!p) {
        std::lock_guard<std::mutex> lk(g_sde_scratch_mu);
        p = g_sde_scratch_addr[dev].load(std::memory_order_relaxed);
        if (!p) {
            void* q = nullptr;
            const cudaError_t e = cudaGetSymbolAddress(&q, g_sde_scratch);
            if (e != cudaSuccess || !q)
                return set_error(FF_ERR_CUDA, "sde (no-alloc): cudaGetSymbolAddress failed: %s", cudaGetErrorString(e));
            p = static_cast<float*>(q);
            g_sde_scratch_addr[dev].store(p, std::memory_order_release);
        }
    }
    *out = p;
    return FF_OK;
}

}  // namespace
}  // namespace ff

extern "C" int ff_sde_step_logprob_noalloc(int B, int64_t D, const float* x_t, const float* v, const float* eps,
                                           float* x_next, const float* t, const float* t_next, const float* sigma,
                                           int mode, int reduce, float* logp, int ld, cudaStream_t stream) {
    using namespace ff;
    if (B <= 0 || D <= 0) return set_error(FF_ERR_INVALID_ARG, "sde (no-alloc): B=%d D=%lld must be positive", B, (long long)D);
    if (D % 4) return set_error(FF_ERR_UNSUPPORTED, "sde (no-alloc): D=%lld not a multiple of 4", (long long)D);
    // the scratch limits come first, so an oversized call is rejected
    // whatever its pointers are
    if (B > kNoAllocMaxSamples)
        return set_error(FF_ERR_UNSUPPORTED, "sde (no-alloc): B=%d exceeds the built-in scratch's %d samples; use "
                         "ff_sde_step_logprob with a workspace", B, kNoAllocMaxSamples);
    const int nc = nchunks(D);
    if (static_cast<int64_t>(B) * nc > kNoAllocMaxPartials)
        return set_error(FF_ERR_UNSUPPORTED,
                         "sde (no-alloc): B * min(ceil(D / %d), %d) = %lld partial sums exceed the built-in scratch "
                         "of %d; use ff_sde_step_logprob with a workspace",
                         kChunk, kMaxBlocksPerSample, (long long)B * nc, kNoAllocMaxPartials);
    if (mode != FF_SDE_SAMPLE && mode != FF_SDE_EVAL) return set_error(FF_ERR_INVALID_ARG, "sde (no-alloc): bad mode %d", mode);
    if (reduce != FF_LP_SUM && reduce != FF_LP_MEAN)
        return set_error(FF_ERR_INVALID_ARG, "sde (no-alloc): bad reduce %d", reduce);
    if (!x_t || !v || !x_next || !t || !t_next || !sigma || !logp || (mode == FF_SDE_SAMPLE && !eps))
        return set_error(FF_ERR_INVALID_ARG, "sde (no-alloc): null pointer");
    if (!aligned16(x_t) || !aligned16(v) || !aligned16(x_next) || (mode == FF_SDE_SAMPLE && !aligned16(eps)))
        return set_error(FF_ERR_INVALID_ARG, "sde (no-alloc): arrays must be 16-byte aligned");
    if (ld < 1) return set_error(FF_ERR_INVALID_ARG, "sde (no-alloc): ld=%d < 1", ld);
    float* scratch = nullptr;
    const int rc0 = sde_scratch_address(&scratch);
    if (rc0) return rc0;
    unsigned* ticket = reinterpret_cast<unsigned*>(scratch);
    float* partial = scratch + kNoAllocMaxSamples;
    return launch_sde_step(B, D, nc, x_t, v, eps, x_next, t, t_next, sigma, mode, reduce, logp, ld, ticket, partial,
                           PhiloxKey{0, 0}, 0u, stream);
}

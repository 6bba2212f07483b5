// grpo.cu -- group-relative advantage and the clipped-ratio policy loss of
// Flow-GRPO (paper Sec. 2.3 "advantage computation", Sec. 3.1).
//
// Advantage: G / 4 lanes per group (G a power of two in [4, 128]), else one
// warp per group.  Mean and population std are fp32 sums of the rewards
// shifted by a pivot (the group's first reward), then
// A = (r - mean) / (std + eps_A).  The tests bound the result against the
// fp64 oracle at 1e-5 relative to the group's spread.
//
// Loss: rho = exp(lp_new - lp_old) per (sample, step);
//   obj = min(rho A, clip(rho, 1 - lo, 1 + hi) A), loss = -sum(obj) / (B T),
//   grad_lp_new = -A rho / (B T) where the unclipped term is the minimum.
// One launch: every block writes one fp32 partial (the grid size depends only
// on B T), takes a ticket, and the block with the last ticket adds the
// partials in a fixed order, writes the loss and resets the ticket to zero.
// All fp32 (fp64 arithmetic is slow on this part): per-thread sums of a few
// terms, shuffles, then at most 1216 partials, about 1e-6 relative error.
#include "internal.h"
#include "ptx.cuh"

namespace ff {
namespace {

constexpr int kThreads = 256;
constexpr int kElemsPerBlock = kThreads * 16;
constexpr int kMaxLossBlocks = 1216;   // 8 blocks of 256 threads on each of 152 SMs
// Workspace: the ticket word at offset 0 (its own 16 bytes), then the fp32
// partials.
constexpr size_t kLossTicketBytes = 16;

// The group sums run on values shifted by a pivot (the group's first
// reward): mean = pivot + sum(r - pivot) / G.  A constant group then gets
// exactly zero advantages (an fp32 mean of G equal values need not equal
// them), and the shift removes most of the cancellation when the rewards
// share a large offset.
//
// G in {4, 8, 16, 32, 64, 128}: each lane owns 4 consecutive samples (one
// float4) and a group spans G / 4 lanes; the reductions shuffle within those
// lanes.  fp32 sums over at most 128 values (the tests bound them against
// fp64).
__global__ void __launch_bounds__(kThreads) group_advantage_vec_kernel(int64_t n4, int G, const float4* r, float eps,
                                                                       float4* adv) {
    const int64_t i = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x;
    const bool live = i < n4;
    const float4 x = live ? r[i] : make_float4(0.f, 0.f, 0.f, 0.f);
    const int lanes = G >> 2;
    const float pivot = __shfl_sync(0xffffffffu, x.x, (threadIdx.x & 31) & ~(lanes - 1));
    float s = ((x.x - pivot) + (x.y - pivot)) + ((x.z - pivot) + (x.w - pivot));
    for (int o = 1; o < lanes; o <<= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    const float mean = pivot + s / G;
    const float d0 = x.x - mean, d1 = x.y - mean, d2 = x.z - mean, d3 = x.w - mean;
    float q = (d0 * d0 + d1 * d1) + (d2 * d2 + d3 * d3);
    for (int o = 1; o < lanes; o <<= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
    const float inv = 1.0f / (sqrtf(q / G) + eps);
    if (live) adv[i] = make_float4(d0 * inv, d1 * inv, d2 * inv, d3 * inv);
}

// Any G: one warp per group, the group re-read from L1 for the second pass.
__global__ void __launch_bounds__(kThreads) group_advantage_kernel(int n_groups, int G, const float* r, float eps,
                                                                   float* adv) {
    const int warp = (blockIdx.x * kThreads + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (warp >= n_groups) return;
    const float* rg = r + static_cast<int64_t>(warp) * G;
    const float pivot = rg[0];
    float s = 0.f;
    for (int i = lane; i < G; i += 32) s += rg[i] - pivot;
#pragma unroll
    for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    const float mean = pivot + s / G;
    float q = 0.f;
    for (int i = lane; i < G; i += 32) {
        const float d = rg[i] - mean;
        q += d * d;
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
    const float denom = sqrtf(q / G) + eps;
    float* ag = adv + static_cast<int64_t>(warp) * G;
    // each lane rewrites only the elements it reads itself, after the
    // reductions above, so adv may alias r
    for (int i = lane; i < G; i += 32) ag[i] = (rg[i] - mean) / denom;
}

// Several rewards per sample, R[i, k] row-major [N, K]: one warp per group.
// WEIGHTED_SUM forms r_i = sum_k w_k R[i, k] on the fly and normalises it;
// PER_REWARD normalises every column within the group and accumulates
// w_k A[i, k] into adv (each lane rewrites only its own samples).
__global__ void __launch_bounds__(kThreads) group_advantage_multi_kernel(int n_groups, int G, int K, const float* R,
                                                                         const float* w, int mode, float eps,
                                                                         float* adv) {
    const int warp = (blockIdx.x * kThreads + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (warp >= n_groups) return;
    const float* Rg = R + static_cast<int64_t>(warp) * G * K;
    float* ag = adv + static_cast<int64_t>(warp) * G;
    auto warp_sum = [](float v) {
#pragma unroll
        for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        return v;
    };
    if (mode == FF_AGG_WEIGHTED_SUM) {
        auto r_of = [&](int i) {
            float r = 0.f;
            for (int k = 0; k < K; ++k) r = fmaf(w[k], Rg[static_cast<int64_t>(i) * K + k], r);
            return r;
        };
        const float pivot = r_of(0);
        float s = 0.f;
        for (int i = lane; i < G; i += 32) s += r_of(i) - pivot;
        const float mean = pivot + warp_sum(s) / G;
        float q = 0.f;
        for (int i = lane; i < G; i += 32) {
            const float d = r_of(i) - mean;
            q = fmaf(d, d, q);
        }
        const float denom = sqrtf(warp_sum(q) / G) + eps;
        for (int i = lane; i < G; i += 32) ag[i] = (r_of(i) - mean) / denom;
        return;
    }
    for (int k = 0; k < K; ++k) {
        const float pivot = Rg[k];
        float s = 0.f;
        for (int i = lane; i < G; i += 32) s += Rg[static_cast<int64_t>(i) * K + k] - pivot;
        const float mean = pivot + warp_sum(s) / G;
        float q = 0.f;
        for (int i = lane; i < G; i += 32) {
            const float d = Rg[static_cast<int64_t>(i) * K + k] - mean;
            q = fmaf(d, d, q);
        }
        const float c = w[k] / (sqrtf(warp_sum(q) / G) + eps);
        for (int i = lane; i < G; i += 32) {
            const float a = c * (Rg[static_cast<int64_t>(i) * K + k] - mean);
            ag[i] = k == 0 ? a : ag[i] + a;
        }
    }
}

// One fp32 partial per thread over float4 groups (sample index b = i / T in
// 32-bit arithmetic), fp64 only for the block and cross-block sums.
// WEIGHTED: GRPO-Guard's per-step weights step_w[k] scale the term of step
// k (objective and gradient).
// ticket: zero on entry; the last block to store its partial sets it back
// to zero.
template <bool WEIGHTED>
__global__ void __launch_bounds__(kThreads) grpo_loss_partial_kernel(int64_t n, int T, const float* lp_new,
                                                                     const float* lp_old, const float* adv,
                                                                     const float* step_w, float lo, float hi,
                                                                     float inv_n, float* grad, float* partial,
                                                                     unsigned* ticket, float* loss) {
    float s = 0.f;
    const int64_t n4 = n >> 2;
    const float4* a4 = reinterpret_cast<const float4*>(lp_new);
    const float4* b4 = reinterpret_cast<const float4*>(lp_old);
    const uint32_t Tu = static_cast<uint32_t>(T);
    auto term = [&](float ln, float lo_, uint32_t idx, float& g) {
        const uint32_t b = idx / Tu;
        const float a = adv[b];
        const float rho = __expf(ln - lo_);
        const float unclipped = rho * a;
        const float clipped = fminf(fmaxf(rho, 1.0f - lo), 1.0f + hi) * a;
        const bool take = unclipped <= clipped;
        const float w = WEIGHTED ? step_w[idx - b * Tu] : 1.0f;
        g = take ? -w * a * rho * inv_n : 0.0f;
        return w * (take ? unclipped : clipped);
    };
    for (int64_t v = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; v < n4;
         v += static_cast<int64_t>(gridDim.x) * kThreads) {
        const float4 x = __ldcs(a4 + v);
        const float4 y = __ldcs(b4 + v);
        const uint32_t i0 = static_cast<uint32_t>(v << 2);
        float4 g;
        s += term(x.x, y.x, i0, g.x);
        s += term(x.y, y.y, i0 + 1, g.y);
        s += term(x.z, y.z, i0 + 2, g.z);
        s += term(x.w, y.w, i0 + 3, g.w);
        if (grad) __stcs(reinterpret_cast<float4*>(grad) + v, g);
    }
    for (int64_t i = (n4 << 2) + static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * kThreads) {
        float g;
        s += term(lp_new[i], lp_old[i], static_cast<uint32_t>(i), g);
        if (grad) grad[i] = g;
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    __shared__ float redf[kThreads / 32];
    if ((threadIdx.x & 31) == 0) redf[threadIdx.x >> 5] = s;
    __syncthreads();
    __shared__ bool last;
    if (threadIdx.x == 0) {
        float t = 0.f;
        for (int w = 0; w < kThreads / 32; ++w) t += redf[w];
        partial[blockIdx.x] = t;
        last = ticket_add_acq_rel(ticket, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (!last) return;
    // every partial is stored (the last ticket acquired them): add them in
    // index order
    float acc = 0.f;
    for (int i = threadIdx.x; i < static_cast<int>(gridDim.x); i += kThreads) acc += __ldcg(partial + i);
#pragma unroll
    for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if ((threadIdx.x & 31) == 0) redf[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        float t = 0.f;
        for (int w = 0; w < kThreads / 32; ++w) t += redf[w];
        *ticket = 0u;
        *loss = -t * inv_n;
    }
}

int loss_blocks(int64_t n) {
    const int64_t b = (n + kElemsPerBlock - 1) / kElemsPerBlock;
    return static_cast<int>(b < kMaxLossBlocks ? b : kMaxLossBlocks);
}

}  // namespace
}  // namespace ff

extern "C" {

int ff_group_advantage(int n_groups, int G, const float* rewards, float eps_A, float* adv, cudaStream_t stream) {
    using namespace ff;
    if (n_groups <= 0 || G <= 0) return set_error(FF_ERR_INVALID_ARG, "advantage: n_groups=%d G=%d", n_groups, G);
    if (G > 4096) return set_error(FF_ERR_UNSUPPORTED, "advantage: G=%d > 4096", G);
    if (!rewards || !adv) return set_error(FF_ERR_INVALID_ARG, "advantage: null pointer");
    if (!(eps_A >= 0.0f)) return set_error(FF_ERR_INVALID_ARG, "advantage: eps_A must be >= 0");
    ProfScope prof(stream, "group_advantage", 0.0, 8.0 * n_groups * G);
    if (G >= 4 && G <= 128 && (G & (G - 1)) == 0 && aligned16(rewards) && aligned16(adv)) {
        const int64_t n4 = static_cast<int64_t>(n_groups) * G / 4;
        const int64_t grid = (n4 + kThreads - 1) / kThreads;
        if (grid > 0x7fffffff) return set_error(FF_ERR_UNSUPPORTED, "advantage: too many samples");
        group_advantage_vec_kernel<<<static_cast<unsigned>(grid), kThreads, 0, stream>>>(
            n4, G, reinterpret_cast<const float4*>(rewards), eps_A, reinterpret_cast<float4*>(adv));
        return check_launch("group_advantage_vec_kernel");
    }
    const int warps_per_block = kThreads / 32;
    const int grid = (n_groups + warps_per_block - 1) / warps_per_block;
    group_advantage_kernel<<<grid, kThreads, 0, stream>>>(n_groups, G, rewards, eps_A, adv);
    return check_launch("group_advantage_kernel");
}

int ff_grpo_loss_workspace_size(int B, int T, size_t* bytes) {
    if (!bytes) return ff::set_error(FF_ERR_INVALID_ARG, "bytes is null");
    if (B <= 0 || T <= 0) return ff::set_error(FF_ERR_INVALID_ARG, "B=%d T=%d must be positive", B, T);
    *bytes = ff::kLossTicketBytes + static_cast<size_t>(ff::loss_blocks(static_cast<int64_t>(B) * T)) * sizeof(float);
    return FF_OK;
}

}  // extern "C"

namespace ff {
namespace {

int grpo_loss_impl(int B, int T, const float* lp_new, const float* lp_old, const float* adv, const float* step_w,
                   float clip_lo, float clip_hi, float* loss, float* grad_lp_new, void* ws, size_t ws_bytes,
                   cudaStream_t stream) {
    if (B <= 0 || T <= 0) return set_error(FF_ERR_INVALID_ARG, "loss: B=%d T=%d must be positive", B, T);
    if (!lp_new || !lp_old || !adv || !loss) return set_error(FF_ERR_INVALID_ARG, "loss: null pointer");
    if (!aligned16(lp_new) || !aligned16(lp_old) || (grad_lp_new && !aligned16(grad_lp_new)))
        return set_error(FF_ERR_INVALID_ARG, "loss: lp_new, lp_old and grad_lp_new must be 16-byte aligned");
    if (static_cast<int64_t>(B) * T >= (int64_t(1) << 32))
        return set_error(FF_ERR_UNSUPPORTED, "loss: B * T must be below 2^32");
    if (!(clip_lo >= 0.0f && clip_lo < 1.0f && clip_hi >= 0.0f))
        return set_error(FF_ERR_INVALID_ARG, "loss: clip range must satisfy 0 <= lo < 1, hi >= 0");
    const int64_t n = static_cast<int64_t>(B) * T;
    const int nb = loss_blocks(n);
    const size_t need = kLossTicketBytes + static_cast<size_t>(nb) * sizeof(float);
    if (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 15))
        return set_error(FF_ERR_WORKSPACE, "loss: workspace %zu B < %zu B needed (or not 16-byte aligned)", ws_bytes,
                         need);
    unsigned* ticket = static_cast<unsigned*>(ws);
    float* partial = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) + kLossTicketBytes);
    const float inv_f = static_cast<float>(1.0 / static_cast<double>(n));
    ProfScope prof(stream, "grpo_loss", 0.0, static_cast<double>(n) * (grad_lp_new ? 12.0 : 8.0) + 4.0 * B);
    if (step_w)
        grpo_loss_partial_kernel<true><<<nb, kThreads, 0, stream>>>(n, T, lp_new, lp_old, adv, step_w, clip_lo,
                                                                    clip_hi, inv_f, grad_lp_new, partial, ticket,
                                                                    loss);
    else
        grpo_loss_partial_kernel<false><<<nb, kThreads, 0, stream>>>(n, T, lp_new, lp_old, adv, nullptr, clip_lo,
                                                                     clip_hi, inv_f, grad_lp_new, partial, ticket,
                                                                     loss);
    return check_launch("grpo_loss_kernel");
}

}  // namespace
}  // namespace ff

extern "C" {

int ff_grpo_loss(int B, int T, const float* lp_new, const float* lp_old, const float* adv, float clip_lo,
                 float clip_hi, float* loss, float* grad_lp_new, void* ws, size_t ws_bytes, cudaStream_t stream) {
    return ff::grpo_loss_impl(B, T, lp_new, lp_old, adv, nullptr, clip_lo, clip_hi, loss, grad_lp_new, ws, ws_bytes,
                              stream);
}

int ff_grpo_loss_weighted(int B, int T, const float* lp_new, const float* lp_old, const float* adv,
                          const float* step_w, float clip_lo, float clip_hi, float* loss, float* grad_lp_new,
                          void* ws, size_t ws_bytes, cudaStream_t stream) {
    if (!step_w) return ff::set_error(FF_ERR_INVALID_ARG, "loss: step_w is null (use ff_grpo_loss)");
    return ff::grpo_loss_impl(B, T, lp_new, lp_old, adv, step_w, clip_lo, clip_hi, loss, grad_lp_new, ws, ws_bytes,
                              stream);
}

int ff_group_advantage_multi(int n_groups, int G, int K, const float* rewards, const float* weights, int mode,
                             float eps_A, float* adv, cudaStream_t stream) {
    using namespace ff;
    if (n_groups <= 0 || G <= 0 || K <= 0)
        return set_error(FF_ERR_INVALID_ARG, "advantage (multi): n_groups=%d G=%d K=%d", n_groups, G, K);
    if (G > 4096 || K > 64) return set_error(FF_ERR_UNSUPPORTED, "advantage (multi): G=%d > 4096 or K=%d > 64", G, K);
    if (!rewards || !weights || !adv) return set_error(FF_ERR_INVALID_ARG, "advantage (multi): null pointer");
    if (mode != FF_AGG_WEIGHTED_SUM && mode != FF_AGG_PER_REWARD)
        return set_error(FF_ERR_INVALID_ARG, "advantage (multi): bad mode %d", mode);
    if (!(eps_A >= 0.0f)) return set_error(FF_ERR_INVALID_ARG, "advantage (multi): eps_A must be >= 0");
    ProfScope prof(stream, "group_advantage_multi", 0.0, 4.0 * n_groups * G * (K + 1));
    const int warps_per_block = kThreads / 32;
    const int grid = (n_groups + warps_per_block - 1) / warps_per_block;
    group_advantage_multi_kernel<<<grid, kThreads, 0, stream>>>(n_groups, G, K, rewards, weights, mode, eps_A, adv);
    return check_launch("group_advantage_multi_kernel");
}

}  // extern "C"

// rollout.cu -- trajectory sampling: S denoise steps of Eq. 1 with the DiT
// velocity (paper Sec. 3.1; the rollout that every GRPO-style trainer runs
// before it trains).  A host-side loop over the library's own entry points:
// per step, one velocity call and one fused SDE step + log-prob, all on the
// caller's stream with no synchronisation, so a caller may capture the whole
// rollout in a CUDA graph.
#include "internal.h"

namespace ff {
namespace {

constexpr size_t kAlign = 256;

size_t align_up(size_t n) { return (n + kAlign - 1) / kAlign * kAlign; }

// Per-sample copies of the shared step times: tb[k * B + b] = t[k],
// sb[k * B + b] = sigma[k] (the velocity and the SDE step take per-sample
// arrays).
__global__ void broadcast_steps_kernel(int S, int B, const float* t, const float* sigma, float* tb, float* sb) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < (S + 1) * B) tb[i] = t[i / B];
    if (i < S * B) sb[i] = sigma[i / B];
}

struct RolloutWs {
    size_t vel, v, tb, sb, sde, total;
};

int rollout_plan(const ff_dit* model, int B, int S, int64_t D, RolloutWs* p) {
    size_t vel = 0, sde = 0;
    FF_TRY(ff_dit_workspace_size(model, B, &vel));
    FF_TRY(ff_sde_workspace_size(B, D, &sde));
    p->vel = 0;
    p->v = align_up(vel);
    p->tb = p->v + align_up(static_cast<size_t>(B) * D * sizeof(float));
    p->sb = p->tb + align_up(static_cast<size_t>(S + 1) * B * sizeof(float));
    p->sde = p->sb + align_up(static_cast<size_t>(S) * B * sizeof(float));
    p->total = p->sde + align_up(sde);
    return FF_OK;
}

int64_t latent_elems(const ff_dit* model) {
    const ff_dit_config& c = model_config(model);
    return static_cast<int64_t>(c.grid_f) * c.grid_h * c.grid_w * c.patch_dim;
}

}  // namespace
}  // namespace ff

extern "C" {

int ff_rollout_workspace_size(const ff_dit* model, int B, int S, size_t* bytes) {
    using namespace ff;
    if (!model || !bytes) return set_error(FF_ERR_INVALID_ARG, "rollout: model/bytes is null");
    if (B <= 0 || S <= 0) return set_error(FF_ERR_INVALID_ARG, "rollout: B=%d S=%d must be positive", B, S);
    RolloutWs p;
    FF_TRY(rollout_plan(model, B, S, latent_elems(model), &p));
    *bytes = p.total;
    return FF_OK;
}

}  // extern "C"

namespace ff {
namespace {

// The rollout loop; step k's noise is eps[k] (eps set) or the counter-based
// noise of (seed, stream k) drawn inside the SDE kernel.
int rollout(const ff_dit* model, int B, int S, float* x, const void* txt, const float* t, const float* sigma,
            const float* eps, uint64_t seed, float* traj, float* logp, int reduce, void* ws, size_t ws_bytes,
            cudaStream_t stream) {
    if (!model) return set_error(FF_ERR_INVALID_ARG, "rollout: model is null");
    if (B <= 0 || S <= 0) return set_error(FF_ERR_INVALID_ARG, "rollout: B=%d S=%d must be positive", B, S);
    if (!x || !txt || !t || !sigma || !logp || !ws) return set_error(FF_ERR_INVALID_ARG, "rollout: null pointer");
    if (!aligned16(x) || (eps && !aligned16(eps)) || (traj && !aligned16(traj)) ||
        (reinterpret_cast<uintptr_t>(ws) % kAlign))
        return set_error(FF_ERR_INVALID_ARG, "rollout: misaligned pointer (arrays 16 B, workspace 256 B)");
    if (reduce != FF_LP_SUM && reduce != FF_LP_MEAN) return set_error(FF_ERR_INVALID_ARG, "rollout: bad reduce %d", reduce);
    const int64_t D = latent_elems(model);
    RolloutWs p;
    FF_TRY(rollout_plan(model, B, S, D, &p));
    if (ws_bytes < p.total) return set_error(FF_ERR_WORKSPACE, "rollout: workspace %zu B < %zu B needed", ws_bytes, p.total);
    uint8_t* base = static_cast<uint8_t*>(ws);
    float* v = reinterpret_cast<float*>(base + p.v);
    float* tb = reinterpret_cast<float*>(base + p.tb);
    float* sb = reinterpret_cast<float*>(base + p.sb);
    // the SDE step's ticket words must be zero before its first launch (each
    // launch leaves them zero); the rest of the workspace needs no clearing
    if (cudaMemsetAsync(base + p.sde, 0, p.total - p.sde, stream) != cudaSuccess)
        return set_error(FF_ERR_CUDA, "rollout: clearing the SDE step's scratch failed");
    const int n = (S + 1) * B;
    broadcast_steps_kernel<<<(n + 255) / 256, 256, 0, stream>>>(S, B, t, sigma, tb, sb);
    FF_TRY(check_launch("broadcast_steps_kernel"));
    const size_t xbytes = static_cast<size_t>(B) * D * sizeof(float);
    if (traj && cudaMemcpyAsync(traj, x, xbytes, cudaMemcpyDeviceToDevice, stream) != cudaSuccess)
        return set_error(FF_ERR_CUDA, "rollout: trajectory copy failed");
    for (int k = 0; k < S; ++k) {
        // with a trajectory, step k reads traj[k] and writes traj[k + 1];
        // without one, x is updated in place
        float* xk = traj ? traj + static_cast<int64_t>(k) * B * D : x;
        float* xn = traj ? traj + static_cast<int64_t>(k + 1) * B * D : x;
        FF_TRY(ff_dit_velocity(model, B, xk, txt, tb + k * B, v, base + p.vel, p.v - p.vel, stream));
        if (eps)
            FF_TRY(ff_sde_step_logprob(B, D, xk, v, eps + static_cast<int64_t>(k) * B * D, xn, tb + k * B,
                                       tb + (k + 1) * B, sb + k * B, FF_SDE_SAMPLE, reduce, logp + k, S, base + p.sde,
                                       p.total - p.sde, stream));
        else
            FF_TRY(ff_sde_step_logprob_philox(B, D, xk, v, xn, tb + k * B, tb + (k + 1) * B, sb + k * B, seed,
                                              static_cast<uint32_t>(k), reduce, logp + k, S, base + p.sde,
                                              p.total - p.sde, stream));
    }
    if (traj && cudaMemcpyAsync(x, traj + static_cast<int64_t>(S) * B * D, xbytes, cudaMemcpyDeviceToDevice,
                                stream) != cudaSuccess)
        return set_error(FF_ERR_CUDA, "rollout: final copy failed");
    return FF_OK;
}

}  // namespace
}  // namespace ff

extern "C" {

int ff_rollout(const ff_dit* model, int B, int S, float* x, const void* txt, const float* t, const float* sigma,
               const float* eps, float* traj, float* logp, int reduce, void* ws, size_t ws_bytes,
               cudaStream_t stream) {
    if (!eps) return ff::set_error(FF_ERR_INVALID_ARG, "rollout: null eps (ff_rollout_philox draws it)");
    return ff::rollout(model, B, S, x, txt, t, sigma, eps, 0, traj, logp, reduce, ws, ws_bytes, stream);
}

int ff_rollout_philox(const ff_dit* model, int B, int S, float* x, const void* txt, const float* t,
                      const float* sigma, uint64_t seed, float* traj, float* logp, int reduce, void* ws,
                      size_t ws_bytes, cudaStream_t stream) {
    return ff::rollout(model, B, S, x, txt, t, sigma, nullptr, seed, traj, logp, reduce, ws, ws_bytes, stream);
}

}  // extern "C"

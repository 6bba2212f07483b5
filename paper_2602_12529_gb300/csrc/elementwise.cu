// elementwise.cu -- the row-wise kernels of the DiT velocity:
//   * ln_modulate: LayerNorm (no affine, eps 1e-6) then x (1 + scale) + shift
//     with the sample's adaLN vectors (or an affine LayerNorm), fp32 in ->
//     bf16 GEMM operand out;
//   * qk_norm_rope: per-head RMSNorm of q and k (learned scale, eps 1e-6)
//     and the rotary embedding over (frame, row, col) slices of the head
//     dim, in place on the bf16 qkv buffer;
//   * timestep_embed: [cos | sin] of 1000 t times the sinusoid frequencies;
//   * f32_to_bf16: operand conversion of the fp32 latent tokens.
#include "internal.h"
#include "ptx.cuh"

namespace ff {
namespace {

constexpr float kLnEps = 1e-6f;
constexpr float kRmsEps = 1e-6f;

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// One CTA of 256 threads per row; thread t holds the float4s t, t + 256, ...
// of the row in registers (PER of them, H <= 1024 PER), so x is read once:
// the mean and the centred sum of squares come from the registers, reduced
// over the CTA through shared memory.
constexpr int kLnThreads = 256;

__device__ __forceinline__ float block_sum(float v, float* red, int lane, int w) {
    v = warp_sum(v);
    if (lane == 0) red[w] = v;
    __syncthreads();
    float t = 0.f;
#pragma unroll
    for (int i = 0; i < kLnThreads / 32; ++i) t += red[i];
    return t;
}

template <int PER>
__global__ void __launch_bounds__(kLnThreads, (PER <= 3 ? 8 : 1)) ln_modulate_kernel(LnModArgs a) {
    __shared__ float red[2][kLnThreads / 32];
    const int row = blockIdx.x;
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    int b, sh, sc;
    if (row < a.rows_txt) {
        b = row / a.n_txt;
        sh = a.shift_txt;
        sc = a.scale_txt;
    } else {
        b = (row - a.rows_txt) / a.n_img;
        sh = a.shift_img;
        sc = a.scale_img;
    }
    const float4* x = reinterpret_cast<const float4*>(a.x + static_cast<int64_t>(row) * a.ldx);
    const int nv = a.H >> 2;
    float4 r[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        const int k = t + kLnThreads * i;
        r[i] = k < nv ? __ldcs(x + k) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < PER; ++i) s += (r[i].x + r[i].y) + (r[i].z + r[i].w);
    const float mean = block_sum(s, red[0], lane, w) / a.H;
    float q = 0.f;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        if (t + kLnThreads * i < nv) {
            const float d0 = r[i].x - mean, d1 = r[i].y - mean, d2 = r[i].z - mean, d3 = r[i].w - mean;
            q += (d0 * d0 + d1 * d1) + (d2 * d2 + d3 * d3);
        }
    }
    const float rstd = rsqrtf(block_sum(q, red[1], lane, w) / a.H + kLnEps);
    uint2* out = reinterpret_cast<uint2*>(a.out + static_cast<int64_t>(row) * a.ldo);
    if (a.aff_w) {
        // affine LayerNorm: LN(x) w + b
        const uint2* w2 = reinterpret_cast<const uint2*>(a.aff_w);
        const uint2* b2 = reinterpret_cast<const uint2*>(a.aff_b);
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const int k = t + kLnThreads * i;
            if (k >= nv) break;
            const float4 v = r[i];
            const uint2 wu = w2[k], bu = b2[k];
            const float2 w0 = unpack_bf16x2(wu.x), w1 = unpack_bf16x2(wu.y);
            const float2 b0 = unpack_bf16x2(bu.x), b1 = unpack_bf16x2(bu.y);
            out[k] = make_uint2(pack_bf16x2((v.x - mean) * rstd * w0.x + b0.x, (v.y - mean) * rstd * w0.y + b0.y),
                                pack_bf16x2((v.z - mean) * rstd * w1.x + b1.x, (v.w - mean) * rstd * w1.y + b1.y));
        }
        return;
    }
    const float4* shift = reinterpret_cast<const float4*>(a.mods + static_cast<int64_t>(b) * a.ld_mods + sh);
    const float4* scale = reinterpret_cast<const float4*>(a.mods + static_cast<int64_t>(b) * a.ld_mods + sc);
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        const int k = t + kLnThreads * i;
        if (k >= nv) break;
        const float4 v = r[i];
        const float4 h = shift[k];
        const float4 c = scale[k];
        const float y0 = (v.x - mean) * rstd * (1.f + c.x) + h.x;
        const float y1 = (v.y - mean) * rstd * (1.f + c.y) + h.y;
        const float y2 = (v.z - mean) * rstd * (1.f + c.z) + h.z;
        const float y3 = (v.w - mean) * rstd * (1.f + c.w) + h.w;
        out[k] = make_uint2(pack_bf16x2(y0, y1), pack_bf16x2(y2, y3));
    }
}

// One warp per (row, head): lane owns E = d/32 consecutive elements (2 or 4),
// i.e. whole rotation pairs.
template <int E>
__global__ void __launch_bounds__(256) qk_norm_rope_kernel(QkNormRopeArgs a) {
    const int64_t gw = (static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (gw >= static_cast<int64_t>(a.rows) * a.heads) return;
    const int row = static_cast<int>(gw / a.heads);
    const int head = static_cast<int>(gw - static_cast<int64_t>(row) * a.heads);
    const bool img = row >= a.rows_txt;
    const int c0 = lane * E;
    const __nv_bfloat16* qs = img ? a.q_scale_img : a.q_scale_txt;
    const __nv_bfloat16* ks = img ? a.k_scale_img : a.k_scale_txt;

    // rotation of this lane's pairs (identity for text tokens at position 0)
    float cs[E / 2], sn[E / 2];
    if (img && a.rope) {
        const int n = (row - a.rows_txt) % a.n_img;
        const int hw = a.grid_h * a.grid_w;
        const float pos[3] = {static_cast<float>(n / hw), static_cast<float>((n / a.grid_w) % a.grid_h),
                              static_cast<float>(n % a.grid_w)};
        const float log2_theta = log2f(a.theta);
#pragma unroll
        for (int p = 0; p < E / 2; ++p) {
            const int pair = c0 / 2 + p;
            int axis, j, width;
            if (pair < a.axes0 / 2) {
                axis = 0; j = pair; width = a.axes0;
            } else if (pair < (a.axes0 + a.axes1) / 2) {
                axis = 1; j = pair - a.axes0 / 2; width = a.axes1;
            } else {
                axis = 2; j = pair - (a.axes0 + a.axes1) / 2; width = a.axes2;
            }
            const float freq = exp2f(-(2.0f * j / width) * log2_theta);
            sincosf(pos[axis] * freq, &sn[p], &cs[p]);
        }
    } else {
#pragma unroll
        for (int p = 0; p < E / 2; ++p) { cs[p] = 1.f; sn[p] = 0.f; }
    }

#pragma unroll
    for (int which = 0; which < 2; ++which) {
        if (a.col[which] < 0) continue;
        __nv_bfloat16* ptr = a.qkv + static_cast<int64_t>(row) * a.ld + a.col[which] + head * a.head_dim + c0;
        const __nv_bfloat16* sc = (which == 0 ? qs : ks) + c0;
        float v[E];
        if (E == 4) {
            const uint2 u = *reinterpret_cast<const uint2*>(ptr);
            const float2 f0 = unpack_bf16x2(u.x), f1 = unpack_bf16x2(u.y);
            v[0] = f0.x; v[1] = f0.y; v[2 % E] = f1.x; v[3 % E] = f1.y;
        } else {
            const float2 f0 = unpack_bf16x2(*reinterpret_cast<const uint32_t*>(ptr));
            v[0] = f0.x; v[1 % E] = f0.y;
        }
        float ss = 0.f;
#pragma unroll
        for (int i = 0; i < E; ++i) ss += v[i] * v[i];
        const float r = rsqrtf(warp_sum(ss) / a.head_dim + kRmsEps);
#pragma unroll
        for (int i = 0; i < E; ++i) v[i] = v[i] * r * __bfloat162float(sc[i]);
        float o[E];
#pragma unroll
        for (int p = 0; p < E / 2; ++p) {
            o[2 * p] = v[2 * p] * cs[p] - v[2 * p + 1] * sn[p];
            o[2 * p + 1] = v[2 * p] * sn[p] + v[2 * p + 1] * cs[p];
        }
        if (E == 4) {
            *reinterpret_cast<uint2*>(ptr) = make_uint2(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2 % E], o[3 % E]));
        } else {
            *reinterpret_cast<uint32_t*>(ptr) = pack_bf16x2(o[0], o[1 % E]);
        }
    }
}

__global__ void wan_modulation_kernel(const float* e, const float* e0, const __nv_bfloat16* bias0, int64_t stride,
                                      int L, const __nv_bfloat16* fbias, int H, float* mods, int64_t ld_mods) {
    const int b = blockIdx.y;
    const int64_t n = static_cast<int64_t>(L) * 6 * H + 2 * H;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        float v;
        if (i < static_cast<int64_t>(L) * 6 * H) {
            const int l = static_cast<int>(i / (6 * H));
            const int j = static_cast<int>(i - static_cast<int64_t>(l) * 6 * H);
            v = e0[static_cast<int64_t>(b) * 6 * H + j] + __bfloat162float(bias0[l * stride + j]);
        } else {
            const int j = static_cast<int>(i - static_cast<int64_t>(L) * 6 * H);
            v = e[static_cast<int64_t>(b) * H + (j % H)] + __bfloat162float(fbias[j]);
        }
        mods[static_cast<int64_t>(b) * ld_mods + i] = v;
    }
}

__global__ void rope_table_kernel(float2* table, int grid_f, int grid_h, int grid_w, int a0, int a1, int a2,
                                  float theta, int n) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const int h0 = a0 / 2, h1 = a1 / 2, h2 = a2 / 2;
    int pos, j, width;
    if (i < grid_f * h0) {
        pos = i / h0; j = i % h0; width = a0;
    } else if (i < grid_f * h0 + grid_h * h1) {
        const int k = i - grid_f * h0;
        pos = k / h1; j = k % h1; width = a1;
    } else {
        const int k = i - grid_f * h0 - grid_h * h1;
        pos = k / h2; j = k % h2; width = a2;
    }
    // fp32 angle (relative error ~1e-7, i.e. < 1e-5 rad at the largest
    // positions here -- far below the bf16 rounding of q and k)
    const float ang = static_cast<float>(pos) * exp2f(-(2.0f * j / width) * log2f(theta));
    float sn, cs;
    sincosf(ang, &sn, &cs);
    table[i] = make_float2(cs, sn);
}

__global__ void timestep_embed_kernel(const float* t, int B, int dim, __nv_bfloat16* out) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= B * dim) return;
    const int b = i / dim;
    const int j = i - b * dim;
    const int half = dim / 2;
    const int f = j < half ? j : j - half;
    // fp32 throughout (fp64 arithmetic is slow on this part): the argument
    // (at most 1000) is off by about 1e-4 rad, far below the bf16 rounding of
    // the result
    const float freq = expf(-9.21034037f * static_cast<float>(f) / static_cast<float>(half));   // ln(1e4)
    const float arg = 1000.0f * t[b] * freq;
    float sn, cs;
    sincosf(arg, &sn, &cs);
    out[i] = __float2bfloat16_rn(j < half ? cs : sn);
}

__global__ void f32_to_bf16_kernel(const float4* in, uint2* out, int64_t n4) {
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const float4 v = __ldcs(in + i);
        out[i] = make_uint2(pack_bf16x2(v.x, v.y), pack_bf16x2(v.z, v.w));
    }
}

}  // namespace

int ln_modulate(const LnModArgs& a, cudaStream_t stream) {
    if (a.rows <= 0) return FF_OK;
    if (a.H % 128 || a.ldx % 4 || a.ldo % 4 || a.ld_mods % 4 || (a.shift_txt | a.scale_txt | a.shift_img | a.scale_img) % 4)
        return set_error(FF_ERR_UNSUPPORTED, "ln_modulate: H=%d must be a multiple of 128", a.H);
    const int per = (a.H / 4 + kLnThreads - 1) / kLnThreads;   // float4s per thread
    ProfScope prof(stream, "ln_modulate", 0.0, static_cast<double>(a.rows) * a.H * 6.0);
    switch (per) {
        case 1: ln_modulate_kernel<1><<<a.rows, kLnThreads, 0, stream>>>(a); break;
        case 2: ln_modulate_kernel<2><<<a.rows, kLnThreads, 0, stream>>>(a); break;
        case 3: ln_modulate_kernel<3><<<a.rows, kLnThreads, 0, stream>>>(a); break;
        case 4: ln_modulate_kernel<4><<<a.rows, kLnThreads, 0, stream>>>(a); break;
        case 5: ln_modulate_kernel<5><<<a.rows, kLnThreads, 0, stream>>>(a); break;
        case 6: ln_modulate_kernel<6><<<a.rows, kLnThreads, 0, stream>>>(a); break;
        case 7: ln_modulate_kernel<7><<<a.rows, kLnThreads, 0, stream>>>(a); break;
        case 8: ln_modulate_kernel<8><<<a.rows, kLnThreads, 0, stream>>>(a); break;
        default: return set_error(FF_ERR_UNSUPPORTED, "ln_modulate: H=%d above 8192", a.H);
    }
    return check_launch("ln_modulate_kernel");
}

int qk_norm_rope(const QkNormRopeArgs& a, cudaStream_t stream) {
    if (a.rows <= 0) return FF_OK;
    const int64_t warps = static_cast<int64_t>(a.rows) * a.heads;
    const int64_t grid = (warps + 7) / 8;
    if (grid > 0x7fffffff) return set_error(FF_ERR_UNSUPPORTED, "qk_norm_rope: too many rows");
    ProfScope prof(stream, "qk_norm_rope", 0.0, static_cast<double>(a.rows) * a.heads * a.head_dim * 8.0);
    if (a.head_dim == 128)
        qk_norm_rope_kernel<4><<<static_cast<unsigned>(grid), 256, 0, stream>>>(a);
    else if (a.head_dim == 64)
        qk_norm_rope_kernel<2><<<static_cast<unsigned>(grid), 256, 0, stream>>>(a);
    else
        return set_error(FF_ERR_UNSUPPORTED, "qk_norm_rope: head_dim %d", a.head_dim);
    return check_launch("qk_norm_rope_kernel");
}

int timestep_embed(const float* t, int B, int dim, __nv_bfloat16* out, cudaStream_t stream) {
    const int n = B * dim;
    ProfScope prof(stream, "timestep_embed", 0.0, 4.0 * B + 2.0 * n);
    timestep_embed_kernel<<<(n + 255) / 256, 256, 0, stream>>>(t, B, dim, out);
    return check_launch("timestep_embed_kernel");
}

int f32_to_bf16(const float* in, __nv_bfloat16* out, int64_t n, cudaStream_t stream) {
    if (n % 4) return set_error(FF_ERR_UNSUPPORTED, "f32_to_bf16: n %% 4 != 0");
    const int64_t n4 = n / 4;
    int64_t grid = (n4 + 255) / 256;
    if (grid > 4 * num_sms() * 8) grid = 4 * num_sms() * 8;
    ProfScope prof(stream, "f32_to_bf16", 0.0, 6.0 * n);
    f32_to_bf16_kernel<<<static_cast<unsigned>(grid), 256, 0, stream>>>(reinterpret_cast<const float4*>(in),
                                                                        reinterpret_cast<uint2*>(out), n4);
    return check_launch("f32_to_bf16_kernel");
}

int wan_modulation(const float* e, const float* e0, const __nv_bfloat16* bias0, int64_t stride, int L,
                   const __nv_bfloat16* fbias, int B, int H, float* mods, int64_t ld_mods, cudaStream_t stream) {
    const dim3 grid(64, B);
    ProfScope prof(stream, "wan_modulation", 0.0, static_cast<double>(B) * (L * 6.0 * H + 2.0 * H) * 10.0);
    wan_modulation_kernel<<<grid, 256, 0, stream>>>(e, e0, bias0, stride, L, fbias, H, mods, ld_mods);
    return check_launch("wan_modulation_kernel");
}

int rope_table_size(int grid_f, int grid_h, int grid_w, int a0, int a1, int a2) {
    return grid_f * (a0 / 2) + grid_h * (a1 / 2) + grid_w * (a2 / 2);
}

int rope_table(float2* table, int grid_f, int grid_h, int grid_w, int a0, int a1, int a2, float theta,
               cudaStream_t stream) {
    const int n = rope_table_size(grid_f, grid_h, grid_w, a0, a1, a2);
    if (n <= 0) return FF_OK;
    ProfScope prof(stream, "rope_table", 0.0, 8.0 * n);
    rope_table_kernel<<<(n + 255) / 256, 256, 0, stream>>>(table, grid_f, grid_h, grid_w, a0, a1, a2, theta, n);
    return check_launch("rope_table_kernel");
}

}  // namespace ff

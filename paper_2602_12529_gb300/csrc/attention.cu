// attention.cu -- joint (text + image) non-causal attention,
//   O = softmax(Q K^T / sqrt(d)) V   per (sample, head),
// over the concatenated token sequence [segment 0; segment 1] of each sample
// (MMDiT joint attention: text tokens then image tokens).  Q, K and V are
// read straight out of the bf16 QKV GEMM outputs (row = token, q at column
// h*d, k at H + h*d, v at 2H + h*d); segments may live in different buffers.
//
// Flash-style single pass: a CTA owns 128 query rows of one (sample, head);
// 8 warps x 16 rows; K/V tiles of 64 tokens are double-buffered in shared
// memory with cp.async (16-byte chunks, XOR-swizzled by row so ldmatrix is
// conflict-free); scores and P.V run on bf16 mma.sync with fp32 accumulation;
// the running max / sum softmax keeps everything in registers (base-2
// exponentials with log2(e) folded into the scale).
#include "internal.h"
#include "ptx.cuh"

namespace ff {
namespace {

constexpr int kBM = 128;
constexpr int kBN = 64;
constexpr int kThreads = 256;

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(valid ? 16 : 0)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// byte offset of 16-byte chunk c of row r in a [rows, HD] bf16 tile
template <int HD>
__device__ __forceinline__ uint32_t swz(int r, int c) {
    return static_cast<uint32_t>(r * HD * 2 + ((c ^ (r & 7)) << 4));
}

struct SegPtr {
    const __nv_bfloat16* base0;
    const __nv_bfloat16* base1;
    int64_t ld0, ld1;
    int n0;
    __device__ __forceinline__ const __nv_bfloat16* row(int i) const {
        return i < n0 ? base0 + static_cast<int64_t>(i) * ld0 : base1 + static_cast<int64_t>(i - n0) * ld1;
    }
};

template <int HD>
__global__ void __launch_bounds__(kThreads, 1)
flash_attn_kernel(AttnSegment s0, AttnSegment s1, int H, float scale_log2) {
    constexpr int CH = HD / 8;   // 16-byte chunks per row
    extern __shared__ __align__(128) uint8_t smem[];
    const uint32_t sQ = smem_u32(smem);
    const uint32_t sK = sQ + kBM * HD * 2;
    const uint32_t sV = sK + 2 * kBN * HD * 2;

    const int b = blockIdx.z;
    const int h = blockIdx.y;
    const int q0 = blockIdx.x * kBM;
    const int N = s0.n + s1.n;
    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;

    SegPtr in;
    in.base0 = s0.qkv + static_cast<int64_t>(b) * s0.n * s0.ld;
    in.base1 = s1.qkv + static_cast<int64_t>(b) * s1.n * s1.ld;
    in.ld0 = s0.ld;
    in.ld1 = s1.ld;
    in.n0 = s0.n;

    const int col_q = h * HD, col_k = H + h * HD, col_v = 2 * H + h * HD;

    // ---- Q tile
    for (int idx = tid; idx < kBM * CH; idx += kThreads) {
        const int r = idx / CH, c = idx % CH;
        const int tok = q0 + r;
        const bool ok = tok < N;
        const __nv_bfloat16* src = ok ? in.row(tok) + col_q + c * 8 : s0.qkv;
        cp_async16(sQ + swz<HD>(r, c), ok ? src : (const void*)in.base1, ok);
    }
    auto load_kv = [&](int tile, int stage) {
        const int kv0 = tile * kBN;
        const uint32_t dk = sK + stage * kBN * HD * 2;
        const uint32_t dv = sV + stage * kBN * HD * 2;
        for (int idx = tid; idx < kBN * CH; idx += kThreads) {
            const int r = idx / CH, c = idx % CH;
            const int tok = kv0 + r;
            const bool ok = tok < N;
            const __nv_bfloat16* row = ok ? in.row(tok) : in.base1;
            cp_async16(dk + swz<HD>(r, c), ok ? (const void*)(row + col_k + c * 8) : (const void*)row, ok);
            cp_async16(dv + swz<HD>(r, c), ok ? (const void*)(row + col_v + c * 8) : (const void*)row, ok);
        }
    };
    load_kv(0, 0);
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();

    // ---- Q fragments (16 rows per warp, HD/16 k-steps)
    uint32_t qf[HD / 16][4];
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
        const int r = warp * 16 + (lane & 15);
        const int c = kk * 2 + (lane >> 4);
        ldsm_x4(sQ + swz<HD>(r, c), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
    }

    float o[HD / 8][4];
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
    float m_i[2] = {-INFINITY, -INFINITY};
    float l_i[2] = {0.f, 0.f};

    const int ntiles = (N + kBN - 1) / kBN;
    for (int j = 0; j < ntiles; ++j) {
        if (j + 1 < ntiles) {
            load_kv(j + 1, (j + 1) & 1);
            cp_async_commit();
            cp_async_wait<1>();
        } else {
            cp_async_wait<0>();
        }
        __syncthreads();
        const uint32_t tk = sK + (j & 1) * kBN * HD * 2;
        const uint32_t tv = sV + (j & 1) * kBN * HD * 2;

        // S = Q K^T (16 x 64 per warp)
        float s[kBN / 8][4];
#pragma unroll
        for (int i = 0; i < kBN / 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
            for (int p = 0; p < kBN / 16; ++p) {
                const int mat = lane >> 3;
                const int r = 16 * p + ((mat >> 1) << 3) + (lane & 7);
                const int c = 2 * kk + (mat & 1);
                uint32_t b0, b1, b2, b3;
                ldsm_x4(tk + swz<HD>(r, c), b0, b1, b2, b3);
                mma_bf16(s[2 * p], qf[kk], b0, b1);
                mma_bf16(s[2 * p + 1], qf[kk], b2, b3);
            }
        }
        // scale, mask, running max
        const int kv0 = j * kBN;
        float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
        for (int nf = 0; nf < kBN / 8; ++nf) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int col = kv0 + nf * 8 + 2 * (lane & 3) + (e & 1);
                const float v = col < N ? s[nf][e] * scale_log2 : -INFINITY;
                s[nf][e] = v;
                mx[e >> 1] = fmaxf(mx[e >> 1], v);
            }
        }
        float alpha[2];
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
            mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
            const float m_new = fmaxf(m_i[r], mx[r]);
            alpha[r] = exp2f(m_i[r] - m_new);
            m_i[r] = m_new;
            l_i[r] *= alpha[r];
        }
        // P = exp2(S - m), packed to bf16 A fragments
        uint32_t pf[kBN / 16][4];
#pragma unroll
        for (int nf = 0; nf < kBN / 8; ++nf) {
            const float p0 = exp2f(s[nf][0] - m_i[0]);
            const float p1 = exp2f(s[nf][1] - m_i[0]);
            const float p2 = exp2f(s[nf][2] - m_i[1]);
            const float p3 = exp2f(s[nf][3] - m_i[1]);
            l_i[0] += p0 + p1;
            l_i[1] += p2 + p3;
            pf[nf >> 1][(nf & 1) * 2 + 0] = pack_bf16x2(p0, p1);
            pf[nf >> 1][(nf & 1) * 2 + 1] = pack_bf16x2(p2, p3);
        }
#pragma unroll
        for (int i = 0; i < HD / 8; ++i) {
            o[i][0] *= alpha[0];
            o[i][1] *= alpha[0];
            o[i][2] *= alpha[1];
            o[i][3] *= alpha[1];
        }
        // O += P V
#pragma unroll
        for (int kk = 0; kk < kBN / 16; ++kk) {
#pragma unroll
            for (int pd = 0; pd < HD / 16; ++pd) {
                const int mat = lane >> 3;
                const int r = 16 * kk + ((mat & 1) << 3) + (lane & 7);
                const int c = 2 * pd + (mat >> 1);
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(tv + swz<HD>(r, c), b0, b1, b2, b3);
                mma_bf16(o[2 * pd], pf[kk], b0, b1);
                mma_bf16(o[2 * pd + 1], pf[kk], b2, b3);
            }
        }
        __syncthreads();
    }

    // ---- normalise and store
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        l_i[r] += __shfl_xor_sync(0xffffffffu, l_i[r], 1);
        l_i[r] += __shfl_xor_sync(0xffffffffu, l_i[r], 2);
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        const int tok = q0 + warp * 16 + (lane >> 2) + r * 8;
        if (tok >= N) continue;
        const float inv = 1.f / l_i[r];
        __nv_bfloat16* dst = tok < s0.n
                                 ? s0.out + (static_cast<int64_t>(b) * s0.n + tok) * s0.ldo + h * HD
                                 : s1.out + (static_cast<int64_t>(b) * s1.n + tok - s0.n) * s1.ldo + h * HD;
#pragma unroll
        for (int nd = 0; nd < HD / 8; ++nd) {
            const int c = nd * 8 + 2 * (lane & 3);
            *reinterpret_cast<uint32_t*>(dst + c) = pack_bf16x2(o[nd][2 * r] * inv, o[nd][2 * r + 1] * inv);
        }
    }
}

template <int HD>
int launch_attn(const AttnSegment& s0, const AttnSegment& s1, int B, int heads, int H, cudaStream_t stream) {
    const int smem = (kBM + 4 * kBN) * HD * 2;
    if (cudaFuncSetAttribute(flash_attn_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
        return set_error(FF_ERR_CUDA, "attention: cannot set shared memory size");
    const int N = s0.n + s1.n;
    const dim3 grid((N + kBM - 1) / kBM, heads, B);
    const float scale_log2 = static_cast<float>(1.4426950408889634 / sqrt(static_cast<double>(HD)));
    const double nn = static_cast<double>(N) * N;
    ProfScope prof(stream, "attention", 4.0 * B * heads * nn * HD, 8.0 * B * static_cast<double>(N) * H);
    flash_attn_kernel<HD><<<grid, kThreads, smem, stream>>>(s0, s1, H, scale_log2);
    return check_launch("flash_attn_kernel");
}

}  // namespace

int attention(const AttnSegment& s0, const AttnSegment& s1, int B, int heads, int head_dim, int H,
              cudaStream_t stream) {
    if (B <= 0 || heads <= 0 || s0.n < 0 || s1.n < 0 || s0.n + s1.n <= 0)
        return set_error(FF_ERR_INVALID_ARG, "attention: bad shape");
    if (B > 65535 || heads > 65535) return set_error(FF_ERR_UNSUPPORTED, "attention: grid too large");
    if ((s0.n && (!s0.qkv || !s0.out)) || (s1.n && (!s1.qkv || !s1.out)) || !s1.qkv)
        return set_error(FF_ERR_INVALID_ARG, "attention: null segment");
    if (s0.ld % 8 || s1.ld % 8 || s0.ldo % 8 || s1.ldo % 8)
        return set_error(FF_ERR_INVALID_ARG, "attention: leading dimensions must be multiples of 8");
    if (head_dim == 128) return launch_attn<128>(s0, s1, B, heads, H, stream);
    if (head_dim == 64) return launch_attn<64>(s0, s1, B, heads, H, stream);
    return set_error(FF_ERR_UNSUPPORTED, "attention: head_dim %d", head_dim);
}

}  // namespace ff

// attention.cu -- joint (text + image) non-causal attention on tcgen05,
//   O = softmax(Q K^T / sqrt(d)) V   per (sample, head),
// over the concatenated token sequence [segment 0; segment 1] of each sample
// (MMDiT joint attention: text tokens then image tokens).  Q, K and V are
// read straight out of the bf16 QKV GEMM outputs (row = token, q at column
// h*d, k at H + h*d, v at 2H + h*d) by TMA; the segments may live in
// different buffers.
//
// One CTA = 128 query rows of one segment of one (sample, head); two CTAs
// share an SM.  Warp roles (6 warps):
//   warp 0      TMA producer: the Q tile once, then 64-token K/V tiles into a
//               2-deep ring (K/V tiles never straddle the segment boundary;
//               rows past the segment end are masked).
//   warp 1      TMEM allocator; lane 0 issues the MMAs:
//                 S_j = Q K_j^T   (M 128, N 64, K d)  into TMEM buffer j % 2
//                 O  += P_j V_j   (M 128, N d,  K 64) into the TMEM O tile,
//               issuing S_{j+1} before O += P_j V_j so the tensor core works
//               while the softmax warps process S_j.
//   warps 2..5  softmax: thread = query row = TMEM lane.  Reads S_j,
//               updates the running max / sum in base 2 (log2 e folded into
//               the scale), writes P_j = exp2(S - m) as bf16 into a
//               128-byte-swizzled shared tile (the A operand of P V), and
//               rescales the O rows in TMEM only when the running max grows
//               by more than 8 (2^8 headroom in fp32/bf16), which makes
//               corrections rare.  Finally O / l goes out as bf16.
// Every wait is bounded; on a timeout the kernel records the status word,
// drains its tensor-core work, frees TMEM and returns.
#include "internal.h"
#include "ptx.cuh"

namespace ff {
namespace {

constexpr int kBM = 128;         // query rows per CTA
constexpr int kBN = 64;          // tokens per K/V tile
constexpr int kStages = 2;
constexpr int kThreads = 192;
constexpr float kRescaleThreshold = 8.0f;   // log2 units

template <int HD>
struct ACfg {
    static constexpr int kQBytes = kBM * HD * 2;
    static constexpr int kKBytes = kBN * HD * 2;
    static constexpr int kStageBytes = 2 * kKBytes;     // K + V
    static constexpr int kPBytes = kBM * kBN * 2;
    static constexpr int kSmemBytes = kQBytes + kStages * kStageBytes + kPBytes + 256;
    static constexpr int kTmemCols = 256;               // S0 | S1 | O
    static constexpr int kColS0 = 0, kColS1 = kBN, kColO = 2 * kBN;
};

struct AttnParams {
    int n[2];            // tokens per sample in each segment
    int qtiles0;         // query tiles of segment 0 (then segment 1's follow)
    int H;
    float scale_log2;
    __nv_bfloat16* out[2];
    int64_t ldo[2];
};

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ void tmem_st_x32(uint32_t taddr, const uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
        "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
        "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]),
        "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]),
        "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// B operand stored MN-major with 128-byte swizzle (V: rows = K = tokens,
// 64 contiguous d per 128-byte row): leading byte offset = distance between
// 64-wide d blocks, stride byte offset = distance between 8-token groups.
__device__ __forceinline__ uint64_t smem_desc_mn_sw128(uint32_t saddr, uint32_t lbo_bytes) {
    uint64_t d = 0;
    d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
    d |= static_cast<uint64_t>((lbo_bytes >> 4) & 0x3FFFu) << 16;
    d |= static_cast<uint64_t>(1024 >> 4) << 32;
    d |= static_cast<uint64_t>(1) << 46;
    d |= static_cast<uint64_t>(2) << 61;
    return d;
}

template <int HD>
__global__ void __launch_bounds__(kThreads, 2)
attn_tcgen05_kernel(const __grid_constant__ CUtensorMap tm_q0, const __grid_constant__ CUtensorMap tm_q1,
                    const __grid_constant__ CUtensorMap tm_kv0, const __grid_constant__ CUtensorMap tm_kv1,
                    const AttnParams p, int* status) {
    using C = ACfg<HD>;
    extern __shared__ __align__(1024) uint8_t smem[];
    uint8_t* sQ = smem;
    uint8_t* sKV = smem + C::kQBytes;
    uint8_t* sP = sKV + kStages * C::kStageBytes;
    uint64_t* bars = reinterpret_cast<uint64_t*>(sP + C::kPBytes);
    uint64_t* q_full = bars;                 // [1]
    uint64_t* kv_full = bars + 1;            // [kStages]
    uint64_t* kv_empty = kv_full + kStages;  // [kStages]
    uint64_t* s_full = kv_empty + kStages;   // [2]
    uint64_t* s_free = s_full + 2;           // [2]
    uint64_t* p_full = s_free + 2;           // [1]
    uint64_t* o_done = p_full + 1;           // [1]
    uint64_t* drain = o_done + 1;            // [1]
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int b = blockIdx.z;
    const int h = blockIdx.y;
    const int seg = blockIdx.x < p.qtiles0 ? 0 : 1;
    const int q0 = (blockIdx.x - (seg ? p.qtiles0 : 0)) * kBM;   // first query row within the segment
    const int nt0 = (p.n[0] + kBN - 1) / kBN;
    const int ntiles = nt0 + (p.n[1] + kBN - 1) / kBN;

    if (threadIdx.x == 0) {
        if (smem_u32(smem) & 1023u) {   // the swizzled tiles need 1024-byte alignment
            report_status(status, kStatusBadArgument);
            *abort_flag = 1;
        } else {
            *abort_flag = 0;
        }
        mbar_init(q_full, 1);
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&kv_full[s], 1);
            mbar_init(&kv_empty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&s_full[s], 1);
            mbar_init(&s_free[s], 4);
        }
        mbar_init(p_full, 4);
        mbar_init(o_done, 1);
        mbar_init(drain, 1);
        fence_mbar_init();
        prefetch_tmap(seg ? &tm_q1 : &tm_q0);
        prefetch_tmap(&tm_kv0);
        prefetch_tmap(&tm_kv1);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, C::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const bool aborted_at_start = *abort_flag;

    auto fail = [&]() {
        report_status(status, kStatusWaitTimeout);
        *abort_flag = 1;
    };

    if (aborted_at_start) {
        // nothing issued
    } else if (warp == 0 && lane == 0) {
        // ------------------------------------------------------------ producer
        const CUtensorMap* tq = seg ? &tm_q1 : &tm_q0;
        mbar_arrive_expect_tx(q_full, C::kQBytes);
        for (int c = 0; c < HD / 64; ++c)
            tma_load_2d(sQ + c * (kBM * 128), tq, q_full, h * HD + c * 64, b * p.n[seg] + q0);
        for (int j = 0; j < ntiles && !*abort_flag; ++j) {
            const int s = j % kStages;
            const uint32_t ph = (j / kStages) & 1;
            if (!mbar_wait(&kv_empty[s], ph ^ 1)) { fail(); break; }
            const int ks = j < nt0 ? 0 : 1;
            const int row = b * p.n[ks] + (j - (ks ? nt0 : 0)) * kBN;
            const CUtensorMap* tkv = ks ? &tm_kv1 : &tm_kv0;
            uint8_t* dk = sKV + s * C::kStageBytes;
            uint8_t* dv = dk + C::kKBytes;
            mbar_arrive_expect_tx(&kv_full[s], C::kStageBytes);
            for (int c = 0; c < HD / 64; ++c) {
                tma_load_2d(dk + c * (kBN * 128), tkv, &kv_full[s], p.H + h * HD + c * 64, row);
                tma_load_2d(dv + c * (kBN * 128), tkv, &kv_full[s], 2 * p.H + h * HD + c * 64, row);
            }
        }
    } else if (warp == 1 && lane == 0) {
        // ------------------------------------------------------------ MMA issuer
        constexpr uint32_t idesc_s = idesc_bf16_f32(kBM, kBN);
        constexpr uint32_t idesc_o = idesc_bf16_f32(kBM, HD) | (1u << 16);   // B (V) is MN-major
        const uint32_t aQ = smem_u32(sQ);
        const uint32_t aP = smem_u32(sP);
        bool ok = mbar_wait(q_full, 0);
        if (!ok) fail();
        auto issue_pv = [&](int j) -> bool {
            // O += P_j V_j once the softmax has published P_j
            if (!mbar_wait(p_full, j & 1)) return false;
            tc_fence_after();
            const int s = j % kStages;
            const uint32_t aV = smem_u32(sKV + s * C::kStageBytes + C::kKBytes);
#pragma unroll
            for (int k = 0; k < kBN / 16; ++k) {
                const uint64_t da = smem_desc_k_sw128(aP) + static_cast<uint64_t>(2 * k);
                const uint64_t db = smem_desc_mn_sw128(aV + k * 2048, kBN * 128);
                tc_mma_bf16(tmem + C::kColO, da, db, idesc_o, (j | k) != 0 ? 1u : 0u);
            }
            tc_commit(o_done);
            tc_commit(&kv_empty[s]);
            return true;
        };
        for (int j = 0; ok && j < ntiles && !*abort_flag; ++j) {
            const int s = j % kStages;
            if (!mbar_wait(&kv_full[s], (j / kStages) & 1)) { fail(); ok = false; break; }
            if (!mbar_wait(&s_free[j & 1], ((j >> 1) & 1) ^ 1)) { fail(); ok = false; break; }
            tc_fence_after();
            const uint32_t aK = smem_u32(sKV + s * C::kStageBytes);
            const uint32_t dS = tmem + ((j & 1) ? C::kColS1 : C::kColS0);
#pragma unroll
            for (int k = 0; k < HD / 16; ++k) {
                const uint32_t off_q = (k / 4) * (kBM * 128) + (k % 4) * 32;
                const uint32_t off_k = (k / 4) * (kBN * 128) + (k % 4) * 32;
                tc_mma_bf16(dS, smem_desc_k_sw128(aQ + off_q), smem_desc_k_sw128(aK + off_k), idesc_s,
                            k != 0 ? 1u : 0u);
            }
            tc_commit(&s_full[j & 1]);
            if (j >= 1 && !issue_pv(j - 1)) { fail(); ok = false; break; }
        }
        if (ok && !*abort_flag && ntiles > 0 && !issue_pv(ntiles - 1)) fail();
        tc_commit(drain);
        if (!mbar_wait(drain, 0)) report_status(status, kStatusWaitTimeout);
    } else if (warp >= 2) {
        // ------------------------------------------------------------ softmax
        const int q = warp & 3;
        const int r = q * 32 + lane;                     // query row within the tile = TMEM lane
        const uint32_t lane_base = static_cast<uint32_t>(q * 32) << 16;
        float m_used = -INFINITY;
        float l = 0.f;
        bool ok = true;
        for (int j = 0; j < ntiles; ++j) {
            if (*abort_flag) { ok = false; break; }
            if (!mbar_wait(&s_full[j & 1], (j >> 1) & 1)) { fail(); ok = false; break; }
            tc_fence_after();
            uint32_t sr[kBN];
            {
                uint32_t (&a)[32] = *reinterpret_cast<uint32_t(*)[32]>(&sr[0]);
                uint32_t (&c)[32] = *reinterpret_cast<uint32_t(*)[32]>(&sr[32]);
                const uint32_t ts = tmem + lane_base + ((j & 1) ? C::kColS1 : C::kColS0);
                tmem_ld_x32(ts, a);
                tmem_ld_x32(ts + 32, c);
                tmem_ld_wait();
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&s_free[j & 1]);

            const int ks = j < nt0 ? 0 : 1;
            const int valid = p.n[ks] - (j - (ks ? nt0 : 0)) * kBN;   // columns < valid are real tokens
            float mx = -INFINITY;
#pragma unroll
            for (int i = 0; i < kBN; ++i) {
                const float v = i < valid ? __uint_as_float(sr[i]) * p.scale_log2 : -INFINITY;
                sr[i] = __float_as_uint(v);
                mx = fmaxf(mx, v);
            }
            const bool grow = mx > m_used + kRescaleThreshold;
            const float m_new = grow ? mx : m_used;
            const float alpha = ex2(m_used - m_new);   // 0 on the first tile, 1 without growth
            uint32_t pk[kBN / 2];
            float sum = 0.f;
#pragma unroll
            for (int i = 0; i < kBN; i += 2) {
                const float e0 = ex2(__uint_as_float(sr[i]) - m_new);
                const float e1 = ex2(__uint_as_float(sr[i + 1]) - m_new);
                sum += e0 + e1;
                pk[i / 2] = pack_bf16x2(e0, e1);
            }
            l = l * alpha + sum;
            m_used = m_new;

            // P buffer and O are free once O += P_{j-1} V_{j-1} has completed
            if (j >= 1) {
                if (!mbar_wait(o_done, (j - 1) & 1)) { fail(); ok = false; break; }
                tc_fence_after();
                if (__any_sync(0xffffffffu, grow)) {
                    // rescale this warp's O rows (alpha = 1 for rows whose max held)
#pragma unroll 1
                    for (int c = 0; c < HD; c += 32) {
                        uint32_t o[32];
                        const uint32_t to = tmem + lane_base + C::kColO + c;
                        tmem_ld_x32(to, o);
                        tmem_ld_wait();
#pragma unroll
                        for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
                        tmem_st_x32(to, o);
                    }
                    tmem_st_wait();
                }
            }
            // P row r: 64 bf16 = one 128-byte swizzle row, 8 chunks of 16 bytes
            {
                uint8_t* prow = sP + (r >> 3) * 1024 + (r & 7) * 128;
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    *reinterpret_cast<uint4*>(prow + ((c ^ (r & 7)) << 4)) =
                        make_uint4(pk[4 * c], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(p_full);
        }
        // ---- epilogue: O / l -> bf16
        if (ok && ntiles > 0 && mbar_wait(o_done, (ntiles - 1) & 1)) {
            tc_fence_after();
            const float inv = 1.f / l;
            const int row = q0 + r;
            const bool live = row < p.n[seg];
            __nv_bfloat16* dst = p.out[seg] + (static_cast<int64_t>(b) * p.n[seg] + row) * p.ldo[seg] + h * HD;
#pragma unroll 1
            for (int c = 0; c < HD; c += 32) {
                uint32_t o[32];
                tmem_ld_x32(tmem + lane_base + C::kColO + c, o);
                tmem_ld_wait();
                if (live) {
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const float* f = reinterpret_cast<const float*>(o) + 8 * k;
                        *reinterpret_cast<uint4*>(dst + c + 8 * k) =
                            make_uint4(pack_bf16x2(f[0] * inv, f[1] * inv), pack_bf16x2(f[2] * inv, f[3] * inv),
                                       pack_bf16x2(f[4] * inv, f[5] * inv), pack_bf16x2(f[6] * inv, f[7] * inv));
                    }
                }
            }
        } else if (ok && ntiles > 0) {
            fail();
        }
    }

    if (*abort_flag) {
        const uint64_t t0 = global_timer_ns();
        while (global_timer_ns() - t0 < 50000ull) {
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::kTmemCols);
    }
}

template <int HD>
int launch_attn(const AttnSegment& s0, const AttnSegment& s1, int B, int heads, int H, cudaStream_t stream) {
    using C = ACfg<HD>;
    if (cudaFuncSetAttribute(attn_tcgen05_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) !=
        cudaSuccess)
        return set_error(FF_ERR_CUDA, "attention: cannot set shared memory size");
    const AttnSegment* seg[2] = {&s0, &s1};
    CUtensorMap tq[2], tkv[2];
    for (int i = 0; i < 2; ++i) {
        // a segment with no tokens still needs a valid map: point it at the other one
        const AttnSegment& s = seg[i]->n > 0 ? *seg[i] : *seg[1 - i];
        const int64_t rows = static_cast<int64_t>(B) * s.n;
        int rc = make_tmap_bf16(&tq[i], s.qkv, rows, 3 * static_cast<int64_t>(H), s.ld, kBM);
        if (rc) return rc;
        rc = make_tmap_bf16(&tkv[i], s.qkv, rows, 3 * static_cast<int64_t>(H), s.ld, kBN);
        if (rc) return rc;
    }
    AttnParams p;
    p.n[0] = s0.n;
    p.n[1] = s1.n;
    p.qtiles0 = (s0.n + kBM - 1) / kBM;
    p.H = H;
    p.scale_log2 = static_cast<float>(1.4426950408889634 / sqrt(static_cast<double>(HD)));
    p.out[0] = s0.out;
    p.out[1] = s1.out;
    p.ldo[0] = s0.ldo;
    p.ldo[1] = s1.ldo;
    const int N = s0.n + s1.n;
    const dim3 grid(p.qtiles0 + (s1.n + kBM - 1) / kBM, heads, B);
    const double nn = static_cast<double>(N) * N;
    ProfScope prof(stream, "attention", 4.0 * B * heads * nn * HD, 8.0 * B * static_cast<double>(N) * H);
    attn_tcgen05_kernel<HD><<<grid, kThreads, C::kSmemBytes, stream>>>(tq[0], tq[1], tkv[0], tkv[1], p,
                                                                        device_status_ptr());
    return check_launch("attn_tcgen05_kernel");
}

}  // namespace

int attention(const AttnSegment& s0, const AttnSegment& s1, int B, int heads, int head_dim, int H,
              cudaStream_t stream) {
    if (B <= 0 || heads <= 0 || s0.n < 0 || s1.n < 0 || s0.n + s1.n <= 0)
        return set_error(FF_ERR_INVALID_ARG, "attention: bad shape");
    if (B > 65535 || heads > 65535) return set_error(FF_ERR_UNSUPPORTED, "attention: grid too large");
    if ((s0.n && (!s0.qkv || !s0.out)) || (s1.n && (!s1.qkv || !s1.out)))
        return set_error(FF_ERR_INVALID_ARG, "attention: null segment");
    if (s0.ld % 8 || s1.ld % 8 || s0.ldo % 8 || s1.ldo % 8)
        return set_error(FF_ERR_INVALID_ARG, "attention: leading dimensions must be multiples of 8");
    if ((s0.n && !aligned16(s0.out)) || (s1.n && !aligned16(s1.out)))
        return set_error(FF_ERR_INVALID_ARG, "attention: outputs must be 16-byte aligned");
    if (H % 64) return set_error(FF_ERR_UNSUPPORTED, "attention: H %% 64 != 0");
    if (head_dim == 128) return launch_attn<128>(s0, s1, B, heads, H, stream);
    if (head_dim == 64) return launch_attn<64>(s0, s1, B, heads, H, stream);
    return set_error(FF_ERR_UNSUPPORTED, "attention: head_dim %d", head_dim);
}

}  // namespace ff

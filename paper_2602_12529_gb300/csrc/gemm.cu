// gemm.cu -- persistent, warp-specialised tcgen05 GEMM for sm_103a.
//
//   D[M, N] = A[M, K] * B[N, K]^T      (bf16 operands, fp32 accumulation)
//
// Every Linear of the DiT (nn.Linear weights [out, in], activations [tokens,
// in]) runs through this kernel.  Layout per CTA (one CTA per SM):
//   warp 0      TMA producer: 128x64 A tile + BNx64 B tile per stage, 128-byte
//               swizzle, STAGES-deep mbarrier ring.
//   warp 1      TMEM allocator; lane 0 issues tcgen05.mma (M=128, N=BN, K=16
//               per instruction) into one of two TMEM accumulators.
//   warps 2..5  epilogue: tcgen05.ld of the accumulator (one TMEM lane = one
//               output row per thread), then the fused tail -- bias, GELU or
//               SiLU, and either a bf16/fp32 store (optionally split over two
//               outputs by column; each warp stages 32 x 32 blocks in shared
//               memory and writes them with TMA bulk stores) or the adaLN
//               gated residual update x += gate[b] * (acc + bias) on the fp32
//               residual stream.
// The two TMEM accumulators let the epilogue of tile i overlap the main loop
// of tile i+1.  Tiles are visited in groups of 16 M-blocks so that the A and
// B panels being read at any moment stay resident in L2.
//
// Every wait is bounded (ptx.cuh); on a timeout the kernel records
// kStatusWaitTimeout in the device status word, drains its own tensor-core
// work, frees TMEM and returns.
#include <type_traits>

#include "internal.h"
#include "ptx.cuh"

namespace ff {
namespace {

constexpr int BM = 128;
constexpr int BK = 64;
constexpr int kThreads = 192;
constexpr int kGroupM = 16;

template <int BN>
struct Cfg {
    static constexpr int kStages = BN == 256 ? 4 : (BN == 128 ? 6 : 8);
    static constexpr int kABytes = BM * BK * 2;
    static constexpr int kBBytes = BN * BK * 2;
    static constexpr int kStageBytes = kABytes + kBBytes;
    static constexpr int kTmemCols = 2 * BN;
    static constexpr int kBarrierBytes = 256;
    static constexpr int kResidBytes = BM * 32 * 4;   // one 128 x 32 fp32 residual chunk (two buffers)
    static constexpr int kEpiBytes = 2 * kResidBytes;  // epilogue staging: residual chunks or output blocks
    static constexpr int kStageBufs = kEpiBytes / (4 * 4096);   // 4 KB output blocks per epilogue warp
    static constexpr int kSmemBytes = kStages * kStageBytes + kEpiBytes + 1024 + kBarrierBytes;
};

__device__ __forceinline__ void tile_coords(int tile, int num_m, int num_n, int& mb, int& nb) {
    const int group_tiles = kGroupM * num_n;
    const int group = tile / group_tiles;
    const int first_m = group * kGroupM;
    const int gm = min(num_m - first_m, kGroupM);
    const int local = tile - group * group_tiles;
    mb = first_m + local % gm;
    nb = local / gm;
}

__device__ __forceinline__ void bias_add8(float* v, const __nv_bfloat16* b) {
    const uint4 u = *reinterpret_cast<const uint4*>(b);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 f = unpack_bf16x2(w[i]);
        v[2 * i] += f.x;
        v[2 * i + 1] += f.y;
    }
}

// 32 consecutive values of one row as bf16 (four 16-byte stores), and back.
__device__ __forceinline__ void store_bf16x32(__nv_bfloat16* p, const float* v) {
    uint4* o = reinterpret_cast<uint4*>(p);
#pragma unroll
    for (int j = 0; j < 4; ++j)
        o[j] = make_uint4(pack_bf16x2(v[8 * j], v[8 * j + 1]), pack_bf16x2(v[8 * j + 2], v[8 * j + 3]),
                          pack_bf16x2(v[8 * j + 4], v[8 * j + 5]), pack_bf16x2(v[8 * j + 6], v[8 * j + 7]));
}
__device__ __forceinline__ void load_bf16x32(const __nv_bfloat16* p, float* v) {
    const uint4* s = reinterpret_cast<const uint4*>(p);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const uint4 u = s[j];
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = unpack_bf16x2(w[i]);
            v[8 * j + 2 * i] = f.x;
            v[8 * j + 2 * i + 1] = f.y;
        }
    }
}

// Gated residual, one 32-column chunk: x[row, n..n+31] += gate[b(row), n..] *
// (acc + bias).  The residual chunk of the whole 128-row tile sits in shared
// memory (loaded by TMA with 128-byte swizzle, 16-byte piece j of row r at
// position j ^ (r % 8)); each thread updates its own row there, and the
// chunk goes back by a TMA store.
__device__ __forceinline__ void gated_update(const GemmEpilogue& e, int M, int row, int r, int n, const float (&v)[32],
                                             uint8_t* rbuf) {
    float4 g[8];
    if (row < M) {
        if (e.gate) {
            const float4* gp = reinterpret_cast<const float4*>(e.gate + static_cast<int64_t>(row / e.rows_per_sample) *
                                                                         e.ld_gate + n);
#pragma unroll
            for (int j = 0; j < 8; ++j) g[j] = gp[j];
        } else {
#pragma unroll
            for (int j = 0; j < 8; ++j) g[j] = make_float4(1.f, 1.f, 1.f, 1.f);
        }
    } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) g[j] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    uint8_t* rowp = rbuf + r * 128;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        float4* px = reinterpret_cast<float4*>(rowp + ((j ^ (r & 7)) << 4));
        float4 x = *px;
        x.x = fmaf(g[j].x, v[4 * j], x.x);
        x.y = fmaf(g[j].y, v[4 * j + 1], x.y);
        x.z = fmaf(g[j].z, v[4 * j + 2], x.z);
        x.w = fmaf(g[j].w, v[4 * j + 3], x.w);
        *px = x;
    }
}

// Fused QKV tail: per-head RMSNorm of q / k (bias first, eps 1e-6, learned
// scale), then RoPE from the cos/sin table, then the bf16 store.  Two passes
// over each head's TMEM columns: the first sums squares, the second
// normalises, rotates and stores.  The row is one token; its rotation pairs
// (2j, 2j+1) lie inside each 32-column chunk.
__device__ __forceinline__ void qk_norm_tile(const GemmEpilogue& e, int M, int row, int n0, uint32_t t_acc, int BN) {
    const int d = e.head_dim;
    const int half = e.qk_cols >> 1;
    const bool rot = e.rope_cs != nullptr && row >= e.rope_row0;
    const int h0 = e.axes0 >> 1, h1 = e.axes1 >> 1, h2 = e.axes2 >> 1;
    // table offsets of this token's frame / row / column entries
    int base0 = 0, base1 = 0, base2 = 0;
    if (rot) {
        const int n = (row - e.rope_row0) % e.n_img;
        const int hw = e.grid_h * e.grid_w;
        base0 = (n / hw) * h0;
        base1 = e.grid_f * h0 + ((n / e.grid_w) % e.grid_h) * h1 - h0;
        base2 = e.grid_f * h0 + e.grid_h * h1 + (n % e.grid_w) * h2 - h0 - h1;
    }
    for (int c0 = 0; c0 < BN; c0 += d) {
        const int col = n0 + c0;                       // first column of this head
        float ss = 0.f;
        for (int c = 0; c < d; c += 32) {
            uint32_t r[32];
            tmem_ld_x32(t_acc + c0 + c, r);
            tmem_ld_wait();
            float v[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
            if (e.bias) {
#pragma unroll
                for (int j = 0; j < 4; ++j) bias_add8(v + 8 * j, e.bias + col + c + 8 * j);
            }
            if (e.aux && row < M) store_bf16x32(e.aux + static_cast<int64_t>(row) * e.ld_aux + col + c, v);
#pragma unroll
            for (int i = 0; i < 32; ++i) ss = fmaf(v[i], v[i], ss);
        }
        const float rstd = rsqrtf(ss / d + 1e-6f);
        const __nv_bfloat16* sc = col < half ? e.q_scale : e.k_scale;
        for (int c = 0; c < d; c += 32) {
            uint32_t r[32];
            tmem_ld_x32(t_acc + c0 + c, r);
            tmem_ld_wait();
            float v[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
            if (e.bias) {
#pragma unroll
                for (int j = 0; j < 4; ++j) bias_add8(v + 8 * j, e.bias + col + c + 8 * j);
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const uint4 u = *reinterpret_cast<const uint4*>(sc + c + 8 * j);
                const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float2 f = unpack_bf16x2(w[i]);
                    v[8 * j + 2 * i] *= rstd * f.x;
                    v[8 * j + 2 * i + 1] *= rstd * f.y;
                }
            }
            if (rot) {
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const int pair = (c >> 1) + i;
                    const int idx = pair < h0 ? base0 + pair : (pair < h0 + h1 ? base1 + pair : base2 + pair);
                    const float2 cs = e.rope_cs[idx];
                    const float x0 = v[2 * i], x1 = v[2 * i + 1];
                    v[2 * i] = x0 * cs.x - x1 * cs.y;
                    v[2 * i + 1] = x0 * cs.y + x1 * cs.x;
                }
            }
            if (row < M) {
                uint4* o = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(e.out0) + static_cast<int64_t>(row) * e.ld0 +
                                                    col + c);
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float* s4 = v + 8 * j;
                    o[j] = make_uint4(pack_bf16x2(s4[0], s4[1]), pack_bf16x2(s4[2], s4[3]), pack_bf16x2(s4[4], s4[5]),
                                      pack_bf16x2(s4[6], s4[7]));
                }
            }
        }
    }
}

// Bias of a 32-column chunk (bf16 pairs), loaded ahead of its use.
__device__ __forceinline__ void load_bias32(const __nv_bfloat16* bias, int n, uint4 (&u)[4]) {
#pragma unroll
    for (int j = 0; j < 4; ++j) u[j] = bias ? reinterpret_cast<const uint4*>(bias + n)[j] : make_uint4(0, 0, 0, 0);
}

// Bias and activation of one 32-column chunk of the row held by this thread
// (plus the optional pre-activation copy and activation-derivative factor).
__device__ __forceinline__ void epilogue_values(const GemmEpilogue& e, int row, int M, int n, const uint4 (&bu)[4],
                                                float (&v)[32]) {
    if (e.bias) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const uint32_t w[4] = {bu[j].x, bu[j].y, bu[j].z, bu[j].w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float2 f = unpack_bf16x2(w[i]);
                v[8 * j + 2 * i] += f.x;
                v[8 * j + 2 * i + 1] += f.y;
            }
        }
    }
    if (e.aux && row < M) store_bf16x32(e.aux + static_cast<int64_t>(row) * e.ld_aux + n, v);
    if (e.gelu_pre && n >= e.act_from && row < M) {
        float pre[32];
        load_bf16x32(e.gelu_pre + static_cast<int64_t>(row) * e.ld_pre + (n - e.act_from), pre);
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] *= gelu_tanh_grad(pre[i]);
    }
    if (e.act != ACT_NONE && n >= e.act_from) {
        if (e.act == ACT_GELU) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = gelu_tanh(v[i]);
        } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = silu(v[i]);
        }
    }
}

// Output maps of a launch: problem i stores columns [0, split_n) through
// m[2 i] and columns [split_n, N) through m[2 i + 1] (based at out1 + col1).
struct OutMaps {
    CUtensorMap m[4];
};

// One 32 x 32 output block of this warp (lane = row) into its shared staging
// buffer, in the swizzled layout of the output map: fp32 rows of 128 bytes
// (16-byte piece j of row r at j ^ (r % 8)), bf16 rows of 64 bytes (piece j at
// j ^ ((r / 2) % 4)).  Either way the 8 lanes of a store phase hit distinct
// banks.
__device__ __forceinline__ void stage_chunk(bool f32, int lane, const float (&v)[32], uint8_t* buf) {
    if (f32) {
        uint8_t* row = buf + lane * 128;
#pragma unroll
        for (int j = 0; j < 8; ++j)
            *reinterpret_cast<float4*>(row + ((j ^ (lane & 7)) << 4)) =
                make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
    } else {
        uint8_t* row = buf + lane * 64;
#pragma unroll
        for (int j = 0; j < 4; ++j)
            *reinterpret_cast<uint4*>(row + ((j ^ ((lane >> 1) & 3)) << 4)) =
                make_uint4(pack_bf16x2(v[8 * j], v[8 * j + 1]), pack_bf16x2(v[8 * j + 2], v[8 * j + 3]),
                           pack_bf16x2(v[8 * j + 4], v[8 * j + 5]), pack_bf16x2(v[8 * j + 6], v[8 * j + 7]));
    }
}

// One tile of the epilogue for the 128 rows m0.. held in this CTA's TMEM
// (t_acc: this warp's lane quarter of the accumulator).  With EW = 8
// epilogue warps, two warps share each lane quarter and split the tile's
// columns in halves (column group g = (warp - 2) / 4); each group has its own
// pair of residual buffers and barriers and its own leader.  `to` are the
// problem's two output maps; the warp owns SB staging blocks of 4 KB and `sc`
// counts its store steps, which rotate through them.  Returns false after a
// bounded wait gave up.
template <int BN, int SB, int EW>
__device__ __forceinline__ bool epilogue_tile(const GemmEpilogue& epi, int M, int N, int m0, int nb, uint32_t t_acc,
                                              int q, int lane, int warp, bool leader, const CUtensorMap* tr,
                                              const CUtensorMap* to, uint8_t* rbuf, uint64_t* rfull_bar,
                                              uint64_t* rdone_bar, uint32_t (&ruse)[2], uint32_t& sc, int* status,
                                              volatile int* abort_flag) {
    using C = Cfg<BN>;
    constexpr int CG = BN * 4 / EW;             // columns per column group
    const int g = EW == 8 ? (warp - 2) >> 2 : 0;
    const bool gated = epi.epi == EPI_GATED_RESIDUAL;
    const int r = q * 32 + lane;                // row within the tile = TMEM lane
    const int row = m0 + r;
    if (gated) {
        bool ok = true;
        rbuf += 2 * g * C::kResidBytes;
        rfull_bar += 2 * g;
        rdone_bar += 2 * g;
        const int c_end = (g + 1) * (CG / 32);
        for (int c = g * (CG / 32); c < c_end; ++c) {
            const int n = nb * BN + c * 32;
            const int b = (c - g * (CG / 32)) & 1;
            uint32_t rr[32];
            tmem_ld_x32(t_acc + c * 32, rr);
            tmem_ld_wait();
            float v[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(rr[i]);
            if (epi.bias) {
#pragma unroll
                for (int j = 0; j < 4; ++j) bias_add8(v + 8 * j, epi.bias + n + 8 * j);
            }
            if (epi.aux && row < M) store_bf16x32(epi.aux + static_cast<int64_t>(row) * epi.ld_aux + n, v);
            if (!mbar_wait(&rfull_bar[b], ruse[b] & 1)) {
                report_status(status, kStatusWaitTimeout);
                *abort_flag = 1;
                ok = false;
            }
            if (ok) gated_update(epi, M, row, r, n, v, rbuf + b * C::kResidBytes);
            fence_proxy_async_smem();
            mbar_arrive(&rdone_bar[b]);
            // the leader stores the chunk once every thread has updated it
            // (an mbarrier, not bar.sync: a thread that gave up on a wait
            // must not be able to stall the others)
            if (leader && ok && !mbar_wait(&rdone_bar[b], ruse[b] & 1)) {
                report_status(status, kStatusWaitTimeout);
                *abort_flag = 1;
                ok = false;
            }
            ++ruse[b];
            if (leader && ok) {
                tma_store_2d(&to[0], rbuf + b * C::kResidBytes, n, m0);
                bulk_commit();
                if (c + 2 < c_end) {
                    bulk_wait_read<0>();
                    mbar_arrive_expect_tx(&rfull_bar[b], C::kResidBytes);
                    tma_load_2d(rbuf + b * C::kResidBytes, tr, &rfull_bar[b], n + 64, m0);
                }
            }
        }
        if (!ok) return false;
    } else if (epi.qk_cols > 0 && nb * BN < epi.qk_cols) {
        qk_norm_tile(epi, M, row, nb * BN + g * CG, t_acc + g * CG, CG);
    } else {
        // plain store: bias / activation on the row held by this thread,
        // staged as 32 x 32 blocks and written by TMA bulk stores (rows past
        // M are clipped by the map).  A step covers CW columns (two blocks
        // when the warp has room to double-buffer them, which halves the
        // per-step fence / sync / issue cost); the next step's accumulator
        // columns and bias are requested before this step is processed, and
        // a staging buffer is reused once the store NB steps back has read it
        // out.
        constexpr int CW = SB >= 4 ? 64 : 32;
        constexpr int NB = SB * 32 / CW;
        uint8_t* stage = rbuf + (warp - 2) * (SB * 4096);
        const int row0 = m0 + q * 32;
        const int ncol = N - nb * BN < (g + 1) * CG ? N - nb * BN : (g + 1) * CG;   // a multiple of 32
        uint32_t rr[CW];
        uint4 bnext[CW / 8];
        auto fetch = [&](int c) {
#pragma unroll
            for (int k = 0; k < CW / 32; ++k)
                if (c + 32 * k < ncol) {
                    tmem_ld_x32(t_acc + c + 32 * k, *reinterpret_cast<uint32_t(*)[32]>(&rr[32 * k]));
                    load_bias32(epi.bias, nb * BN + c + 32 * k, *reinterpret_cast<uint4(*)[4]>(&bnext[4 * k]));
                }
        };
        fetch(g * CG);
#pragma unroll 1
        for (int c = g * CG; c < ncol; c += CW) {
            const int nblk = ncol - c < CW ? 1 : CW / 32;
            tmem_ld_wait();
            float v[CW];
#pragma unroll
            for (int i = 0; i < CW; ++i) v[i] = __uint_as_float(rr[i]);
            uint4 bcur[CW / 8];
#pragma unroll
            for (int j = 0; j < CW / 8; ++j) bcur[j] = bnext[j];
            if (c + CW < ncol) fetch(c + CW);
            uint8_t* buf = stage + (sc % NB) * (CW / 32) * 4096;
#pragma unroll
            for (int k = 0; k < CW / 32; ++k)
                if (k < nblk)
                    epilogue_values(epi, row, M, nb * BN + c + 32 * k,
                                    *reinterpret_cast<const uint4(*)[4]>(&bcur[4 * k]),
                                    *reinterpret_cast<float(*)[32]>(&v[32 * k]));
            if (lane == 0) bulk_wait_read<NB - 1>();
            __syncwarp();
#pragma unroll
            for (int k = 0; k < CW / 32; ++k)
                if (k < nblk) stage_chunk(epi.out_f32 != 0, lane, *reinterpret_cast<float(*)[32]>(&v[32 * k]),
                                          buf + k * 4096);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
#pragma unroll
                for (int k = 0; k < CW / 32; ++k) {
                    if (k >= nblk) break;
                    const int n = nb * BN + c + 32 * k;
                    if (n < epi.split_n) tma_store_2d(&to[0], buf + k * 4096, n, row0);
                    else tma_store_2d(&to[1], buf + k * 4096, n - epi.split_n, row0);
                }
                bulk_commit();
            }
            ++sc;
        }
    }
    return true;
}

// Up to two independent GEMM problems share one persistent launch: the tile
// space is problem 0's tiles followed by problem 1's, so a small problem
// (the text stream of a double-stream block) fills the tail of a large one.
struct GemmGroup {
    int M[2], N[2], K[2];
    int num_m[2], num_n[2];
    int tiles0, tiles;
    GemmEpilogue epi[2];
};

__device__ __forceinline__ void locate(const GemmGroup& g, int tile, int& pr, int& mb, int& nb) {
    pr = tile < g.tiles0 ? 0 : 1;
    const int local = pr ? tile - g.tiles0 : tile;
    tile_coords(local, g.num_m[pr], g.num_n[pr], mb, nb);
}

// LAYOUT: bit 0 = A stored MN-major ([K, M]), bit 1 = B stored MN-major
// ([K, N]); compile-time, so the forward (K-major) kernel issues exactly the
// instructions it would without the option.
template <int BN, int LAYOUT>
__global__ void __launch_bounds__(kThreads, 1)
gemm_tcgen05_kernel(const __grid_constant__ CUtensorMap tm_a0, const __grid_constant__ CUtensorMap tm_b0,
                    const __grid_constant__ CUtensorMap tm_a1, const __grid_constant__ CUtensorMap tm_b1,
                    const __grid_constant__ CUtensorMap tm_r0, const __grid_constant__ CUtensorMap tm_r1,
                    const __grid_constant__ OutMaps om, const __grid_constant__ GemmGroup g, int* status) {
    using C = Cfg<BN>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* rbuf = smem + C::kStages * C::kStageBytes;            // [2][kResidBytes]
    uint64_t* full_bar = reinterpret_cast<uint64_t*>(rbuf + C::kEpiBytes);
    uint64_t* empty_bar = full_bar + C::kStages;
    uint64_t* tfull_bar = empty_bar + C::kStages;   // [2]
    uint64_t* tempty_bar = tfull_bar + 2;           // [2]
    uint64_t* drain_bar = tempty_bar + 2;           // [1]
    uint64_t* rfull_bar = drain_bar + 1;            // [2] residual chunk landed
    uint64_t* rdone_bar = rfull_bar + 2;            // [2] all 128 epilogue threads updated the chunk
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(rdone_bar + 2);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::kStages; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull_bar[a], 1);
            mbar_init(&tempty_bar[a], 4);
        }
        mbar_init(drain_bar, 1);
        mbar_init(&rfull_bar[0], 1);
        mbar_init(&rfull_bar[1], 1);
        mbar_init(&rdone_bar[0], 128);
        mbar_init(&rdone_bar[1], 128);
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tm_a0);
        prefetch_tmap(&tm_b0);
        if (g.tiles > g.tiles0) {
            prefetch_tmap(&tm_a1);
            prefetch_tmap(&tm_b1);
        }
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, C::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer
        int stage = 0;
        uint32_t phase = 0;
        for (int tile = blockIdx.x; tile < g.tiles && !*abort_flag; tile += gridDim.x) {
            int pr, mb, nb;
            locate(g, tile, pr, mb, nb);
            const CUtensorMap* ta = pr ? &tm_a1 : &tm_a0;
            const CUtensorMap* tb = pr ? &tm_b1 : &tm_b0;
            const int num_k = (g.K[pr] + BK - 1) / BK;
            for (int kb = 0; kb < num_k; ++kb) {
                if (!mbar_wait(&empty_bar[stage], phase ^ 1)) {
                    report_status(status, kStatusWaitTimeout);
                    *abort_flag = 1;
                    break;
                }
                uint8_t* sa = smem + stage * C::kStageBytes;
                uint8_t* sb = sa + C::kABytes;
                mbar_arrive_expect_tx(&full_bar[stage], C::kStageBytes);
                // K-major operands: one box of rows x 64 K; MN-major: boxes
                // of 64 K rows x 64 MN per 64-wide block (8 KB each)
                if (LAYOUT & 1) {
                    for (int j = 0; j < BM / 64; ++j)
                        tma_load_2d(sa + j * 8192, ta, &full_bar[stage], mb * BM + 64 * j, kb * BK);
                } else {
                    tma_load_2d(sa, ta, &full_bar[stage], kb * BK, mb * BM);
                }
                if (LAYOUT & 2) {
                    for (int j = 0; j < BN / 64; ++j)
                        tma_load_2d(sb + j * 8192, tb, &full_bar[stage], nb * BN + 64 * j, kb * BK);
                } else {
                    tma_load_2d(sb, tb, &full_bar[stage], kb * BK, nb * BN);
                }
                if (++stage == C::kStages) { stage = 0; phase ^= 1; }
            }
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer
        constexpr bool amn = (LAYOUT & 1) != 0, bmn = (LAYOUT & 2) != 0;
        constexpr uint32_t idesc = idesc_bf16_f32(BM, BN) | (static_cast<uint32_t>(amn) << 15) |
                                   (static_cast<uint32_t>(bmn) << 16);
        constexpr uint64_t a_step = amn ? 128 : 2, b_step = bmn ? 128 : 2;   // one K16 step, encoded >> 4
        int stage = 0;
        uint32_t phase = 0;
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int tile = blockIdx.x; tile < g.tiles && !*abort_flag; tile += gridDim.x) {
            const int pr = tile < g.tiles0 ? 0 : 1;
            const int num_k = (g.K[pr] + BK - 1) / BK;
            if (!mbar_wait(&tempty_bar[acc], acc_phase ^ 1)) {
                report_status(status, kStatusWaitTimeout);
                *abort_flag = 1;
                break;
            }
            tc_fence_after();
            const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
            bool ok = true;
            for (int kb = 0; kb < num_k; ++kb) {
                if (!mbar_wait(&full_bar[stage], phase)) {
                    report_status(status, kStatusWaitTimeout);
                    *abort_flag = 1;
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t sa = smem_u32(smem + stage * C::kStageBytes);
                const uint32_t sb = sa + C::kABytes;
                const uint64_t da = amn ? smem_desc_mn_sw128(sa, 8192) : smem_desc_k_sw128(sa);
                const uint64_t db = bmn ? smem_desc_mn_sw128(sb, 8192) : smem_desc_k_sw128(sb);
#pragma unroll
                for (int k = 0; k < BK / 16; ++k)
                    tc_mma_bf16(d_tmem, da + a_step * k, db + b_step * k, idesc, (kb | k) != 0 ? 1u : 0u);
                tc_commit(&empty_bar[stage]);
                if (++stage == C::kStages) { stage = 0; phase ^= 1; }
            }
            if (!ok) break;
            tc_commit(&tfull_bar[acc]);
            if (++acc == 2) { acc = 0; acc_phase ^= 1; }
        }
        // all tensor-core work of this thread finished before TMEM is freed
        tc_commit(drain_bar);
        if (!mbar_wait(drain_bar, 0)) report_status(status, kStatusWaitTimeout);
    } else if (warp >= 2) {
        // ---------------- epilogue (4 warps; warp w reads TMEM lanes 32*(w%4)..)
        const int q = warp & 3;
        const bool leader = warp == 2 && lane == 0;     // issues the residual TMA traffic
        uint32_t ruse[2] = {0, 0};                      // residual loads consumed per buffer
        uint32_t sc = 0;                                // output blocks staged by this warp
        const uint32_t t_acc_base = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int tile = blockIdx.x; tile < g.tiles && !*abort_flag; tile += gridDim.x) {
            int pr, mb, nb;
            locate(g, tile, pr, mb, nb);
            const GemmEpilogue& epi = g.epi[pr];
            const int M = g.M[pr], N = g.N[pr];
            const bool gated = epi.epi == EPI_GATED_RESIDUAL;
            const CUtensorMap* tr = pr ? &tm_r1 : &tm_r0;
            if (gated && leader) {
                // the first two residual chunks of this tile, ahead of the accumulator
                for (int c = 0; c < 2 && c < BN / 32; ++c) {
                    bulk_wait_read<0>();
                    mbar_arrive_expect_tx(&rfull_bar[c], C::kResidBytes);
                    tma_load_2d(rbuf + c * C::kResidBytes, tr, &rfull_bar[c], nb * BN + c * 32, mb * BM);
                }
            }
            if (!mbar_wait(&tfull_bar[acc], acc_phase)) {
                report_status(status, kStatusWaitTimeout);
                *abort_flag = 1;
                break;
            }
            tc_fence_after();
            if (!epilogue_tile<BN, C::kStageBufs, 4>(epi, M, N, mb * BM, nb, t_acc_base + static_cast<uint32_t>(acc * BN), q, lane, warp,
                                   leader, tr, &om.m[2 * pr], rbuf, rfull_bar, rdone_bar, ruse, sc, status,
                                   abort_flag))
                break;
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty_bar[acc]);
            if (++acc == 2) { acc = 0; acc_phase ^= 1; }
        }
        if (lane == 0) bulk_wait<0>();   // this warp's stores complete before the CTA's shared memory goes away
    }

    if (*abort_flag) {
        // let bulk copies already in flight land before the CTA exits
        const uint64_t t0 = global_timer_ns();
        while (global_timer_ns() - t0 < 50000ull) {
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, C::kTmemCols);
    }
}

// ---------------------------------------------------------------------------
// Two-SM variant: a cluster of two CTAs computes one 256 x 256 tile with
// tcgen05.mma.cta_group::2.  Each CTA stages its own 128 rows of A and its
// half (128 rows) of B, so per-SM shared-memory operand traffic per FLOP
// drops by a third against the 128 x 256 single-CTA tile.  The leader CTA
// (rank 0) owns the stage-full barriers (both CTAs' TMA loads complete on
// them) and the accumulator-empty barriers (both CTAs' epilogues arrive on
// them) and issues every MMA; its commits are multicast to the same barrier
// in both CTAs.  Each CTA's epilogue drains its own 128 accumulator rows.
// Every wait is bounded and both CTAs always reach the closing cluster
// barrier, so neither can leave while the other may still signal it.
// ---------------------------------------------------------------------------
constexpr int PBM = 256;   // rows per pair tile
constexpr int PBN = 256;   // columns per pair tile
constexpr int kPairStages = 5;
constexpr int kPairThreads = 320;   // producer, MMA, 8 epilogue warps

struct PairCfg {
    static constexpr int kABytes = 128 * BK * 2;           // this CTA's A rows
    static constexpr int kBBytes = (PBN / 2) * BK * 2;     // this CTA's half of B
    static constexpr int kStageBytes = kABytes + kBBytes;
    static constexpr int kResidBytes = 128 * 32 * 4;
    static constexpr int kEpiBytes = 4 * kResidBytes;   // 2 x 2 residual chunks, or 2 output blocks per warp
    static constexpr int kStageBufs = kEpiBytes / (8 * 4096);
    static constexpr int kBarrierBytes = 256;
    static constexpr int kSmemBytes = kPairStages * kStageBytes + kEpiBytes + 1024 + kBarrierBytes;
};

template <int LAYOUT>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kPairThreads, 1)
gemm_pair_kernel(const __grid_constant__ CUtensorMap tm_a0, const __grid_constant__ CUtensorMap tm_b0,
                 const __grid_constant__ CUtensorMap tm_a1, const __grid_constant__ CUtensorMap tm_b1,
                 const __grid_constant__ CUtensorMap tm_r0, const __grid_constant__ CUtensorMap tm_r1,
                 const __grid_constant__ OutMaps om, const __grid_constant__ GemmGroup g, int* status) {
    using C = PairCfg;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* rbuf = smem + kPairStages * C::kStageBytes;
    uint64_t* full_bar = reinterpret_cast<uint64_t*>(rbuf + C::kEpiBytes);   // used in the leader
    uint64_t* empty_bar = full_bar + kPairStages;                                   // both CTAs
    uint64_t* tfull_bar = empty_bar + kPairStages;   // [2] both CTAs
    uint64_t* tempty_bar = tfull_bar + 2;            // [2] leader, 16 arrivals
    uint64_t* drain_bar = tempty_bar + 2;            // [1] leader
    uint64_t* rfull_bar = drain_bar + 1;             // [2 groups][2] per CTA
    uint64_t* rdone_bar = rfull_bar + 4;             // [2 groups][2] per CTA
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(rdone_bar + 4);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const int cluster = blockIdx.x >> 1;
    const int nclusters = gridDim.x >> 1;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kPairStages; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull_bar[a], 1);
            mbar_init(&tempty_bar[a], 16);
        }
        for (int a = 0; a < 4; ++a) {
            mbar_init(&rfull_bar[a], 1);
            mbar_init(&rdone_bar[a], 128);
        }
        mbar_init(drain_bar, 1);
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tm_a0);
        prefetch_tmap(&tm_b0);
        if (g.tiles > g.tiles0) {
            prefetch_tmap(&tm_a1);
            prefetch_tmap(&tm_b1);
        }
    }
    if (warp == 1) {
        tmem_alloc_pair(tmem_slot, 2 * PBN);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    cluster_sync();   // both CTAs' barriers and TMEM exist before any cross-CTA traffic
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer (both CTAs; completion counted in the leader)
        int stage = 0;
        uint32_t phase = 0;
        for (int tile = cluster; tile < g.tiles && !*abort_flag; tile += nclusters) {
            int pr, mb, nb;
            locate(g, tile, pr, mb, nb);
            const CUtensorMap* ta = pr ? &tm_a1 : &tm_a0;
            const CUtensorMap* tb = pr ? &tm_b1 : &tm_b0;
            const int num_k = (g.K[pr] + BK - 1) / BK;
            for (int kb = 0; kb < num_k; ++kb) {
                if (!mbar_wait(&empty_bar[stage], phase ^ 1)) {
                    report_status(status, kStatusWaitTimeout);
                    *abort_flag = 1;
                    break;
                }
                uint8_t* sa = smem + stage * C::kStageBytes;
                uint8_t* sb = sa + C::kABytes;
                const uint32_t fb = mapa_shared(smem_u32(&full_bar[stage]), 0);
                if (rank == 0) mbar_arrive_expect_tx(&full_bar[stage], 2 * C::kStageBytes);
                const int ma = mb * PBM + rank * 128, nbb = nb * PBN + rank * (PBN / 2);
                if (LAYOUT & 1) {
                    for (int j = 0; j < 2; ++j) tma_load_2d_pair(sa + j * 8192, ta, fb, ma + 64 * j, kb * BK);
                } else {
                    tma_load_2d_pair(sa, ta, fb, kb * BK, ma);
                }
                if (LAYOUT & 2) {
                    for (int j = 0; j < 2; ++j) tma_load_2d_pair(sb + j * 8192, tb, fb, nbb + 64 * j, kb * BK);
                } else {
                    tma_load_2d_pair(sb, tb, fb, kb * BK, nbb);
                }
                if (++stage == kPairStages) { stage = 0; phase ^= 1; }
            }
        }
    } else if (warp == 1 && lane == 0 && rank == 0) {
        // ---------------- MMA issuer (leader only): 256 x 256 x 16 per instruction
        constexpr bool amn = (LAYOUT & 1) != 0, bmn = (LAYOUT & 2) != 0;
        constexpr uint32_t idesc = idesc_bf16_f32(PBM, PBN) | (static_cast<uint32_t>(amn) << 15) |
                                   (static_cast<uint32_t>(bmn) << 16);
        constexpr uint64_t a_step = amn ? 128 : 2, b_step = bmn ? 128 : 2;
        int stage = 0;
        uint32_t phase = 0;
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int tile = cluster; tile < g.tiles && !*abort_flag; tile += nclusters) {
            const int pr = tile < g.tiles0 ? 0 : 1;
            const int num_k = (g.K[pr] + BK - 1) / BK;
            if (!mbar_wait(&tempty_bar[acc], acc_phase ^ 1)) {
                report_status(status, kStatusWaitTimeout);
                *abort_flag = 1;
                break;
            }
            tc_fence_after();
            const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * PBN);
            bool ok = true;
            for (int kb = 0; kb < num_k; ++kb) {
                if (!mbar_wait(&full_bar[stage], phase)) {
                    report_status(status, kStatusWaitTimeout);
                    *abort_flag = 1;
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t sa = smem_u32(smem + stage * C::kStageBytes);
                const uint32_t sb = sa + C::kABytes;
                const uint64_t da = amn ? smem_desc_mn_sw128(sa, 8192) : smem_desc_k_sw128(sa);
                const uint64_t db = bmn ? smem_desc_mn_sw128(sb, 8192) : smem_desc_k_sw128(sb);
#pragma unroll
                for (int k = 0; k < BK / 16; ++k)
                    tc_mma_bf16_pair(d_tmem, da + a_step * k, db + b_step * k, idesc, (kb | k) != 0 ? 1u : 0u);
                tc_commit_pair_mc(&empty_bar[stage], 0x3);
                if (++stage == kPairStages) { stage = 0; phase ^= 1; }
            }
            if (!ok) break;
            tc_commit_pair_mc(&tfull_bar[acc], 0x3);
            if (++acc == 2) { acc = 0; acc_phase ^= 1; }
        }
        tc_commit_pair_mc(drain_bar, 0x1);
        if (!mbar_wait(drain_bar, 0)) report_status(status, kStatusWaitTimeout);
    } else if (warp >= 2) {
        // ---------------- epilogue (both CTAs, own 128 accumulator rows; two
        // warps per TMEM lane quarter, one per column half)
        const int q = warp & 3;
        const int grp = (warp - 2) >> 2;
        const bool leader = (warp == 2 || warp == 6) && lane == 0;
        uint32_t ruse[2] = {0, 0};
        uint32_t sc = 0;
        const uint32_t t_acc_base = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int tile = cluster; tile < g.tiles && !*abort_flag; tile += nclusters) {
            int pr, mb, nb;
            locate(g, tile, pr, mb, nb);
            const GemmEpilogue& epi = g.epi[pr];
            const int M = g.M[pr], N = g.N[pr];
            const int m0 = mb * PBM + rank * 128;
            const CUtensorMap* tr = pr ? &tm_r1 : &tm_r0;
            if (epi.epi == EPI_GATED_RESIDUAL && leader) {
                // the first two residual chunks of this group's column half
                for (int c = 0; c < 2; ++c) {
                    bulk_wait_read<0>();
                    mbar_arrive_expect_tx(&rfull_bar[2 * grp + c], C::kResidBytes);
                    tma_load_2d(rbuf + (2 * grp + c) * C::kResidBytes, tr, &rfull_bar[2 * grp + c],
                                nb * PBN + grp * (PBN / 2) + c * 32, m0);
                }
            }
            if (!mbar_wait(&tfull_bar[acc], acc_phase)) {
                report_status(status, kStatusWaitTimeout);
                *abort_flag = 1;
                break;
            }
            tc_fence_after();
            if (!epilogue_tile<PBN, PairCfg::kStageBufs, 8>(epi, M, N, m0, nb, t_acc_base + static_cast<uint32_t>(acc * PBN), q, lane, warp,
                                    leader, tr, &om.m[2 * pr], rbuf, rfull_bar, rdone_bar, ruse, sc, status,
                                    abort_flag))
                break;
            tc_fence_before();
            __syncwarp();
            // the leader's own warps arrive locally; the peer's through the cluster
            if (lane == 0) {
                if (rank == 0) mbar_arrive(&tempty_bar[acc]);
                else mbar_arrive_cluster(mapa_shared(smem_u32(&tempty_bar[acc]), 0));
            }
            if (++acc == 2) { acc = 0; acc_phase ^= 1; }
        }
        if (lane == 0) bulk_wait<0>();
    }

    if (*abort_flag) {
        const uint64_t t0 = global_timer_ns();
        while (global_timer_ns() - t0 < 50000ull) {
        }
    }
    tc_fence_before();
    cluster_sync();   // nothing crosses the pair after this point
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc_pair(tmem_base, 2 * PBN);
    }
}

// The two output maps of a store epilogue.  A gated-residual problem stores
// through its residual map instead; its entries (and an unsplit problem's
// second one) are copies of a valid map, so every kernel parameter is a
// well-formed tensor map.
int make_out_maps(const GemmArgs& a, CUtensorMap* m) {
    const GemmEpilogue& e = a.epi;
    if (e.epi == EPI_GATED_RESIDUAL) {
        // the updated residual's store map (the input's when updated in place)
        const int rc = make_tmap_f32_sw128(&m[0], e.resid_out ? e.resid_out : e.resid, a.M, a.N, e.ld_resid, 128);
        m[1] = m[0];
        return rc;
    }
    const bool f32 = e.out_f32 != 0;
    const int n0 = e.split_n < a.N ? e.split_n : a.N;
    int rc = make_tmap_out(&m[0], e.out0, a.M, n0, e.ld0, f32);
    if (rc) return rc;
    if (e.split_n < a.N) {
        const uint8_t* base1 = static_cast<const uint8_t*>(e.out1) + static_cast<int64_t>(e.col1) * (f32 ? 4 : 2);
        return make_tmap_out(&m[1], base1, a.M, a.N - e.split_n, e.ld1, f32);
    }
    m[1] = m[0];
    return FF_OK;
}

template <int LAYOUT>
int launch_pair(const GemmArgs* p, int n, cudaStream_t stream) {
    using C = PairCfg;
    if (cudaFuncSetAttribute(gemm_pair_kernel<LAYOUT>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) !=
        cudaSuccess)
        return set_error(FF_ERR_CUDA, "gemm (pair): cannot set shared memory size (%d B)", C::kSmemBytes);
    CUtensorMap ta[2], tb[2], tr[2];
    OutMaps om;
    GemmGroup g{};
    double flops = 0.0, bytes = 0.0;
    for (int i = 0; i < 2; ++i) {
        const GemmArgs& a = p[i < n ? i : 0];
        int rc = make_out_maps(a, &om.m[2 * i]);
        if (rc) return rc;
        rc = a.a_mn ? make_tmap_bf16(&ta[i], a.A, a.K, a.M, a.lda, 64) : make_tmap_bf16(&ta[i], a.A, a.M, a.K, a.lda, 128);
        if (rc) return rc;
        rc = a.b_mn ? make_tmap_bf16(&tb[i], a.B, a.K, a.N, a.ldb, 64)
                    : make_tmap_bf16(&tb[i], a.B, a.N, a.K, a.ldb, PBN / 2);
        if (rc) return rc;
        if (a.epi.epi == EPI_GATED_RESIDUAL) {
            rc = make_tmap_f32_sw128(&tr[i], a.epi.resid, a.M, a.N, a.epi.ld_resid, 128);
            if (rc) return rc;
        } else {
            tr[i] = ta[i];
        }
        g.M[i] = a.M;
        g.N[i] = a.N;
        g.K[i] = a.K;
        g.num_m[i] = (a.M + PBM - 1) / PBM;
        g.num_n[i] = (a.N + PBN - 1) / PBN;
        g.epi[i] = a.epi;
        if (i < n) {
            const double mn = static_cast<double>(a.M) * a.N;
            flops += 2.0 * mn * a.K;
            bytes += 2.0 * (static_cast<double>(a.M) + a.N) * a.K +
                     (a.epi.epi == EPI_GATED_RESIDUAL ? mn * 8.0 : mn * (a.epi.out_f32 ? 4.0 : 2.0));
        }
    }
    for (int i = 0; i < n; ++i)
        if (p[i].epi.epi == EPI_GATED_RESIDUAL && p[i].N % PBN)
            return set_error(FF_ERR_UNSUPPORTED, "gemm (pair): gated residual needs N %% 256 == 0");
    g.tiles0 = g.num_m[0] * g.num_n[0];
    g.tiles = g.tiles0 + (n > 1 ? g.num_m[1] * g.num_n[1] : 0);
    const int clusters = g.tiles < num_sms() / 2 ? g.tiles : num_sms() / 2;
    ProfScope prof(stream, "gemm_bf16", flops, bytes);
    gemm_pair_kernel<LAYOUT><<<2 * clusters, kPairThreads, C::kSmemBytes, stream>>>(ta[0], tb[0], ta[1], tb[1], tr[0], tr[1], om,
                                                                        g, device_status_ptr());
    return check_launch("gemm_pair_kernel");
}

template <int BN, int LAYOUT>
int launch(const GemmArgs* p, int n, cudaStream_t stream) {
    using C = Cfg<BN>;
    if (cudaFuncSetAttribute(gemm_tcgen05_kernel<BN, LAYOUT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             C::kSmemBytes) !=
        cudaSuccess)
        return set_error(FF_ERR_CUDA, "gemm: cannot set shared memory size (%d B)", C::kSmemBytes);
    CUtensorMap ta[2], tb[2], tr[2];
    OutMaps om;
    GemmGroup g{};
    double flops = 0.0, bytes = 0.0;
    for (int i = 0; i < 2; ++i) {
        const GemmArgs& a = p[i < n ? i : 0];
        int rc = make_out_maps(a, &om.m[2 * i]);
        if (rc) return rc;
        rc = a.a_mn ? make_tmap_bf16(&ta[i], a.A, a.K, a.M, a.lda, 64) : make_tmap_bf16(&ta[i], a.A, a.M, a.K, a.lda, BM);
        if (rc) return rc;
        rc = a.b_mn ? make_tmap_bf16(&tb[i], a.B, a.K, a.N, a.ldb, 64) : make_tmap_bf16(&tb[i], a.B, a.N, a.K, a.ldb, BN);
        if (rc) return rc;
        if (a.epi.epi == EPI_GATED_RESIDUAL) {
            rc = make_tmap_f32_sw128(&tr[i], a.epi.resid, a.M, a.N, a.epi.ld_resid, BM);
            if (rc) return rc;
        } else {
            tr[i] = ta[i];   // unused: the problem has no residual
        }
        g.M[i] = a.M;
        g.N[i] = a.N;
        g.K[i] = a.K;
        g.num_m[i] = (a.M + BM - 1) / BM;
        g.num_n[i] = (a.N + BN - 1) / BN;
        g.epi[i] = a.epi;
        if (i < n) {
            const double mn = static_cast<double>(a.M) * a.N;
            flops += 2.0 * mn * a.K;
            bytes += 2.0 * (static_cast<double>(a.M) + a.N) * a.K +
                     (a.epi.epi == EPI_GATED_RESIDUAL ? mn * 8.0 : mn * (a.epi.out_f32 ? 4.0 : 2.0));
        }
    }
    g.tiles0 = g.num_m[0] * g.num_n[0];
    g.tiles = g.tiles0 + (n > 1 ? g.num_m[1] * g.num_n[1] : 0);
    const int grid = g.tiles < num_sms() ? g.tiles : num_sms();
    ProfScope prof(stream, "gemm_bf16", flops, bytes);
    for (int i = 0; i < n; ++i)
        if (p[i].epi.epi == EPI_GATED_RESIDUAL && p[i].N % BN)
            return set_error(FF_ERR_UNSUPPORTED, "gemm: gated residual needs N (%d) to be a multiple of %d", p[i].N, BN);
    gemm_tcgen05_kernel<BN, LAYOUT><<<grid, kThreads, C::kSmemBytes, stream>>>(ta[0], tb[0], ta[1], tb[1], tr[0], tr[1], om,
                                                                       g, device_status_ptr());
    return check_launch("gemm_tcgen05_kernel");
}

// ---------------------------------------------------------------------------
// Few-row GEMM (M <= 8: the per-sample time-embedding and modulation
// products).  out[m, n] = act(A[m, :] . W[n, :] + bias[n]).  It is bound by
// reading W once, so: A is staged in shared memory, each warp streams two W
// rows with 16-byte loads (coalesced along K), keeps M accumulators per row
// and reduces across lanes.  Persistent grid; columns are handed out in
// groups of 16 per block.
// ---------------------------------------------------------------------------
constexpr int kGemvMaxRows = 8;
constexpr int kGemvMaxK = 8192;
constexpr int kGemvThreads = 256;

constexpr int kGemvCols = 4;   // W rows (output columns) per warp

template <int MR>
__global__ void __launch_bounds__(kGemvThreads) gemv_rows_kernel(const __nv_bfloat16* A, int64_t lda, int M,
                                                                 const __nv_bfloat16* W, int64_t ldw, int N, int K,
                                                                 const GemmEpilogue e) {
    extern __shared__ uint4 sA4[];   // [MR][K] bf16; rows >= M are zero
    const int k8 = K / 8;
    for (int i = threadIdx.x; i < MR * k8; i += kGemvThreads) {
        const int m = i / k8, c = i - m * k8;
        sA4[i] = m < M ? *reinterpret_cast<const uint4*>(A + static_cast<int64_t>(m) * lda + c * 8)
                       : make_uint4(0u, 0u, 0u, 0u);
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int kWarps = kGemvThreads / 32;
    for (int n0 = (blockIdx.x * kWarps + warp) * kGemvCols; n0 < N; n0 += gridDim.x * kWarps * kGemvCols) {
        float acc[kGemvCols][MR];
#pragma unroll
        for (int j = 0; j < kGemvCols; ++j)
#pragma unroll
            for (int m = 0; m < MR; ++m) acc[j][m] = 0.f;
        const uint4* w[kGemvCols];
#pragma unroll
        for (int j = 0; j < kGemvCols; ++j)
            w[j] = reinterpret_cast<const uint4*>(W + static_cast<int64_t>(min(n0 + j, N - 1)) * ldw);
        // per lane: K chunks lane, lane + 32, ...; two chunks of every column
        // (8 independent 16-byte loads) per step, and the next step's loads
        // are issued before this step's arithmetic
        uint4 wv[2][kGemvCols];
#pragma unroll
        for (int j = 0; j < kGemvCols; ++j) {
            wv[0][j] = lane < k8 ? __ldcs(w[j] + lane) : make_uint4(0u, 0u, 0u, 0u);
            wv[1][j] = lane + 32 < k8 ? __ldcs(w[j] + lane + 32) : make_uint4(0u, 0u, 0u, 0u);
        }
        for (int c = lane; c < k8; c += 64) {
            const bool two = c + 32 < k8;
            uint4 wn[2][kGemvCols];
#pragma unroll
            for (int j = 0; j < kGemvCols; ++j) {
                wn[0][j] = c + 64 < k8 ? __ldcs(w[j] + c + 64) : make_uint4(0u, 0u, 0u, 0u);
                wn[1][j] = c + 96 < k8 ? __ldcs(w[j] + c + 96) : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                if (u == 1 && !two) break;
#pragma unroll
                for (int m = 0; m < MR; ++m) {
                    const uint4 av = sA4[m * k8 + c + 32 * u];
                    const uint32_t aw[4] = {av.x, av.y, av.z, av.w};
#pragma unroll
                    for (int j = 0; j < kGemvCols; ++j) {
                        const uint32_t ww[4] = {wv[u][j].x, wv[u][j].y, wv[u][j].z, wv[u][j].w};
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const float2 a2 = unpack_bf16x2(aw[i]);
                            const float2 w2 = unpack_bf16x2(ww[i]);
                            acc[j][m] = fmaf(a2.x, w2.x, fmaf(a2.y, w2.y, acc[j][m]));
                        }
                    }
                }
            }
#pragma unroll
            for (int j = 0; j < kGemvCols; ++j) {
                wv[0][j] = wn[0][j];
                wv[1][j] = wn[1][j];
            }
        }
#pragma unroll
        for (int j = 0; j < kGemvCols; ++j)
#pragma unroll
            for (int m = 0; m < MR; ++m)
#pragma unroll
                for (int o = 16; o; o >>= 1) acc[j][m] += __shfl_xor_sync(0xffffffffu, acc[j][m], o);
        if (lane < kGemvCols * MR) {
            const int j = lane / MR, m = lane % MR;
            const int n = n0 + j;
            if (n < N && m < M) {
                float v = 0.f;
#pragma unroll
                for (int jj = 0; jj < kGemvCols; ++jj)
#pragma unroll
                    for (int mm = 0; mm < MR; ++mm)
                        if (jj == j && mm == m) v = acc[jj][mm];
                if (e.bias) v += __bfloat162float(e.bias[n]);
                if (e.aux) e.aux[static_cast<int64_t>(m) * e.ld_aux + n] = __float2bfloat16_rn(v);
                if (e.act != ACT_NONE && n >= e.act_from) v = e.act == ACT_GELU ? gelu_tanh(v) : silu(v);
                if (e.out_f32)
                    static_cast<float*>(e.out0)[static_cast<int64_t>(m) * e.ld0 + n] = v;
                else
                    static_cast<__nv_bfloat16*>(e.out0)[static_cast<int64_t>(m) * e.ld0 + n] = __float2bfloat16_rn(v);
            }
        }
    }
}

template <int MR>
int launch_gemv(const GemmArgs& a, cudaStream_t stream) {
    const int smem = MR * a.K * 2;
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(gemv_rows_kernel<MR>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
        return set_error(FF_ERR_CUDA, "gemv: cannot set shared memory size");
    const int cols_per_block = (kGemvThreads / 32) * kGemvCols;
    int grid = (a.N + cols_per_block - 1) / cols_per_block;
    const int cap = 2 * num_sms();
    if (grid > cap) grid = cap;
    ProfScope prof(stream, "gemm_bf16", 2.0 * a.M * a.N * static_cast<double>(a.K),
                   2.0 * static_cast<double>(a.N) * a.K + 2.0 * a.M * a.K);
    gemv_rows_kernel<MR><<<grid, kGemvThreads, smem, stream>>>(static_cast<const __nv_bfloat16*>(a.A), a.lda, a.M,
                                                               static_cast<const __nv_bfloat16*>(a.B), a.ldb, a.N,
                                                               a.K, a.epi);
    return check_launch("gemv_rows_kernel");
}

// Passes of at most 8 rows; a row's result is the same in every pass shape
// (per-lane K order and the shuffle reduction do not depend on MR).
int launch_gemv_rows(const GemmArgs& a, cudaStream_t stream) {
    for (int m0 = 0; m0 < a.M; m0 += kGemvMaxRows) {
        GemmArgs p = a;
        p.M = a.M - m0 < kGemvMaxRows ? a.M - m0 : kGemvMaxRows;
        p.A = static_cast<const __nv_bfloat16*>(a.A) + static_cast<int64_t>(m0) * a.lda;
        p.epi.out0 = a.epi.out_f32 ? static_cast<void*>(static_cast<float*>(a.epi.out0) + m0 * a.epi.ld0)
                                   : static_cast<void*>(static_cast<__nv_bfloat16*>(a.epi.out0) + m0 * a.epi.ld0);
        if (a.epi.aux) p.epi.aux = a.epi.aux + m0 * a.epi.ld_aux;
        int rc;
        if (p.M <= 1) rc = launch_gemv<1>(p, stream);
        else if (p.M <= 2) rc = launch_gemv<2>(p, stream);
        else if (p.M <= 4) rc = launch_gemv<4>(p, stream);
        else rc = launch_gemv<8>(p, stream);
        if (rc) return rc;
    }
    return FF_OK;
}

int check_args(const GemmArgs& a) {
    const GemmEpilogue& e = a.epi;
    const int M = a.M, N = a.N, K = a.K;
    if (!a.A || !a.B) return set_error(FF_ERR_INVALID_ARG, "gemm: null operand");
    if (M <= 0 || N <= 0 || K <= 0) return set_error(FF_ERR_INVALID_ARG, "gemm: bad shape %d x %d x %d", M, N, K);
    if (N % 32 != 0) return set_error(FF_ERR_UNSUPPORTED, "gemm: N=%d not a multiple of 32", N);
    if (K % 8 != 0 || a.lda % 8 != 0 || a.ldb % 8 != 0 || a.lda < (a.a_mn ? M : K) || a.ldb < (a.b_mn ? N : K))
        return set_error(FF_ERR_UNSUPPORTED, "gemm: K/ld must be multiples of 8 and cover the rows (K=%d lda=%lld ldb=%lld)",
                         K, (long long)a.lda, (long long)a.ldb);
    if (e.bias && !aligned16(e.bias)) return set_error(FF_ERR_INVALID_ARG, "gemm: bias not 16-byte aligned");
    if (e.epi == EPI_GATED_RESIDUAL) {
        if (!e.resid || e.rows_per_sample <= 0 || !aligned16(e.resid) || (e.gate && !aligned16(e.gate)) ||
            (e.resid_out && !aligned16(e.resid_out)) || e.ld_resid % 4 || e.ld_gate % 4)
            return set_error(FF_ERR_INVALID_ARG, "gemm: bad gated-residual epilogue");
    } else {
        if (!e.out0 || !aligned16(e.out0)) return set_error(FF_ERR_INVALID_ARG, "gemm: bad output");
        const int vec = e.out_f32 ? 4 : 8;
        if (e.ld0 % vec) return set_error(FF_ERR_INVALID_ARG, "gemm: output ld not vector aligned");
        if (e.split_n < N) {
            if (e.split_n % 32 || !e.out1 || !aligned16(e.out1) || e.ld1 % vec || e.col1 % vec)
                return set_error(FF_ERR_INVALID_ARG, "gemm: bad split output");
        }
    }
    if (e.act != ACT_NONE && e.act_from % 32) return set_error(FF_ERR_INVALID_ARG, "gemm: act_from % 32 != 0");
    if (e.aux && (!aligned16(e.aux) || e.ld_aux % 8 || e.ld_aux < N))
        return set_error(FF_ERR_INVALID_ARG, "gemm: bad pre-activation copy");
    if (e.gelu_pre && (!aligned16(e.gelu_pre) || e.ld_pre % 8 || e.act_from % 32 || e.act != ACT_NONE ||
                       e.epi != EPI_STORE || e.qk_cols > 0 || e.ld_pre < N - e.act_from))
        return set_error(FF_ERR_INVALID_ARG, "gemm: bad activation-backward epilogue");
    if (e.qk_cols > 0) {
        // whole heads per 256-wide tile: head_dim | 256 and qk_cols | 256
        if (e.epi != EPI_STORE || e.out_f32 || (e.head_dim != 64 && e.head_dim != 128) || e.qk_cols % 256 ||
            e.qk_cols > N || e.qk_cols > e.split_n || !e.q_scale || !e.k_scale || N <= 128 ||
            (e.rope_cs && (e.n_img <= 0 || e.grid_h <= 0 || e.grid_w <= 0 || e.rope_row0 < 0)))
            return set_error(FF_ERR_INVALID_ARG, "gemm: bad fused QK-norm epilogue");
    }
    return FF_OK;
}

}  // namespace

// Calls f with the operand layout as a compile-time constant.
template <class F>
int with_layout(int layout, F&& f) {
    switch (layout) {
        case 0: return f(std::integral_constant<int, 0>{});
        case 1: return f(std::integral_constant<int, 1>{});
        case 2: return f(std::integral_constant<int, 2>{});
        default: return f(std::integral_constant<int, 3>{});
    }
}

int gemm_bf16_group(const GemmArgs* p, int n, cudaStream_t stream) {
    if (!p || n < 1 || n > 2) return set_error(FF_ERR_INVALID_ARG, "gemm: 1 or 2 problems per launch");
    bool qk = false;
    for (int i = 0; i < n; ++i) {
        const int rc = check_args(p[i]);
        if (rc) return rc;
        qk = qk || p[i].epi.qk_cols > 0;
    }
    if (n == 2 && (p[0].epi.epi == EPI_GATED_RESIDUAL) != (p[1].epi.epi == EPI_GATED_RESIDUAL))
        return set_error(FF_ERR_INVALID_ARG, "gemm: grouped problems must share the epilogue kind");
    // two-SM 256 x 256 tiles when every problem's N is a multiple of 256 and
    // there is enough work for them
    bool pair = true;
    int max_m = 0;
    for (int i = 0; i < n; ++i) {
        pair = pair && p[i].N % 256 == 0 && p[i].epi.rows_gemv == 0;
        max_m = p[i].M > max_m ? p[i].M : max_m;
    }
    const int layout = p[0].a_mn | (p[0].b_mn << 1);
    if (n == 2 && (p[1].a_mn | (p[1].b_mn << 1)) != layout)
        return set_error(FF_ERR_INVALID_ARG, "gemm: grouped problems must share the operand layout");
    if (pair && max_m >= 512) return with_layout(layout, [&](auto L) { return launch_pair<L.value>(p, n, stream); });
    if (n == 2 || qk) {
        for (int i = 0; i < n; ++i)
            if (p[i].N <= 128) return set_error(FF_ERR_UNSUPPORTED, "gemm: grouped / fused problems need N > 128");
        return with_layout(layout, [&](auto L) { return launch<256, L.value>(p, n, stream); });
    }
    const GemmArgs& a = p[0];
    const bool gemv_ok = !a.a_mn && !a.b_mn && a.K <= kGemvMaxK && a.epi.epi == EPI_STORE && a.epi.split_n >= a.N &&
                         a.epi.qk_cols == 0 && !a.epi.gelu_pre &&
                         aligned16(a.A) && aligned16(a.B) && a.lda % 8 == 0 && a.ldb % 8 == 0;
    if (a.epi.rows_gemv && !gemv_ok) return set_error(FF_ERR_UNSUPPORTED, "gemm: rows_gemv needs K <= 8192 and a plain store");
    if (gemv_ok && (a.epi.rows_gemv || a.M <= kGemvMaxRows)) return launch_gemv_rows(a, stream);
    // narrow tiles when wide ones would leave most SMs idle
    const int64_t mblocks = (a.M + BM - 1) / BM;
    const bool few = mblocks * ((a.N + 255) / 256) < num_sms() / 2;
    if (a.N <= 64 || few) return with_layout(layout, [&](auto L) { return launch<64, L.value>(p, 1, stream); });
    if (a.N <= 128) return with_layout(layout, [&](auto L) { return launch<128, L.value>(p, 1, stream); });
    return with_layout(layout, [&](auto L) { return launch<256, L.value>(p, 1, stream); });
}

int gemm_bf16(const void* A, int64_t lda, const void* B, int64_t ldb, int M, int N, int K, const GemmEpilogue& e,
              cudaStream_t stream) {
    const GemmArgs a{A, lda, B, ldb, M, N, K, e};
    return gemm_bf16_group(&a, 1, stream);
}

}  // namespace ff

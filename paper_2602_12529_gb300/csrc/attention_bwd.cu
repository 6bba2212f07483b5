// attention_bwd.cu -- backward of the attention O = softmax(Q K^T / sqrt(d)) V
// (d = 64 or 128) on tcgen05, for the training pass that follows the rollout
// (paper Sec. 3.1: the policy gradient through the velocity network).  Queries
// come from up to two query segments and keys / values from up to two key
// segments, each with its own source buffer and columns: the joint
// [text; image] self-attention of the MMDiT (the same rows on both sides) and
// the WAN block's cross-attention (latent queries, text keys and values).
//
// With P = softmax(S), S = Q K^T a (a = 1/sqrt(d)) per (sample, head) and the
// forward's per-row log-sum-exp (base 2, lse2 = log2 sum_j 2^(S_ij log2 e)):
//   P_ij = 2^(S_ij log2(e) - lse2_i),  D_i = sum_c dO_ic O_ic,
//   dP = dO V^T,  dS = P (dP - D),  dV = P^T dO,  dQ = a dS K,  dK = a dS^T Q.
// Three kernels:
//   delta   D_i, one warp per (row, head), into the workspace (lse layout);
//   dq      one 128-row query tile per CTA, K/V tiles streamed: S = Q K_j^T
//           and dP = dO V_j^T in TMEM (whole 128-key tiles), dS to its own
//           TMEM columns as bf16, then dQ += dS K_j with dS read from TMEM
//           and K_j taken as an MN-major operand (the same shared-memory tile
//           feeds S as K-major);
//   dkdv    one 128-key tile per CTA, query tiles streamed: S^T = K Q_i^T and
//           dP^T = V dO_i^T in TMEM (whole 128-query tiles), P^T and dS^T
//           written over them, then dV += P^T dO_i and dK += dS^T Q_i (Q_i,
//           dO_i as MN-major operands); lse and D of the query tile arrive by
//           bulk copies with the tiles.
// Query (key) rows past a segment's end read neighbouring or zero-filled
// rows; their columns are selected to zero (never multiplied, so padding
// can hold anything) and their rows are not stored.  Every wait is bounded;
// on a timeout a kernel records the status word, drains its tensor-core
// work, frees TMEM and returns.
#include "internal.h"
#include "ptx.cuh"

namespace ff {
namespace {

constexpr int kT = 128;                        // rows of a query / key tile
constexpr int kSlotsDq = 5;                     // streamed K / V tiles in flight (dQ kernel):
constexpr int kKSlots = 3, kVSlots = 2;         //   three K slots, then two V slots
static_assert(kKSlots + kVSlots == kSlotsDq, "dQ slots");
constexpr int kSlotsDkdv = 4;                   // streamed Q / dO tiles in flight (dK dV kernel)
constexpr int kThreads = 320;                   // producer, MMA, 8 elementwise warps (two per TMEM lane quarter)
constexpr int kEw = 8;                          // elementwise warps
constexpr int kBarBytes = 256;

struct BwdParams {
    int nq[2], nk[2];      // tokens per sample of each query / key segment
    int qtiles0, ktiles0;  // 128-row tiles of query / key segment 0 (segment 1's follow)
    int q_col, k_col, v_col;   // first column of head 0's q, k, v in the source rows
    float scale_log2;      // log2(e) / sqrt(d)
    float scale;           // 1 / sqrt(d)
    const float* lse;      // [B, heads, lse_rows] base-2 log-sum-exp of the forward
    const float* delta;    // D in the same layout
    int lse_rows, lse_base[2];
    __nv_bfloat16* dq[2];  // head h at column h d
    int64_t ldq[2];
    __nv_bfloat16 *dk[2], *dv[2];
    int64_t ldkv[2];
};

// The streamed tiles of step i (K_i and V_i in the dQ kernel, Q_i and dO_i
// in the dK dV kernel; item 2 i and 2 i + 1 of the ring, in slots n % S)
// arrive on one barrier, and one commit after the step's last MMA that reads
// them releases both slots.  A parity wait on a ring of four barriers is
// unambiguous while its waiter is at most three phases behind, which the
// ring's slot count guarantees; the two-phase barriers are waited in
// lockstep with their producers.
struct Bars {
    uint64_t fixed_full;           // the CTA's own tiles landed
    uint64_t grp_full[4];          // producer -> MMA: both streamed tiles of step i landed (entry i % 4)
    uint64_t rel[4];               // MMA -> producer (and dQ's elementwise warps): step i's MMAs are done
    uint64_t s0_full;              // MMA -> elementwise: S^T and dP^T of the step in TMEM (dK dV kernel)
    uint64_t s0_ring[4];           // MMA -> elementwise and producer: S and dP of step j in TMEM (entry
                                   // j % 4), so V_j is read (dQ kernel)
    uint64_t p_full[2];            // elementwise -> MMA: dQ kernel: [0] S / dP read, [1] dS written;
                                   // dK dV kernel: [0] P^T and dS^T written
    uint64_t done;                 // MMA -> elementwise: the accumulators are final
    uint64_t drain;
    uint32_t tmem_slot;
    int abort_flag;
};

__device__ __forceinline__ void bulk_load_1d(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}

// Stores `cols` fp32 TMEM columns of this thread's row as bf16 (times mul).
__device__ __forceinline__ void store_row_bf16(uint32_t taddr, float mul, __nv_bfloat16* dst, bool live,
                                               int cols) {
#pragma unroll 1
    for (int c = 0; c < cols; c += 32) {
        uint32_t o[32];
        tmem_ld_x32(taddr + c, o);
        tmem_ld_wait();
        if (live) {
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float* f = reinterpret_cast<const float*>(o) + 8 * k;
                *reinterpret_cast<uint4*>(dst + c + 8 * k) =
                    make_uint4(pack_bf16x2(f[0] * mul, f[1] * mul), pack_bf16x2(f[2] * mul, f[3] * mul),
                               pack_bf16x2(f[4] * mul, f[5] * mul), pack_bf16x2(f[6] * mul, f[7] * mul));
            }
        }
    }
}

// D_i = sum_c dO_ic O_ic: one warp per (token row, head), HD / 32 columns per
// lane.  With the forward's low parts (o_lo), O = o + o_lo: D = rowsum(P dP)
// subtracts nearly equal terms when the rows of V are close to each other,
// and bf16 O alone would leave a relative error of 2^-9 |dO| |O| in D.
template <int HD>
__global__ void __launch_bounds__(256) attn_bwd_delta_kernel(int B, int heads, int n0, int n1,
                                                             const __nv_bfloat16* o0, const __nv_bfloat16* do0,
                                                             const __nv_bfloat16* o1, const __nv_bfloat16* do1,
                                                             int64_t ldo0, int64_t ldo1, int64_t ldg0, int64_t ldg1,
                                                             const __nv_bfloat16* ol0, const __nv_bfloat16* ol1,
                                                             int64_t ldl0, int64_t ldl1, int lse_rows, int base1,
                                                             float* delta) {
    const int64_t w = (static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    const int64_t rows0 = static_cast<int64_t>(B) * n0;
    const int64_t total = (rows0 + static_cast<int64_t>(B) * n1) * heads;
    if (w >= total) return;
    const int h = static_cast<int>(w % heads);
    const int64_t r = w / heads;                    // token row over both segments
    const bool s1 = r >= rows0;
    const int64_t rr = s1 ? r - rows0 : r;
    const int n = s1 ? n1 : n0;
    const int b = static_cast<int>(rr / n);
    const int row = static_cast<int>(rr - static_cast<int64_t>(b) * n);
    constexpr int E = HD / 32;
    const __nv_bfloat16* o = (s1 ? o1 : o0) + rr * (s1 ? ldo1 : ldo0) + h * HD + lane * E;
    const __nv_bfloat16* g = (s1 ? do1 : do0) + rr * (s1 ? ldg1 : ldg0) + h * HD + lane * E;
    const __nv_bfloat16* olb = s1 ? ol1 : ol0;
    const __nv_bfloat16* ol = olb ? olb + rr * (s1 ? ldl1 : ldl0) + h * HD + lane * E : nullptr;
    float s = 0.f;
#pragma unroll
    for (int e = 0; e < E; e += 2) {
        float2 of = unpack_bf16x2(*reinterpret_cast<const uint32_t*>(o + e));
        if (ol) {
            const float2 lf = unpack_bf16x2(*reinterpret_cast<const uint32_t*>(ol + e));
            of.x += lf.x;
            of.y += lf.y;
        }
        const float2 gf = unpack_bf16x2(*reinterpret_cast<const uint32_t*>(g + e));
        s = fmaf(of.x, gf.x, fmaf(of.y, gf.y, s));
    }
#pragma unroll
    for (int k = 16; k; k >>= 1) s += __shfl_xor_sync(0xffffffffu, s, k);
    if (lane == 0) delta[(static_cast<int64_t>(b) * heads + h) * lse_rows + (s1 ? base1 : 0) + row] = s;
}

// ------------------------------------------------------------------ dQ
// One 128-row query tile per CTA; K / V tiles streamed through the ring.
// TMEM: S = Q K_j^T at columns 0..127 and dP = dO V_j^T at 128..255 (fp32,
// the whole 128-key tile: N = 128 MMAs), dS as bf16 pairs at 256..319, dQ
// (d columns) at 384.  Per key tile j the elementwise warps load their S and
// dP columns into registers and hand the buffer back at once, so the MMAs of
// tile j + 1 (S, dP) run while they form dS_j; dS_j goes to its own columns,
// and dQ += dS_j K_j follows.  The MMA thread's work per tile: three waits
// (S / dP consumed, operands of j + 1, dS_j written) and two commits (S / dP
// of j + 1 done, which also frees V_j+1's slot; dQ_j done, which frees K_j's
// slot and the dS columns).  Shared memory: Q tile, dO tile, then three
// K slots and two V slots: V_j is free once dP_j is done, K_j only once dQ_j
// is, so separate rings let V_j + 2 load a whole tile earlier than one ring
// of K / V pairs would (a clock trace of the single ring showed the MMA
// thread waiting 1300-1700 cycles per 3600-cycle tile for V).
template <int HD>
__global__ void __launch_bounds__(kThreads, 1)
attn_bwd_dq_kernel(const __grid_constant__ CUtensorMap tm_q0, const __grid_constant__ CUtensorMap tm_q1,
                   const __grid_constant__ CUtensorMap tm_kv0, const __grid_constant__ CUtensorMap tm_kv1,
                   const __grid_constant__ CUtensorMap tm_do0, const __grid_constant__ CUtensorMap tm_do1,
                   const BwdParams p, int* status) {
    constexpr int S_ = kSlotsDq;
    constexpr int kTileBytes = kT * HD * 2;              // one bf16 tile: HD / 64 boxes of 128 rows x 64 columns
    constexpr int NB = HD / 64;
    constexpr uint32_t kColS = 0, kColP = kT, kColDs = 2 * kT, kColDq = 384;
    extern __shared__ __align__(1024) uint8_t smem[];
    uint8_t* sQ = smem;
    uint8_t* sdO = smem + kTileBytes;
    uint8_t* sKV = smem + 2 * kTileBytes;                     // [S_][tile]
    Bars& bar = *reinterpret_cast<Bars*>(sKV + S_ * kTileBytes);
    volatile int* abort_flag = &bar.abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int b = blockIdx.z, h = blockIdx.y;
    const int seg = blockIdx.x < p.qtiles0 ? 0 : 1;
    const int q0 = (blockIdx.x - (seg ? p.qtiles0 : 0)) * kT;
    const int nt0 = (p.nk[0] + kT - 1) / kT;
    const int ntiles = nt0 + (p.nk[1] + kT - 1) / kT;
    if (threadIdx.x == 0) {
        *abort_flag = 0;
        if (smem_u32(smem) & 1023u) {
            report_status(status, kStatusBadArgument);
            *abort_flag = 1;
        }
        mbar_init(&bar.fixed_full, 1);
        for (int g = 0; g < 4; ++g) {
            mbar_init(&bar.grp_full[g], 2);
            mbar_init(&bar.rel[g], 1);
        }
        for (int g = 0; g < 4; ++g) mbar_init(&bar.s0_ring[g], 1);   // S and dP of tile j in TMEM
        mbar_init(&bar.p_full[0], kEw);    // every elementwise warp has read S / dP of tile j
        mbar_init(&bar.p_full[1], kEw);    // every elementwise warp has written its dS_j
        mbar_init(&bar.done, 1);
        mbar_init(&bar.drain, 1);
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&bar.tmem_slot, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = bar.tmem_slot;
    auto fail = [&]() {
        report_status(status, kStatusWaitTimeout);
        *abort_flag = 1;
    };
    if (*abort_flag) {
    } else if (warp == 0 && lane == 0) {
        // ---- producer: Q and dO of this tile, then K_0, V_0, K_1, ...: K_j
        // into K slot j % 3 once dQ_j-3 is done, V_j into V slot j % 2 once
        // S / dP of tile j - 2 are done
        const CUtensorMap* tq = seg ? &tm_q1 : &tm_q0;
        const CUtensorMap* td = seg ? &tm_do1 : &tm_do0;
        mbar_arrive_expect_tx(&bar.fixed_full, 2 * kTileBytes);
        for (int c = 0; c < NB; ++c) {
            tma_load_2d(sQ + c * (kT * 128), tq, &bar.fixed_full, p.q_col + h * HD + c * 64, b * p.nq[seg] + q0);
            tma_load_2d(sdO + c * (kT * 128), td, &bar.fixed_full, h * HD + c * 64, b * p.nq[seg] + q0);
        }
        for (int j = 0; j < ntiles; ++j) {
            const int ks = j < nt0 ? 0 : 1;
            const int row = b * p.nk[ks] + (j - (ks ? nt0 : 0)) * kT;
            uint64_t* fb = &bar.grp_full[j & 3];
            if (j >= kKSlots && !mbar_wait(&bar.rel[(j - kKSlots) & 3], ((j - kKSlots) >> 2) & 1)) { fail(); break; }
            uint8_t* dk = sKV + (j % kKSlots) * kTileBytes;
            mbar_arrive_expect_tx(fb, kTileBytes);
            for (int c = 0; c < NB; ++c)
                tma_load_2d(dk + c * (kT * 128), ks ? &tm_kv1 : &tm_kv0, fb, p.k_col + h * HD + c * 64, row);
            if (j >= kVSlots && !mbar_wait(&bar.s0_ring[(j - kVSlots) & 3], ((j - kVSlots) >> 2) & 1)) { fail(); break; }
            uint8_t* dv = sKV + (kKSlots + j % kVSlots) * kTileBytes;
            mbar_arrive_expect_tx(fb, kTileBytes);
            for (int c = 0; c < NB; ++c)
                tma_load_2d(dv + c * (kT * 128), ks ? &tm_kv1 : &tm_kv0, fb, p.v_col + h * HD + c * 64, row);
        }
    } else if (warp == 1 && lane == 0) {
        // ---- MMA issuer
        constexpr uint32_t idesc_s = idesc_bf16_f32(kT, kT);
        constexpr uint32_t idesc_q = idesc_bf16_f32(kT, HD) | (1u << 16);   // B = K_j, MN-major
        bool ok = mbar_wait(&bar.fixed_full, 0);
        if (!ok) fail();
        const uint64_t dq_ = smem_desc_k_sw128(smem_u32(sQ));
        const uint64_t ddo = smem_desc_k_sw128(smem_u32(sdO));
        auto wait_kv = [&](int j) { return mbar_wait(&bar.grp_full[j & 3], (j >> 2) & 1); };
        // S = Q K_j^T and dP = dO V_j^T of the whole key tile
        auto issue_sdp = [&](int j) {
            const uint64_t dk = smem_desc_k_sw128(smem_u32(sKV + (j % kKSlots) * kTileBytes));
            const uint64_t dv = smem_desc_k_sw128(smem_u32(sKV + (kKSlots + j % kVSlots) * kTileBytes));
#pragma unroll
            for (int k = 0; k < HD / 16; ++k) {
                const uint32_t off = ((k / 4) * (kT * 128) + (k % 4) * 32) >> 4;
                tc_mma_bf16(tmem + kColS, dq_ + off, dk + off, idesc_s, k != 0 ? 1u : 0u);
                tc_mma_bf16(tmem + kColP, ddo + off, dv + off, idesc_s, k != 0 ? 1u : 0u);
            }
            tc_commit(&bar.s0_ring[j & 3]);
        };
        if (ok && !wait_kv(0)) { fail(); ok = false; }
        if (ok) {
            tc_fence_after();
            issue_sdp(0);
        }
        for (int j = 0; ok && j < ntiles; ++j) {
            // the elementwise warps hold S_j / dP_j in registers: the next tile's may go in
            if (!mbar_wait(&bar.p_full[0], j & 1)) { fail(); ok = false; break; }
            if (j + 1 < ntiles) {
                if (!wait_kv(j + 1)) { fail(); ok = false; break; }
                tc_fence_after();
                issue_sdp(j + 1);
            }
            if (!mbar_wait(&bar.p_full[1], j & 1)) { fail(); ok = false; break; }
            tc_fence_after();
            // dQ += dS_j K_j: dS (keys 16 k.. at columns 8 k..) from TMEM, K_j rows as [keys (K) x d (N)]
            const uint64_t dkm = smem_desc_mn_sw128(smem_u32(sKV + (j % kKSlots) * kTileBytes), kT * 128);
#pragma unroll
            for (int k = 0; k < kT / 16; ++k)
                tc_mma_bf16_ts(tmem + kColDq, tmem + kColDs + k * 8, dkm + static_cast<uint64_t>(k * (2048 >> 4)),
                               idesc_q, (j | k) != 0 ? 1u : 0u);
            tc_commit(&bar.rel[j & 3]);   // K_j and the dS columns are free again
        }
        if (ok) tc_commit(&bar.done);
        tc_commit(&bar.drain);
        if (!mbar_wait(&bar.drain, 0)) report_status(status, kStatusWaitTimeout);
    } else if (warp >= 2) {
        // ---- elementwise: thread = query row = TMEM lane; the two warps of a
        // lane quarter take 64 key columns each of a tile
        const int q = warp & 3;
        const int cg = (warp - 2) >> 2;
        const int r = q * 32 + lane;
        const int row = q0 + r;
        const uint32_t tS = tmem + (static_cast<uint32_t>(q * 32) << 16);
        const int64_t li = (static_cast<int64_t>(b) * gridDim.y + h) * p.lse_rows + p.lse_base[seg] + row;
        const bool live = row < p.nq[seg];
        const bool full_rows = q0 + kT <= p.nq[seg];   // every row of the tile is real (warp-uniform)
        const float lse = live ? p.lse[li] : 0.f;
        const float dd = live ? p.delta[li] : 0.f;
        bool ok = true;
        for (int j = 0; j < ntiles; ++j) {
            if (!mbar_wait(&bar.s0_ring[j & 3], (j >> 2) & 1)) { fail(); ok = false; break; }
            tc_fence_after();
            uint32_t sr[64], pr_[64];
            tmem_ld_x32(tS + kColS + cg * 64, *reinterpret_cast<uint32_t(*)[32]>(&sr[0]));
            tmem_ld_x32(tS + kColS + cg * 64 + 32, *reinterpret_cast<uint32_t(*)[32]>(&sr[32]));
            tmem_ld_x32(tS + kColP + cg * 64, *reinterpret_cast<uint32_t(*)[32]>(&pr_[0]));
            tmem_ld_x32(tS + kColP + cg * 64 + 32, *reinterpret_cast<uint32_t(*)[32]>(&pr_[32]));
            tmem_ld_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bar.p_full[0]);   // S_j / dP_j consumed: the buffer may be refilled
            const int ks = j < nt0 ? 0 : 1;
            // key columns < valid of this warp's 64 are real
            const int valid = p.nk[ks] - (j - (ks ? nt0 : 0)) * kT - cg * 64;
            if (valid >= 64 && full_rows) {
                // every column and row real: paired fp32 arithmetic, no selects
                const float2 c2 = make_float2(p.scale_log2, p.scale_log2), nl2 = make_float2(-lse, -lse);
                const float2 nd2 = make_float2(-dd, -dd);
#pragma unroll
                for (int i = 0; i < 64; i += 2) {
                    const float2 x = __ffma2_rn(make_float2(__uint_as_float(sr[i]), __uint_as_float(sr[i + 1])), c2, nl2);
                    const float2 dp = __fadd2_rn(make_float2(__uint_as_float(pr_[i]), __uint_as_float(pr_[i + 1])), nd2);
                    const float2 ds = __fmul2_rn(make_float2(ex2(x.x), ex2(x.y)), dp);
                    sr[i / 2] = pack_bf16x2(ds.x, ds.y);
                }
            } else {
#pragma unroll
                for (int i = 0; i < 64; i += 2) {
                    float ds[2];
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        const float pv = ex2(fmaf(__uint_as_float(sr[i + e]), p.scale_log2, -lse));
                        ds[e] = (i + e < valid && live) ? pv * (__uint_as_float(pr_[i + e]) - dd) : 0.f;
                    }
                    sr[i / 2] = pack_bf16x2(ds[0], ds[1]);
                }
            }
            // dS_j over the dS columns once dQ_j-1 has read them
            if (j > 0 && !mbar_wait(&bar.rel[(j - 1) & 3], ((j - 1) >> 2) & 1)) { fail(); ok = false; break; }
            tc_fence_after();
            tmem_st_x32(tS + kColDs + cg * 32, sr);
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bar.p_full[1]);
        }
        if (ok && mbar_wait(&bar.done, 0)) {
            tc_fence_after();
            store_row_bf16(tS + kColDq + cg * (HD / 2), p.scale,
                           p.dq[seg] + (static_cast<int64_t>(b) * p.nq[seg] + row) * p.ldq[seg] + h * HD + cg * (HD / 2),
                           live, HD / 2);
        } else if (ok) {
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
        tmem_dealloc(tmem, 512);
    }
}

// ------------------------------------------------------------------ dK, dV
// TMEM: S^T = K Q_i^T at columns 0..127 and dP^T = V dO_i^T at 128..255
// (fp32, the whole 128-query tile: N = 128 MMAs); each elementwise warp
// writes its 64 columns of P^T and dS^T as bf16 pairs over the first 32 of
// its own S^T / dP^T columns; dV at 256, dK at 256 + d.  Per query tile i
// the MMA thread issues dV += P^T dO_i and dK += dS^T Q_i, then at once
// S^T / dP^T of tile i + 1: the tensor pipe runs one thread's MMAs in issue
// order, so they overwrite P^T / dS^T only after dV / dK have read them.  Its
// work per tile: two waits (P^T / dS^T written, operands of i + 1) and two
// commits (tile i's slots free; S^T / dP^T of i + 1 ready).  Shared memory:
// the K and V tiles of this CTA, then a ring of Q_i / dO_i tiles, then lse /
// D of each streamed query tile.
template <int HD>
__global__ void __launch_bounds__(kThreads, 1)
attn_bwd_dkdv_kernel(const __grid_constant__ CUtensorMap tm_q0, const __grid_constant__ CUtensorMap tm_q1,
                     const __grid_constant__ CUtensorMap tm_kv0, const __grid_constant__ CUtensorMap tm_kv1,
                     const __grid_constant__ CUtensorMap tm_do0, const __grid_constant__ CUtensorMap tm_do1,
                     const BwdParams p, int* status) {
    constexpr int S_ = kSlotsDkdv;
    constexpr int kTileBytes = kT * HD * 2;
    constexpr int NB = HD / 64;
    extern __shared__ __align__(1024) uint8_t smem[];
    uint8_t* sK = smem;
    uint8_t* sV = smem + kTileBytes;
    uint8_t* sQD = smem + 2 * kTileBytes;                     // [S_][tile]: Q_i, dO_i, Q_i+1, ...
    float* sLD = reinterpret_cast<float*>(sQD + S_ * kTileBytes);   // [S_ / 2][2][kT]: lse, D
    Bars& bar = *reinterpret_cast<Bars*>(reinterpret_cast<uint8_t*>(sLD) + (S_ / 2) * 2 * kT * 4);
    volatile int* abort_flag = &bar.abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int b = blockIdx.z, h = blockIdx.y;
    const int seg = blockIdx.x < p.ktiles0 ? 0 : 1;
    const int k0 = (blockIdx.x - (seg ? p.ktiles0 : 0)) * kT;
    const int nt0 = (p.nq[0] + kT - 1) / kT;
    const int ntiles = nt0 + (p.nq[1] + kT - 1) / kT;
    const int64_t lrow = (static_cast<int64_t>(b) * gridDim.y + h) * p.lse_rows;
    if (threadIdx.x == 0) {
        *abort_flag = 0;
        if (smem_u32(smem) & 1023u) {
            report_status(status, kStatusBadArgument);
            *abort_flag = 1;
        }
        mbar_init(&bar.fixed_full, 1);
        for (int g = 0; g < 4; ++g) {
            mbar_init(&bar.grp_full[g], 2);
            mbar_init(&bar.rel[g], 1);
        }
        mbar_init(&bar.s0_full, 1);
        for (int s = 0; s < 2; ++s) mbar_init(&bar.p_full[s], kEw);
        mbar_init(&bar.done, 1);
        mbar_init(&bar.drain, 1);
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&bar.tmem_slot, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = bar.tmem_slot;
    auto fail = [&]() {
        report_status(status, kStatusWaitTimeout);
        *abort_flag = 1;
    };
    if (*abort_flag) {
    } else if (warp == 0 && lane == 0) {
        // ---- producer: K and V of this tile, then per query tile i its Q_i
        // and dO_i (one slot each) with lse_i / D_i riding on dO_i's barrier
        const CUtensorMap* tk = seg ? &tm_kv1 : &tm_kv0;
        mbar_arrive_expect_tx(&bar.fixed_full, 2 * kTileBytes);
        for (int c = 0; c < NB; ++c) {
            tma_load_2d(sK + c * (kT * 128), tk, &bar.fixed_full, p.k_col + h * HD + c * 64, b * p.nk[seg] + k0);
            tma_load_2d(sV + c * (kT * 128), tk, &bar.fixed_full, p.v_col + h * HD + c * 64, b * p.nk[seg] + k0);
        }
        for (int n = 0; n < 2 * ntiles; ++n) {
            const int s = n % S_;
            if (n >= S_) {   // slot s held a tile of step (n - S_) / 2
                const int r = (n - S_) >> 1;
                if (!mbar_wait(&bar.rel[r & 3], (r >> 2) & 1)) { fail(); break; }
            }
            uint64_t* fb = &bar.grp_full[(n >> 1) & 3];
            const int i = n >> 1;
            const int qs = i < nt0 ? 0 : 1;
            const int qi = (i - (qs ? nt0 : 0)) * kT;
            const int row = b * p.nq[qs] + qi;
            uint8_t* dst = sQD + s * kTileBytes;
            if (n & 1) {
                float* ld = sLD + (s >> 1) * 2 * kT;
                mbar_arrive_expect_tx(fb, kTileBytes + 2 * kT * 4);
                for (int c = 0; c < NB; ++c)
                    tma_load_2d(dst + c * (kT * 128), qs ? &tm_do1 : &tm_do0, fb, h * HD + c * 64, row);
                bulk_load_1d(ld, p.lse + lrow + p.lse_base[qs] + qi, kT * 4, fb);
                bulk_load_1d(ld + kT, p.delta + lrow + p.lse_base[qs] + qi, kT * 4, fb);
            } else {
                mbar_arrive_expect_tx(fb, kTileBytes);
                for (int c = 0; c < NB; ++c)
                    tma_load_2d(dst + c * (kT * 128), qs ? &tm_q1 : &tm_q0, fb, p.q_col + h * HD + c * 64, row);
            }
        }
    } else if (warp == 1 && lane == 0) {
        // ---- MMA issuer
        constexpr uint32_t idesc_s = idesc_bf16_f32(kT, kT);
        constexpr uint32_t idesc_g = idesc_bf16_f32(kT, HD) | (1u << 16);   // B = Q_i / dO_i, MN-major
        bool ok = mbar_wait(&bar.fixed_full, 0);
        if (!ok) fail();
        const uint64_t dk_ = smem_desc_k_sw128(smem_u32(sK));
        const uint64_t dv_ = smem_desc_k_sw128(smem_u32(sV));
        auto wait_qd = [&](int i) { return mbar_wait(&bar.grp_full[i & 3], (i >> 2) & 1); };
        // S^T = K Q_i^T and dP^T = V dO_i^T of the whole query tile
        auto issue_sdp = [&](int i) {
            const uint64_t dq_ = smem_desc_k_sw128(smem_u32(sQD + ((2 * i) % S_) * kTileBytes));
            const uint64_t ddo = smem_desc_k_sw128(smem_u32(sQD + ((2 * i + 1) % S_) * kTileBytes));
#pragma unroll
            for (int k = 0; k < HD / 16; ++k) {
                const uint32_t off = ((k / 4) * (kT * 128) + (k % 4) * 32) >> 4;
                tc_mma_bf16(tmem, dk_ + off, dq_ + off, idesc_s, k != 0 ? 1u : 0u);
                tc_mma_bf16(tmem + kT, dv_ + off, ddo + off, idesc_s, k != 0 ? 1u : 0u);
            }
            tc_commit(&bar.s0_full);
        };
        if (ok && !wait_qd(0)) { fail(); ok = false; }
        if (ok) {
            tc_fence_after();
            issue_sdp(0);
        }
        for (int i = 0; ok && i < ntiles; ++i) {
            if (!mbar_wait(&bar.p_full[0], i & 1)) { fail(); ok = false; break; }
            tc_fence_after();
            const uint64_t dqm = smem_desc_mn_sw128(smem_u32(sQD + ((2 * i) % S_) * kTileBytes), kT * 128);
            const uint64_t ddom = smem_desc_mn_sw128(smem_u32(sQD + ((2 * i + 1) % S_) * kTileBytes), kT * 128);
#pragma unroll
            for (int k = 0; k < kT / 16; ++k) {
                const uint64_t step = static_cast<uint64_t>(k * (2048 >> 4));
                const uint32_t acc = (i | k) != 0 ? 1u : 0u;
                // queries 16 k.. : each warp's 64 queries packed over the first 32 of its columns
                const uint32_t a = tmem + (k >> 2) * 64 + (k & 3) * 8;
                tc_mma_bf16_ts(tmem + 256, a, ddom + step, idesc_g, acc);             // dV += P^T dO
                tc_mma_bf16_ts(tmem + 256 + HD, a + kT, dqm + step, idesc_g, acc);    // dK += dS^T Q
            }
            tc_commit(&bar.rel[i & 3]);   // Q_i, dO_i, lse_i and D_i read for the last time
            if (i + 1 < ntiles) {
                if (!wait_qd(i + 1)) { fail(); ok = false; break; }
                tc_fence_after();
                issue_sdp(i + 1);
            }
        }
        if (ok) tc_commit(&bar.done);
        tc_commit(&bar.drain);
        if (!mbar_wait(&bar.drain, 0)) report_status(status, kStatusWaitTimeout);
    } else if (warp >= 2) {
        // ---- elementwise: thread = key row = TMEM lane; the two warps of a
        // lane quarter take 64 query columns each of a tile
        const int q = warp & 3;
        const int cg = (warp - 2) >> 2;
        const int r = q * 32 + lane;
        const int row = k0 + r;
        const uint32_t tS = tmem + (static_cast<uint32_t>(q * 32) << 16);
        const bool live = row < p.nk[seg];
        bool ok = true;
        for (int i = 0; i < ntiles; ++i) {
            if (!mbar_wait(&bar.s0_full, i & 1)) { fail(); ok = false; break; }
            tc_fence_after();
            const int nd = 2 * i + 1;
            const float* lse = sLD + ((nd % S_) >> 1) * 2 * kT + cg * 64;
            const float* dl = lse + kT;
            const int qs = i < nt0 ? 0 : 1;
            // query columns < valid of this warp's 64 are real
            const int valid = p.nq[qs] - (i - (qs ? nt0 : 0)) * kT - cg * 64;
            const uint32_t tb = tS + cg * 64;
            uint32_t sr[64], pr_[64];
            tmem_ld_x32(tb, *reinterpret_cast<uint32_t(*)[32]>(&sr[0]));
            tmem_ld_x32(tb + 32, *reinterpret_cast<uint32_t(*)[32]>(&sr[32]));
            tmem_ld_x32(tb + kT, *reinterpret_cast<uint32_t(*)[32]>(&pr_[0]));
            tmem_ld_x32(tb + kT + 32, *reinterpret_cast<uint32_t(*)[32]>(&pr_[32]));
            tmem_ld_wait();
            if (valid >= 64) {
                // every query column real: paired fp32 arithmetic, no selects
                const float2 c2 = make_float2(p.scale_log2, p.scale_log2);
#pragma unroll
                for (int c = 0; c < 64; c += 2) {
                    const float2 l2 = *reinterpret_cast<const float2*>(lse + c);
                    const float2 d2 = *reinterpret_cast<const float2*>(dl + c);
                    const float2 x = __ffma2_rn(make_float2(__uint_as_float(sr[c]), __uint_as_float(sr[c + 1])), c2,
                                                make_float2(-l2.x, -l2.y));
                    const float2 pv = make_float2(ex2(x.x), ex2(x.y));
                    const float2 dp = __fadd2_rn(make_float2(__uint_as_float(pr_[c]), __uint_as_float(pr_[c + 1])),
                                                 make_float2(-d2.x, -d2.y));
                    const float2 ds = __fmul2_rn(pv, dp);
                    sr[c / 2] = pack_bf16x2(pv.x, pv.y);
                    pr_[c / 2] = pack_bf16x2(ds.x, ds.y);
                }
            } else {
#pragma unroll
                for (int c = 0; c < 64; c += 2) {
                    float pv[2], ds[2];
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        const bool real = c + e < valid;
                        const float x = ex2(fmaf(__uint_as_float(sr[c + e]), p.scale_log2, -lse[c + e]));
                        pv[e] = real ? x : 0.f;
                        ds[e] = real ? x * (__uint_as_float(pr_[c + e]) - dl[c + e]) : 0.f;
                    }
                    sr[c / 2] = pack_bf16x2(pv[0], pv[1]);
                    pr_[c / 2] = pack_bf16x2(ds[0], ds[1]);
                }
            }
            // packed over this warp's own (already read) S^T / dP^T columns
            tmem_st_x32(tb, sr);
            tmem_st_x32(tb + kT, pr_);
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bar.p_full[0]);
        }
        if (ok && mbar_wait(&bar.done, 0)) {
            tc_fence_after();
            const int64_t r = (static_cast<int64_t>(b) * p.nk[seg] + row) * p.ldkv[seg] + h * HD;
            if (cg == 0) store_row_bf16(tS + 256, 1.0f, p.dv[seg] + r, live, HD);      // dV
            else store_row_bf16(tS + 256 + HD, p.scale, p.dk[seg] + r, live, HD);     // dK
        } else if (ok) {
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
        tmem_dealloc(tmem, 512);
    }
}

template <int HD>
constexpr int smem_dq() { return 2 * kT * HD * 2 + kSlotsDq * kT * HD * 2 + kBarBytes; }
template <int HD>
constexpr int smem_dkdv() { return 2 * kT * HD * 2 + kSlotsDkdv * kT * HD * 2 + (kSlotsDkdv / 2) * 2 * kT * 4 + kBarBytes; }
static_assert(sizeof(Bars) <= kBarBytes, "barrier block too small");

}  // namespace

size_t attention_backward_ws_bytes(int B, int heads, int n0, int n1) {
    return static_cast<size_t>(B) * heads * attn_lse_rows(n0, n1) * sizeof(float);
}

namespace {

template <int HD>
int attention_backward_hd(const AttnBwdSpec& a, void* ws, size_t ws_bytes, cudaStream_t stream) {
    constexpr int kSmemDq = smem_dq<HD>(), kSmemDkdv = smem_dkdv<HD>();
    const int B = a.B, heads = a.heads;
    const int nq0 = a.q[0].n, nq1 = a.q[1].n, nk0 = a.kv[0].n, nk1 = a.kv[1].n;
    if (B <= 0 || heads <= 0 || B > 65535 || heads > 65535 || nq0 < 0 || nq1 < 0 || nk0 < 0 || nk1 < 0 ||
        nq0 + nq1 <= 0 || nk0 + nk1 <= 0)
        return set_error(FF_ERR_INVALID_ARG, "attention backward: bad shape");
    if (!a.lse || !ws) return set_error(FF_ERR_INVALID_ARG, "attention backward: null lse or workspace");
    const int H = heads * HD;
    if (a.q_col < 0 || a.k_col < 0 || a.v_col < 0 || a.q_col % 8 || a.k_col % 8 || a.v_col % 8)
        return set_error(FF_ERR_INVALID_ARG, "attention backward: q / k / v columns must be multiples of 8");
    const int kv_cols = (a.k_col > a.v_col ? a.k_col : a.v_col) + H;
    for (int i = 0; i < 2; ++i) {
        const AttnBwdQuerySeg& q = a.q[i];
        if (q.n && (!q.q || !q.o || !q.dout || !q.dq || !aligned16(q.q) || !aligned16(q.o) || !aligned16(q.dout) ||
                    !aligned16(q.dq) || q.ld % 8 || q.ldo % 8 || q.ldg % 8 || q.ldq % 8 || q.ld < a.q_col + H ||
                    q.ldo < H || q.ldg < H || q.ldq < H))
            return set_error(FF_ERR_INVALID_ARG, "attention backward: bad query segment %d", i);
        const AttnBwdKvSeg& k = a.kv[i];
        if (k.n && (!k.kv || !k.dk || !k.dv || !aligned16(k.kv) || !aligned16(k.dk) || !aligned16(k.dv) ||
                    k.ld % 8 || k.ldd % 8 || k.ld < kv_cols || k.ldd < H))
            return set_error(FF_ERR_INVALID_ARG, "attention backward: bad key / value segment %d", i);
    }
    const size_t need = attention_backward_ws_bytes(B, heads, nq0, nq1);
    if (ws_bytes < need || !aligned16(ws))
        return set_error(FF_ERR_WORKSPACE, "attention backward: workspace %zu B < %zu B", ws_bytes, need);
    for (auto* f : {(const void*)attn_bwd_dq_kernel<HD>, (const void*)attn_bwd_dkdv_kernel<HD>}) {
        const int bytes = f == (const void*)attn_bwd_dq_kernel<HD> ? kSmemDq : kSmemDkdv;
        if (cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) != cudaSuccess)
            return set_error(FF_ERR_CUDA, "attention backward: cannot set shared memory size");
    }
    // an empty segment still needs a valid map: it takes its neighbour's
    CUtensorMap tq[2], tkv[2], tdo[2];
    for (int i = 0; i < 2; ++i) {
        const AttnBwdQuerySeg& q = a.q[i].n > 0 ? a.q[i] : a.q[1 - i];
        FF_TRY(make_tmap_bf16(&tq[i], q.q, static_cast<int64_t>(B) * q.n, a.q_col + H, q.ld, kT));
        FF_TRY(make_tmap_bf16(&tdo[i], q.dout, static_cast<int64_t>(B) * q.n, H, q.ldg, kT));
        const AttnBwdKvSeg& k = a.kv[i].n > 0 ? a.kv[i] : a.kv[1 - i];
        FF_TRY(make_tmap_bf16(&tkv[i], k.kv, static_cast<int64_t>(B) * k.n, kv_cols, k.ld, kT));
    }
    float* delta = static_cast<float*>(ws);
    const int rows = attn_lse_rows(nq0, nq1);
    {
        const int64_t warps = (static_cast<int64_t>(B) * (nq0 + nq1)) * heads;
        const bool lo = a.q[0].o_lo || a.q[1].o_lo;
        ProfScope prof(stream, "attn_bwd_delta", 0.0, (lo ? 6.0 : 4.0) * warps * HD);
        attn_bwd_delta_kernel<HD><<<static_cast<unsigned>((warps + 7) / 8), 256, 0, stream>>>(
            B, heads, nq0, nq1, a.q[0].o, a.q[0].dout, a.q[1].o, a.q[1].dout, a.q[0].ldo, a.q[1].ldo, a.q[0].ldg,
            a.q[1].ldg, a.q[0].o_lo, a.q[1].o_lo, a.q[0].ldo_lo, a.q[1].ldo_lo, rows, attn_pad128(nq0), delta);
        FF_TRY(check_launch("attn_bwd_delta_kernel"));
    }
    BwdParams p;
    p.nq[0] = nq0;
    p.nq[1] = nq1;
    p.nk[0] = nk0;
    p.nk[1] = nk1;
    p.qtiles0 = (nq0 + kT - 1) / kT;
    p.ktiles0 = (nk0 + kT - 1) / kT;
    p.q_col = a.q_col;
    p.k_col = a.k_col;
    p.v_col = a.v_col;
    p.scale_log2 = static_cast<float>(1.4426950408889634 / sqrt(static_cast<double>(HD)));
    p.scale = static_cast<float>(1.0 / sqrt(static_cast<double>(HD)));
    p.lse = a.lse;
    p.delta = delta;
    p.lse_rows = rows;
    p.lse_base[0] = 0;
    p.lse_base[1] = attn_pad128(nq0);
    for (int i = 0; i < 2; ++i) {
        p.dq[i] = a.q[i].dq;
        p.ldq[i] = a.q[i].ldq;
        p.dk[i] = a.kv[i].dk;
        p.dv[i] = a.kv[i].dv;
        p.ldkv[i] = a.kv[i].ldd;
    }
    const double NN = static_cast<double>(nq0 + nq1) * static_cast<double>(nk0 + nk1);
    {
        ProfScope prof(stream, "attn_bwd_dq", 6.0 * B * heads * NN * HD, 0.0);
        const dim3 grid(p.qtiles0 + (nq1 + kT - 1) / kT, heads, B);
        attn_bwd_dq_kernel<HD><<<grid, kThreads, kSmemDq, stream>>>(tq[0], tq[1], tkv[0], tkv[1], tdo[0], tdo[1], p,
                                                                 device_status_ptr());
        FF_TRY(check_launch("attn_bwd_dq_kernel"));
    }
    ProfScope prof(stream, "attn_bwd_dkdv", 8.0 * B * heads * NN * HD, 0.0);
    const dim3 grid(p.ktiles0 + (nk1 + kT - 1) / kT, heads, B);
    attn_bwd_dkdv_kernel<HD><<<grid, kThreads, kSmemDkdv, stream>>>(tq[0], tq[1], tkv[0], tkv[1], tdo[0], tdo[1], p,
                                                                 device_status_ptr());
    return check_launch("attn_bwd_dkdv_kernel");
}

}  // namespace

int attention_backward_general(const AttnBwdSpec& a, void* ws, size_t ws_bytes, cudaStream_t stream) {
    if (a.head_dim == 128) return attention_backward_hd<128>(a, ws, ws_bytes, stream);
    if (a.head_dim == 64) return attention_backward_hd<64>(a, ws, ws_bytes, stream);
    return set_error(FF_ERR_UNSUPPORTED, "attention backward: head_dim %d (64 or 128)", a.head_dim);
}

int attention_backward(const AttnBwdSeg& s0, const AttnBwdSeg& s1, int B, int heads, int head_dim, const float* lse,
                       void* ws, size_t ws_bytes, cudaStream_t stream) {
    const int64_t H = static_cast<int64_t>(heads) * head_dim;
    const AttnBwdSeg* sg[2] = {&s0, &s1};
    AttnBwdSpec a{};
    for (int i = 0; i < 2; ++i) {
        const AttnBwdSeg& s = *sg[i];
        // the joint layout: q, k, v (and their gradients) side by side in one row
        if (s.n && (!s.dqkv || s.ld < 3 * H || s.ldd < 3 * H))
            return set_error(FF_ERR_INVALID_ARG, "attention backward: bad segment %d", i);
        a.q[i] = AttnBwdQuerySeg{s.qkv, s.ld, s.n, s.o, s.ldo, s.dout, s.ldg ? s.ldg : s.ldo, s.dqkv, s.ldd, s.o_lo,
                                 s.ldo_lo};
        a.kv[i] = AttnBwdKvSeg{s.qkv, s.ld, s.n, s.dqkv ? s.dqkv + H : nullptr, s.dqkv ? s.dqkv + 2 * H : nullptr,
                               s.ldd};
    }
    a.q_col = 0;
    a.k_col = static_cast<int>(H);
    a.v_col = static_cast<int>(2 * H);
    a.B = B;
    a.heads = heads;
    a.head_dim = head_dim;
    a.lse = lse;
    return attention_backward_general(a, ws, ws_bytes, stream);
}

}  // namespace ff

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
constexpr int kQSlots = 3, kDoSlots = 2;       // streamed Q_i / dO_i tiles in flight (dK dV kernel)
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
    const float* nlse;     // -lse in the same layout (workspace copy, read by the dK dV kernel)
    const float* ndelta;   // -D in the same layout
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
    uint64_t grp_full[4];          // producer -> MMA: both streamed tiles of step i landed (entry i % 4);
                                   // dK dV kernel: Q_i and lse_i landed
    uint64_t do_full[4];           // producer -> MMA: dO_i and D_i landed (dK dV kernel, entry i % 4)
    uint64_t rel[4];               // MMA -> producer (and dQ's elementwise warps): step i's MMAs are done
    uint64_t s0_full;              // MMA -> elementwise: S^T of the step in TMEM (dK dV kernel)
    uint64_t s1_full;              // MMA -> elementwise: dP^T of the step in TMEM (dK dV kernel)
    uint64_t s0_ring[4];           // MMA -> elementwise and producer: S and dP of step j in TMEM (entry
                                   // j % 4), so V_j is read (dQ kernel)
    uint64_t p_full[2];            // elementwise -> MMA: dQ kernel: [0] S / dP read, [1] dS written;
                                   // dK dV kernel: [0] P^T written, [1] dS^T written
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

// D_i = sum_c dO_ic O_ic, stored negated, with a negated copy of lse_i
// beside it (the dK dV kernel adds both per score).  A block takes kDeltaRows
// consecutive token rows of one head, sample and segment (so its lse / D
// reads and writes are contiguous); the d / 8 threads of a row each load 16
// bytes of O and of dO (a head's row is 2 d contiguous bytes) and are summed
// by shuffles; each thread takes four rows, their loads issued together.
// With the forward's low parts (o_lo), O = o + o_lo: D = rowsum(P dP)
// subtracts nearly equal terms when the rows of V are close to each other,
// and bf16 O alone would leave a relative error of 2^-9 |dO| |O| in D.
template <int HD>
constexpr int delta_rows() { return 4 * 8 * (32 / (HD / 8)); }   // four rows per thread, 256 threads
template <int HD>
__global__ void __launch_bounds__(256) attn_bwd_delta_kernel(int B, int heads, int n0, int n1,
                                                             const __nv_bfloat16* o0, const __nv_bfloat16* do0,
                                                             const __nv_bfloat16* o1, const __nv_bfloat16* do1,
                                                             int64_t ldo0, int64_t ldo1, int64_t ldg0, int64_t ldg1,
                                                             const __nv_bfloat16* ol0, const __nv_bfloat16* ol1,
                                                             int64_t ldl0, int64_t ldl1, int lse_rows, int base1,
                                                             const float* lse, float* ndelta, float* nlse) {
    constexpr int kLanes = HD / 8;                  // threads per row
    constexpr int kRowsPerPass = 256 / kLanes;      // rows one pass of the block covers
    constexpr int R = delta_rows<HD>();
    constexpr int kPer = R / kRowsPerPass;          // rows per thread
    const int t0 = (n0 + R - 1) / R, t1 = (n1 + R - 1) / R;
    const int b = blockIdx.x / (t0 + t1);
    const int t = blockIdx.x - b * (t0 + t1);
    const bool s1 = t >= t0;
    const int n = s1 ? n1 : n0;
    const int h = blockIdx.y;
    const int c = threadIdx.x & (kLanes - 1);
    const int first = (s1 ? t - t0 : t) * R + threadIdx.x / kLanes;
    const int64_t ld_o = s1 ? ldo1 : ldo0, ld_g = s1 ? ldg1 : ldg0, ld_l = s1 ? ldl1 : ldl0;
    const int64_t rowbase = static_cast<int64_t>(b) * n;
    const __nv_bfloat16* o = (s1 ? o1 : o0) + h * HD + c * 8;
    const __nv_bfloat16* g = (s1 ? do1 : do0) + h * HD + c * 8;
    const __nv_bfloat16* ol = s1 ? ol1 : ol0;
    const int64_t lbase = (static_cast<int64_t>(b) * heads + h) * lse_rows + (s1 ? base1 : 0);
    uint4 ov[kPer], gv[kPer], lv[kPer];
    float lse_v[kPer];
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
        const int row = first + k * kRowsPerPass;
        ov[k] = gv[k] = lv[k] = make_uint4(0u, 0u, 0u, 0u);
        lse_v[k] = 0.f;
        if (row >= n) continue;
        const int64_t r = rowbase + row;
        ov[k] = *reinterpret_cast<const uint4*>(o + r * ld_o);
        gv[k] = *reinterpret_cast<const uint4*>(g + r * ld_g);
        if (ol) lv[k] = *reinterpret_cast<const uint4*>(ol + h * HD + c * 8 + r * ld_l);
        if (c == 0) lse_v[k] = lse[lbase + row];
    }
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
        const int row = first + k * kRowsPerPass;
        const uint32_t ow[4] = {ov[k].x, ov[k].y, ov[k].z, ov[k].w}, gw[4] = {gv[k].x, gv[k].y, gv[k].z, gv[k].w},
                       lw[4] = {lv[k].x, lv[k].y, lv[k].z, lv[k].w};
        float s = 0.f;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            float2 of = unpack_bf16x2(ow[e]);
            const float2 lf = unpack_bf16x2(lw[e]);
            of.x += lf.x;
            of.y += lf.y;
            const float2 gf = unpack_bf16x2(gw[e]);
            s = fmaf(of.x, gf.x, fmaf(of.y, gf.y, s));
        }
        // rows past n summed zeros; every lane takes part in the shuffles
#pragma unroll
        for (int m = kLanes / 2; m; m >>= 1) s += __shfl_xor_sync(0xffffffffu, s, m);
        if (c == 0 && row < n) {
            ndelta[lbase + row] = -s;
            nlse[lbase + row] = -lse_v[k];
        }
    }
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
        // slot descriptors: slot s starts s * kTileBytes further on, s * kTileBytes / 16
        // in the descriptor's start-address field
        constexpr uint32_t kSlotStep = kTileBytes >> 4;
        const uint64_t k_k0 = smem_desc_k_sw128(smem_u32(sKV));
        const uint64_t k_m0 = smem_desc_mn_sw128(smem_u32(sKV), kT * 128);
        const uint64_t v_k0 = smem_desc_k_sw128(smem_u32(sKV + kKSlots * kTileBytes));
        // S = Q K_j^T and dP = dO V_j^T of the whole key tile (K_j in K slot ks, V_j in V slot vs)
        auto issue_sdp = [&](int j, int ks, int vs) {
            const uint64_t dk = k_k0 + ks * kSlotStep;
            const uint64_t dv = v_k0 + vs * kSlotStep;
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
            issue_sdp(0, 0, 0);
        }
        int ks = 0, vs = 0;   // slots of K_j and V_j
        for (int j = 0; ok && j < ntiles; ++j) {
            const uint64_t dkm = k_m0 + ks * kSlotStep;
            ks = ks + 1 == kKSlots ? 0 : ks + 1;
            vs = vs + 1 == kVSlots ? 0 : vs + 1;
            // the elementwise warps hold S_j / dP_j in registers: the next tile's may go in
            if (!mbar_wait(&bar.p_full[0], j & 1)) { fail(); ok = false; break; }
            if (j + 1 < ntiles) {   // the arrival also covers K_j+1 / V_j+1
                tc_fence_after();
                issue_sdp(j + 1, ks, vs);
            }
            if (!mbar_wait(&bar.p_full[1], j & 1)) { fail(); ok = false; break; }
            tc_fence_after();
            // dQ += dS_j K_j: dS (keys 16 k.. at columns 8 k..) from TMEM, K_j rows as [keys (K) x d (N)]
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
        const float ndd = live ? p.ndelta[li] : 0.f;   // -D
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
            // K_j+1 and V_j+1 landed too: the MMA thread issues S_j+1 / dP_j+1 on this arrival alone
            if (!warp_wait(&bar.grp_full[(j + 1) & 3], ((j + 1) >> 2) & 1, j + 1 < ntiles, lane)) {
                fail();
                ok = false;
                break;
            }
            if (lane == 0) mbar_arrive(&bar.p_full[0]);   // S_j / dP_j consumed: the buffer may be refilled
            const int ks = j < nt0 ? 0 : 1;
            // key columns < valid of this warp's 64 are real
            const int valid = p.nk[ks] - (j - (ks ? nt0 : 0)) * kT - cg * 64;
            if (valid >= 64 && full_rows) {
                // every column and row real: paired fp32 arithmetic, no selects
                const float2 c2 = make_float2(p.scale_log2, p.scale_log2), nl2 = make_float2(-lse, -lse);
                const float2 nd2 = make_float2(ndd, ndd);
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
                        ds[e] = (i + e < valid && live) ? pv * (__uint_as_float(pr_[i + e]) + ndd) : 0.f;
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
// the MMA thread issues dV += P^T dO_i once P^T is written, S^T of tile
// i + 1 behind it, dK += dS^T Q_i once dS^T is written, then dP^T of i + 1:
// the tensor pipe runs one thread's MMAs in issue order, so S^T_{i+1}
// overwrites P^T_i only after dV_i has read it (dP^T_{i+1} and dS^T_i
// likewise), and the elementwise work of a tile runs under the MMAs of its
// neighbours.  Shared memory: the K and V tiles of this CTA, three Q_i slots,
// two dO_i slots, lse_i per Q slot and D_i per dO slot.  Q_i and dO_i are
// both read for the last time by dK_i / dV_i, but Q_i + 1 is needed a whole
// step before dO_i + 1 (S^T comes first), so it gets the deeper ring.
template <int HD>
__global__ void __launch_bounds__(kThreads, 1)
attn_bwd_dkdv_kernel(const __grid_constant__ CUtensorMap tm_q0, const __grid_constant__ CUtensorMap tm_q1,
                     const __grid_constant__ CUtensorMap tm_kv0, const __grid_constant__ CUtensorMap tm_kv1,
                     const __grid_constant__ CUtensorMap tm_do0, const __grid_constant__ CUtensorMap tm_do1,
                     const BwdParams p, int* status) {
    constexpr int kTileBytes = kT * HD * 2;
    constexpr int NB = HD / 64;
    extern __shared__ __align__(1024) uint8_t smem[];
    uint8_t* sK = smem;
    uint8_t* sV = smem + kTileBytes;
    uint8_t* sQ = smem + 2 * kTileBytes;                      // [kQSlots][tile]: Q_i in slot i % 3
    uint8_t* sDo = sQ + kQSlots * kTileBytes;                 // [kDoSlots][tile]: dO_i in slot i % 2
    float* sL = reinterpret_cast<float*>(sDo + kDoSlots * kTileBytes);   // [kQSlots][kT]: -lse_i
    float* sD = sL + kQSlots * kT;                                         // [kDoSlots][kT]: -D_i
    Bars& bar = *reinterpret_cast<Bars*>(sD + kDoSlots * kT);
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
            mbar_init(&bar.grp_full[g], 1);
            mbar_init(&bar.do_full[g], 1);
            mbar_init(&bar.rel[g], 1);
        }
        mbar_init(&bar.s0_full, 1);
        mbar_init(&bar.s1_full, 1);
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
        // ---- producer: K and V of this tile, then Q_0, then per step n
        // Q_n+1 and dO_n: both wait for step n - 2's MMAs (Q_n+1 goes into
        // the slot of Q_n-2, dO_n into that of dO_n-2); lse_i rides on Q_i's
        // barrier, D_i on dO_i's
        const CUtensorMap* tk = seg ? &tm_kv1 : &tm_kv0;
        mbar_arrive_expect_tx(&bar.fixed_full, 2 * kTileBytes);
        for (int c = 0; c < NB; ++c) {
            tma_load_2d(sK + c * (kT * 128), tk, &bar.fixed_full, p.k_col + h * HD + c * 64, b * p.nk[seg] + k0);
            tma_load_2d(sV + c * (kT * 128), tk, &bar.fixed_full, p.v_col + h * HD + c * 64, b * p.nk[seg] + k0);
        }
        auto tile_row = [&](int i, int& qs, int& qi) {
            qs = i < nt0 ? 0 : 1;
            qi = (i - (qs ? nt0 : 0)) * kT;
        };
        auto load_q = [&](int i) {
            int qs, qi;
            tile_row(i, qs, qi);
            uint64_t* fb = &bar.grp_full[i & 3];
            mbar_arrive_expect_tx(fb, kTileBytes + kT * 4);
            uint8_t* dst = sQ + (i % kQSlots) * kTileBytes;
            for (int c = 0; c < NB; ++c)
                tma_load_2d(dst + c * (kT * 128), qs ? &tm_q1 : &tm_q0, fb, p.q_col + h * HD + c * 64, b * p.nq[qs] + qi);
            bulk_load_1d(sL + (i % kQSlots) * kT, p.nlse + lrow + p.lse_base[qs] + qi, kT * 4, fb);
        };
        auto load_do = [&](int i) {
            int qs, qi;
            tile_row(i, qs, qi);
            uint64_t* fb = &bar.do_full[i & 3];
            mbar_arrive_expect_tx(fb, kTileBytes + kT * 4);
            uint8_t* dst = sDo + (i % kDoSlots) * kTileBytes;
            for (int c = 0; c < NB; ++c)
                tma_load_2d(dst + c * (kT * 128), qs ? &tm_do1 : &tm_do0, fb, h * HD + c * 64, b * p.nq[qs] + qi);
            bulk_load_1d(sD + (i % kDoSlots) * kT, p.ndelta + lrow + p.lse_base[qs] + qi, kT * 4, fb);
        };
        static_assert(kQSlots == kDoSlots + 1, "Q_n+1 and dO_n share their release");
        load_q(0);
        for (int n = 0; n < ntiles; ++n) {
            if (n >= kDoSlots) {   // step n - 2's slots
                const int r = n - kDoSlots;
                if (!mbar_wait(&bar.rel[r & 3], (r >> 2) & 1)) { fail(); break; }
            }
            if (n + 1 < ntiles) load_q(n + 1);
            load_do(n);
        }
    } else if (warp == 1 && lane == 0) {
        // ---- MMA issuer
        constexpr uint32_t idesc_s = idesc_bf16_f32(kT, kT);
        constexpr uint32_t idesc_g = idesc_bf16_f32(kT, HD) | (1u << 16);   // B = Q_i / dO_i, MN-major
        bool ok = mbar_wait(&bar.fixed_full, 0);
        if (!ok) fail();
        const uint64_t dk_ = smem_desc_k_sw128(smem_u32(sK));
        const uint64_t dv_ = smem_desc_k_sw128(smem_u32(sV));
        auto wait_q = [&](int i) { return mbar_wait(&bar.grp_full[i & 3], (i >> 2) & 1); };
        auto wait_do = [&](int i) { return mbar_wait(&bar.do_full[i & 3], (i >> 2) & 1); };
        // slot descriptors: slot s of a ring starts s * kTileBytes further on,
        // s * kTileBytes / 16 in the descriptor's start-address field
        constexpr uint32_t kSlotStep = kTileBytes >> 4;
        const uint64_t q_k0 = smem_desc_k_sw128(smem_u32(sQ)), q_m0 = smem_desc_mn_sw128(smem_u32(sQ), kT * 128);
        const uint64_t do_k0 = smem_desc_k_sw128(smem_u32(sDo)), do_m0 = smem_desc_mn_sw128(smem_u32(sDo), kT * 128);
        // S^T = K Q_i^T and dP^T = V dO_i^T of the whole query tile, each
        // published on its own barrier
        auto issue_st = [&](int slot) {
            const uint64_t dq_ = q_k0 + slot * kSlotStep;
#pragma unroll
            for (int k = 0; k < HD / 16; ++k) {
                const uint32_t off = ((k / 4) * (kT * 128) + (k % 4) * 32) >> 4;
                tc_mma_bf16(tmem, dk_ + off, dq_ + off, idesc_s, k != 0 ? 1u : 0u);
            }
            tc_commit(&bar.s0_full);
        };
        auto issue_dpt = [&](int slot) {
            const uint64_t ddo = do_k0 + slot * kSlotStep;
#pragma unroll
            for (int k = 0; k < HD / 16; ++k) {
                const uint32_t off = ((k / 4) * (kT * 128) + (k % 4) * 32) >> 4;
                tc_mma_bf16(tmem + kT, dv_ + off, ddo + off, idesc_s, k != 0 ? 1u : 0u);
            }
            tc_commit(&bar.s1_full);
        };
        if (ok && !wait_q(0)) { fail(); ok = false; }
        if (ok) {
            tc_fence_after();
            issue_st(0);
        }
        if (ok && !wait_do(0)) { fail(); ok = false; }
        if (ok) {
            tc_fence_after();
            issue_dpt(0);
        }
        int qs = 0, ds = 0;   // slots of Q_i and dO_i
        // Per query tile i: dV_i as soon as P^T_i is written, S^T_{i+1} behind
        // it (it overwrites P^T_i, which dV_i has read: the tensor pipe runs
        // one thread's MMAs in order), dK_i once dS^T_i is written, then
        // dP^T_{i+1} over dS^T_i.  The elementwise warps form P^T_{i+1} while
        // dK_i and dP^T_{i+1} run and dS^T_{i+1} while dV_{i+1} and
        // S^T_{i+2} run, so the tensor pipe does not wait for them.
        for (int i = 0; ok && i < ntiles; ++i) {
            const uint64_t dqm = q_m0 + qs * kSlotStep;
            const uint64_t ddom = do_m0 + ds * kSlotStep;
            qs = qs + 1 == kQSlots ? 0 : qs + 1;
            ds = ds + 1 == kDoSlots ? 0 : ds + 1;
            if (!mbar_wait(&bar.p_full[0], i & 1)) { fail(); ok = false; break; }
            tc_fence_after();
#pragma unroll
            for (int k = 0; k < kT / 16; ++k) {
                // queries 16 k.. : each warp's 64 queries packed over the first 32 of its columns
                const uint32_t a = tmem + (k >> 2) * 64 + (k & 3) * 8;
                tc_mma_bf16_ts(tmem + 256, a, ddom + k * (2048 >> 4), idesc_g, (i | k) != 0 ? 1u : 0u);   // dV += P^T dO
            }
            const bool more = i + 1 < ntiles;
            if (more) issue_st(qs);   // the P^T arrival also covers Q_i+1
            if (!mbar_wait(&bar.p_full[1], i & 1)) { fail(); ok = false; break; }
            tc_fence_after();
#pragma unroll
            for (int k = 0; k < kT / 16; ++k) {
                const uint32_t a = tmem + kT + (k >> 2) * 64 + (k & 3) * 8;
                tc_mma_bf16_ts(tmem + 256 + HD, a, dqm + k * (2048 >> 4), idesc_g, (i | k) != 0 ? 1u : 0u);   // dK += dS^T Q
            }
            tc_commit(&bar.rel[i & 3]);   // Q_i, dO_i, lse_i and D_i read for the last time
            if (more) issue_dpt(ds);   // the dS^T arrival also covers dO_i+1
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
            const float* nl = sL + (i % kQSlots) * kT + cg * 64;   // -lse of this warp's 64 queries
            const float* nd = sD + (i % kDoSlots) * kT + cg * 64;  // -D
            const int qs = i < nt0 ? 0 : 1;
            // query columns < valid of this warp's 64 are real
            const int valid = p.nq[qs] - (i - (qs ? nt0 : 0)) * kT - cg * 64;
            const uint32_t tb = tS + cg * 64;
            // P^T = 2^(S^T log2(e) / sqrt(d) - lse), kept in fp32 for dS^T
            float pf[64];
            uint32_t u[64];
            if (!mbar_wait(&bar.s0_full, i & 1)) { fail(); ok = false; break; }
            tc_fence_after();
            tmem_ld_x32(tb, *reinterpret_cast<uint32_t(*)[32]>(&u[0]));
            tmem_ld_x32(tb + 32, *reinterpret_cast<uint32_t(*)[32]>(&u[32]));
            tmem_ld_wait();
            if (valid >= 64) {
                // every query column real: paired fp32 arithmetic, no selects
                const float2 c2 = make_float2(p.scale_log2, p.scale_log2);
#pragma unroll
                for (int c = 0; c < 64; c += 4) {
                    const float4 l4 = *reinterpret_cast<const float4*>(nl + c);
                    const float2 x0 = __ffma2_rn(make_float2(__uint_as_float(u[c]), __uint_as_float(u[c + 1])), c2,
                                                 make_float2(l4.x, l4.y));
                    const float2 x1 = __ffma2_rn(make_float2(__uint_as_float(u[c + 2]), __uint_as_float(u[c + 3])), c2,
                                                 make_float2(l4.z, l4.w));
                    pf[c] = ex2(x0.x);
                    pf[c + 1] = ex2(x0.y);
                    pf[c + 2] = ex2(x1.x);
                    pf[c + 3] = ex2(x1.y);
                }
            } else {
#pragma unroll
                for (int c = 0; c < 64; ++c) {
                    const float x = ex2(fmaf(__uint_as_float(u[c]), p.scale_log2, nl[c]));
                    pf[c] = c < valid ? x : 0.f;
                }
            }
#pragma unroll
            for (int c = 0; c < 64; c += 2) u[c / 2] = pack_bf16x2(pf[c], pf[c + 1]);
            // packed over this warp's own (already read) S^T columns
            tmem_st_x32(tb, *reinterpret_cast<uint32_t(*)[32]>(&u[0]));
            tmem_st_wait();
            tc_fence_before();
            // Q_i+1 and lse_i+1 landed too: S^T_i+1 follows dV_i on this arrival alone
            if (!warp_wait(&bar.grp_full[(i + 1) & 3], ((i + 1) >> 2) & 1, i + 1 < ntiles, lane)) {
                fail();
                ok = false;
                break;
            }
            if (lane == 0) mbar_arrive(&bar.p_full[0]);
            // dS^T = P^T (dP^T - D)
            if (!mbar_wait(&bar.s1_full, i & 1)) { fail(); ok = false; break; }
            tc_fence_after();
            tmem_ld_x32(tb + kT, *reinterpret_cast<uint32_t(*)[32]>(&u[0]));
            tmem_ld_x32(tb + kT + 32, *reinterpret_cast<uint32_t(*)[32]>(&u[32]));
            tmem_ld_wait();
            if (valid >= 64) {
#pragma unroll
                for (int c = 0; c < 64; c += 4) {
                    const float4 d4 = *reinterpret_cast<const float4*>(nd + c);
                    const float2 dp0 = __fadd2_rn(make_float2(__uint_as_float(u[c]), __uint_as_float(u[c + 1])),
                                                  make_float2(d4.x, d4.y));
                    const float2 dp1 = __fadd2_rn(make_float2(__uint_as_float(u[c + 2]), __uint_as_float(u[c + 3])),
                                                  make_float2(d4.z, d4.w));
                    const float2 ds0 = __fmul2_rn(make_float2(pf[c], pf[c + 1]), dp0);
                    const float2 ds1 = __fmul2_rn(make_float2(pf[c + 2], pf[c + 3]), dp1);
                    u[c / 2] = pack_bf16x2(ds0.x, ds0.y);
                    u[c / 2 + 1] = pack_bf16x2(ds1.x, ds1.y);
                }
            } else {
#pragma unroll
                for (int c = 0; c < 64; c += 2) {
                    float ds[2];
#pragma unroll
                    for (int e = 0; e < 2; ++e)
                        ds[e] = c + e < valid ? pf[c + e] * (__uint_as_float(u[c + e]) + nd[c + e]) : 0.f;
                    u[c / 2] = pack_bf16x2(ds[0], ds[1]);
                }
            }
            tmem_st_x32(tb + kT, *reinterpret_cast<uint32_t(*)[32]>(&u[0]));
            tmem_st_wait();
            tc_fence_before();
            // dO_i+1 and D_i+1 landed too: dP^T_i+1 follows dK_i on this arrival alone
            if (!warp_wait(&bar.do_full[(i + 1) & 3], ((i + 1) >> 2) & 1, i + 1 < ntiles, lane)) {
                fail();
                ok = false;
                break;
            }
            if (lane == 0) mbar_arrive(&bar.p_full[1]);
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
constexpr int smem_dkdv() { return (2 + kQSlots + kDoSlots) * kT * HD * 2 + (kQSlots + kDoSlots) * kT * 4 + kBarBytes; }
static_assert(smem_dkdv<128>() <= 227 * 1024, "dK dV shared memory");
static_assert(sizeof(Bars) <= kBarBytes, "barrier block too small");

}  // namespace

size_t attention_backward_ws_bytes(int B, int heads, int n0, int n1) {
    return 2 * static_cast<size_t>(B) * heads * attn_lse_rows(n0, n1) * sizeof(float);   // -D, then -lse
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
    const int64_t qrows = static_cast<int64_t>(B) * (static_cast<int64_t>(nq0) + nq1);
    if (qrows >= (int64_t{1} << 31))
        return set_error(FF_ERR_INVALID_ARG, "attention backward: too many query rows");
    if (!a.lse || !ws) return set_error(FF_ERR_INVALID_ARG, "attention backward: null lse or workspace");
    const int H = heads * HD;
    if (a.q_col < 0 || a.k_col < 0 || a.v_col < 0 || a.q_col % 8 || a.k_col % 8 || a.v_col % 8)
        return set_error(FF_ERR_INVALID_ARG, "attention backward: q / k / v columns must be multiples of 8");
    const int kv_cols = (a.k_col > a.v_col ? a.k_col : a.v_col) + H;
    for (int i = 0; i < 2; ++i) {
        const AttnBwdQuerySeg& q = a.q[i];
        if (q.n && (!q.q || !q.o || !q.dout || !q.dq || !aligned16(q.q) || !aligned16(q.o) || !aligned16(q.dout) ||
                    !aligned16(q.dq) || q.ld % 8 || q.ldo % 8 || q.ldg % 8 || q.ldq % 8 || q.ld < a.q_col + H ||
                    q.ldo < H || q.ldg < H || q.ldq < H || (q.o_lo && (!aligned16(q.o_lo) || q.ldo_lo % 8 || q.ldo_lo < H))))
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
    float* ndelta = static_cast<float*>(ws);                            // -D
    float* nlse = ndelta + static_cast<size_t>(B) * heads * attn_lse_rows(nq0, nq1);   // -lse
    const int rows = attn_lse_rows(nq0, nq1);
    {
        const int64_t heads_rows = (static_cast<int64_t>(B) * (nq0 + nq1)) * heads;
        const bool lo = a.q[0].o_lo || a.q[1].o_lo;
        constexpr int R = delta_rows<HD>();
        const int64_t blocks = static_cast<int64_t>(B) * ((nq0 + R - 1) / R + (nq1 + R - 1) / R);
        ProfScope prof(stream, "attn_bwd_delta", 0.0, (lo ? 6.0 : 4.0) * heads_rows * HD);
        attn_bwd_delta_kernel<HD><<<dim3(static_cast<unsigned>(blocks), heads), 256, 0, stream>>>(
            B, heads, nq0, nq1, a.q[0].o, a.q[0].dout, a.q[1].o, a.q[1].dout, a.q[0].ldo, a.q[1].ldo, a.q[0].ldg,
            a.q[1].ldg, a.q[0].o_lo, a.q[1].o_lo, a.q[0].ldo_lo, a.q[1].ldo_lo, rows, attn_pad128(nq0), a.lse, ndelta,
            nlse);
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
    p.nlse = nlse;
    p.ndelta = ndelta;
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

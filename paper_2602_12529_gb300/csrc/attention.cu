// attention.cu -- joint (text + image) non-causal attention on tcgen05,
//   O = softmax(Q K^T / sqrt(d)) V   per (sample, head),
// over the concatenated token sequence [segment 0; segment 1] of each sample
// (MMDiT joint attention: text tokens then image tokens).  Q, K and V are
// read straight out of the bf16 QKV GEMM outputs (row = token, q at column
// h*d, k at H + h*d, v at 2H + h*d) by TMA; the segments may live in
// different buffers.
//
// Work item = two 128-row query tiles (256 query rows) of one segment of one
// (sample, head), sharing every K/V tile.  The kernel is persistent: one CTA
// per SM takes items blockIdx.x, blockIdx.x + gridDim.x, ... and runs their
// K/V steps as one stream (global step g), so the ring, the operand groups
// and the per-step barriers carry on across items without a restart; the
// next item's query tile t is loaded as soon as the last S_t of the current
// item is done, and its epilogue (O / l out of TMEM) overlaps the next
// item's first S MMAs.  Warp roles (10 warps):
//   warp 0      TMA producer: both Q tiles once, then the 128-token K and V
//               tiles in the order K_0, V_0, K_1, V_1, ... into a ring of
//               single-operand slots (5 at d = 128), so the operands of the
//               next K/V step are resident a whole step before they are used
//               (K/V tiles never straddle the segment boundary; rows past the
//               segment end are masked).
//   warp 1      TMEM allocator (all 512 columns); lane 0 issues the MMAs.
//               Per query tile t the order is S_t,j = Q_t K_j^T (M 128, N 128,
//               A and B from shared memory) -> softmax -> O_t += P_t,j V_j
//               (M 128, N d, A = P from TMEM, B = V from shared memory) ->
//               S_t,j+1; the two tiles alternate, so the tensor core works on
//               one tile while the other tile's softmax runs.  Keeping P in
//               TMEM halves the shared-memory operand traffic of P V.
//   warps 2..9  two softmax warpgroups, one per query tile: thread = query
//               row = TMEM lane.  Reads its S row (one 128-column TMEM load),
//               writes P = exp2(S scale - m) as bf16 pairs over the S
//               columns and keeps the row sum l; O / l goes out as bf16.
//
// The MMA thread's instruction stream is what bounds this kernel: the tensor
// pipe's queue is short, so every barrier wait or commit the thread executes
// between MMA batches leaves the pipe idle unless it is short.  Hence:
//   * the K/V ring is signalled in groups: group 0 = K_0, group j + 1 =
//     (V_j, K_j+1), the operands of step j's MMAs, one barrier arrival pair
//     per group (ring of four barriers); tile 0's softmax warps check group
//     j + 1 before they publish P_0,j, so the MMA thread's wait for P_0,j
//     covers the operands too;
//   * slots are released by the commit that already publishes S_1,j+1 to
//     tile 1's softmax (a ring of four barriers, one per step): when S_1,j+1
//     is done, every MMA of step j is done, so V_j and K_j+1 may be
//     overwritten.  Step j's MMA thread work is two waits for P and two
//     commits;
//   * the softmax keeps its first tile's row maximum m as the reference for
//     every later tile (softmax does not depend on the reference, and P in
//     bf16 / l in fp32 lose nothing when later scores exceed m), so only
//     the first tile pays for a max pass.  A tile whose row sum passes 2^40
//     (or overflows) is redone against its true maximum, rescaling l and O,
//     which keeps every P at or below 2^40.
// Every wait is bounded; on a timeout the kernel records the status word,
// drains its tensor-core work, frees TMEM and returns.  The MMA and softmax
// loops do not poll the abort flag: a role that gave up stops signalling, so
// the others run into their own bounded waits.
#include <atomic>

#include "internal.h"
#include "ptx.cuh"

namespace ff {
namespace {


constexpr int kBM = 128;         // query rows per query tile (two tiles per CTA)
constexpr int kBN = 128;         // tokens per K/V tile
constexpr int kSplitMaxItems = 96;   // split items per launch (half of 192 SMs)
constexpr int kThreads = 320;    // producer, MMA, 2 x 4 softmax warps
constexpr int kPersistentItemsPerSm = 16;   // persistent launch below this many items per SM,
constexpr int kPersistentMaxSteps = 128;    // or with at most this many K/V steps per item
std::atomic<int> g_launch_override{0};   // tests: 1 persistent unsplit, 2 one item per CTA, 3 persistent split

template <int HD>
struct ACfg {
    static constexpr int kQBytes = kBM * HD * 2;        // one query tile
    static constexpr int kKBytes = kBN * HD * 2;        // one K or V tile = one ring slot
    static constexpr int kBarBytes = 256;
    // At most seven slots: ring item n arrives on group (n + 1) / 2, whose
    // barrier entry it shares with group (n + 1) / 2 - 4, and only the wait
    // for slot n % kSlots (for S_1 of step (n - kSlots + 1) / 2) guarantees
    // that group has completed; with eight slots item 7 (V_3, group 4)
    // would need no wait and could arrive while group 0 still waits for K_0.
    static constexpr int kSlots = (232448 - 2 * kQBytes - kBarBytes) / kKBytes < 7
                                      ? (232448 - 2 * kQBytes - kBarBytes) / kKBytes : 7;
    static constexpr int kSmemBytes = 2 * kQBytes + kSlots * kKBytes + kBarBytes;
    static constexpr int kTmemCols = 512;
    // TMEM columns of query tile t: S (fp32, kBN columns) at t*256, with P
    // (bf16 pairs, kBN/2 columns) written over its first half; O at t*256+128
    static constexpr int kColO = kBN;
};

struct AttnParams {
    int nq[2];           // query tokens per sample in each query segment
    int nkv[2];          // key/value tokens per sample in each key/value segment
    int qpairs0;         // 256-row query blocks of query segment 0 (segment 1's follow)
    int qpairs;          // 256-row query blocks of both segments
    int heads;
    int items;           // B * heads * qpairs work items, item = (b * heads + h) * qpairs + block
    // persistent launch only: items split_first .. split_first + split_n - 1
    // run as two halves of their K/V steps, half h of item split_first + i on
    // CTA 2 i + h; each half leaves O (unnormalised), m and l of its rows in
    // part / part_ml, and the second to finish a row group combines them
    int split_first, split_n;
    float* part;         // [split_n][2 halves][2 tiles][128 rows][d]
    float2* part_ml;     // [split_n][2][2][128]: (m, l)
    unsigned* tickets;   // [split_n][2 tiles][4 lane quarters], zero at launch
    int q_col, k_col, v_col;
    float scale_log2;
    __nv_bfloat16* out[2];
    int64_t ldo[2];
    __nv_bfloat16* out_lo[2];   // optional: O - bf16(O), rounded to bf16 (training)
    int64_t ldo_lo[2];
    float* lse;          // optional per-row log-sum-exp (base 2), see AttnSpec
    int lse_rows;        // its row pitch per (sample, head)
    int lse_base[2];     // first row of each query segment
};

// Barriers.  Per query tile the chain S -> softmax -> P -> O += P V -> next S
// is strictly ordered.  A parity wait is unambiguous as long as its barrier
// cannot complete two phases past the one waited for: the two-phase
// barriers below are waited in lockstep with their producer, and the rings
// of four are waited at most one step behind (ring item n = 2 j (K_j) or
// 2 j + 1 (V_j) lives in slot n % kSlots and belongs to group (n + 1) / 2).
constexpr int kMaxSlots = 7;
struct Bars {
    uint64_t q_full[2];       // producer -> MMA: query tile t of the current item landed (one phase per item)
    uint64_t grp_full[4];     // producer -> MMA: K/V group g landed (ring entry g % 4; two arrivals)
    uint64_t s0_full;         // MMA -> softmax 0: S_0,j is in TMEM (and O_0 += P V_{j-1} done)
    uint64_t s1_ring[4];      // MMA -> softmax 1 and producer: S_1,j done (ring entry j % 4), so
                              // every MMA up to step j - 1 is done and its K/V slots are free
    uint64_t p_full[2];       // softmax -> MMA: P_t,j is in TMEM, O_t rescaled if needed
    uint64_t o_last[2];       // MMA -> softmax: the item's last O += P V has landed (one phase per item)
    uint64_t drain;
    uint32_t tmem_slot;
    int abort_flag;
};

// kPersistent: one CTA per SM over a strided share of the items; otherwise
// one item per CTA (grid = items), the loops below run once and the
// hardware's block scheduler balances the SMs
template <int HD, bool kPersistent>
__global__ void __launch_bounds__(kThreads, 1)
attn_tcgen05_kernel(const __grid_constant__ CUtensorMap tm_q0, const __grid_constant__ CUtensorMap tm_q1,
                    const __grid_constant__ CUtensorMap tm_kv0, const __grid_constant__ CUtensorMap tm_kv1,
                    const AttnParams p, int* status) {
    using C = ACfg<HD>;
    static_assert(sizeof(Bars) <= C::kBarBytes, "barrier block too small");
    static_assert(C::kSlots >= 3 && C::kSlots <= kMaxSlots, "K/V ring size");
    constexpr int S = C::kSlots;
    extern __shared__ __align__(1024) uint8_t smem[];
    uint8_t* sQ = smem;                                   // [2][kQBytes]
    uint8_t* sKV = smem + 2 * C::kQBytes;                 // [kSlots][K or V tile]
    Bars& bar = *reinterpret_cast<Bars*>(sKV + S * C::kKBytes);
    volatile int* abort_flag = &bar.abort_flag;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int nt0 = (p.nkv[0] + kBN - 1) / kBN;
    const int ntiles = nt0 + (p.nkv[1] + kBN - 1) / kBN;   // K/V steps per item
    // persistent: this CTA takes items blockIdx.x, blockIdx.x + gridDim.x, ...
    // and runs their K/V steps as one stream; the global step g counts the
    // CTA's steps over its items in order.  A split launch gives every CTA
    // split_first / gridDim.x whole items and CTAs 0 .. 2 split_n - 1 one half
    // item after them (CTA 2 i + h: half h of item split_first + i)
    const int c_ = static_cast<int>(blockIdx.x), g_ = static_cast<int>(gridDim.x);
    const bool split = kPersistent && p.split_n > 0;
    const int nfull = !kPersistent ? (c_ < p.items ? 1 : 0)
                      : split ? p.split_first / g_
                      : p.items > c_ ? (p.items - 1 - c_) / g_ + 1 : 0;
    const bool has_half = split && c_ < 2 * p.split_n;
    const int nitems = nfull + (has_half ? 1 : 0);
    const int half_at = ntiles >> 1;   // the first half covers steps 0 .. half_at - 1
    // K/V steps [j0, j1) of the CTA's k-th item
    auto seg_j0 = [&](int k) { return k < nfull || !(c_ & 1) ? 0 : half_at; };
    auto seg_j1 = [&](int k) { return k < nfull || (c_ & 1) ? ntiles : half_at; };
    const int nsteps = nfull * ntiles + (has_half ? ((c_ & 1) ? ntiles - half_at : half_at) : 0);
    struct Item { int b, h, seg, q0; };   // q0: first query row within the segment
    auto item_of = [&](int k) {
        const int it = k < nfull ? c_ + k * g_ : p.split_first + (c_ >> 1);
        const int qp = it % p.qpairs;
        const int bh = it / p.qpairs;
        Item r;
        r.h = bh % p.heads;
        r.b = bh / p.heads;
        r.seg = qp < p.qpairs0 ? 0 : 1;
        r.q0 = (qp - (r.seg ? p.qpairs0 : 0)) * (2 * kBM);
        return r;
    };

    if (threadIdx.x == 0) {
        *abort_flag = 0;
        if (smem_u32(smem) & 1023u) {   // the swizzled tiles need 1024-byte alignment
            report_status(status, kStatusBadArgument);
            *abort_flag = 1;
        }
        for (int t = 0; t < 2; ++t) mbar_init(&bar.q_full[t], 1);
        for (int g = 0; g < 4; ++g) {
            mbar_init(&bar.grp_full[g], 2);
            mbar_init(&bar.s1_ring[g], 1);
        }
        mbar_init(&bar.s0_full, 1);
        for (int t = 0; t < 2; ++t) {
            mbar_init(&bar.p_full[t], 4);
            mbar_init(&bar.o_last[t], 1);
        }
        mbar_init(&bar.drain, 1);
        fence_mbar_init();
        prefetch_tmap(&tm_q0);
        prefetch_tmap(&tm_q1);
        prefetch_tmap(&tm_kv0);
        prefetch_tmap(&tm_kv1);
    }
    if (warp == 1) {
        tmem_alloc(&bar.tmem_slot, C::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = bar.tmem_slot;
    const bool aborted_at_start = *abort_flag || nsteps == 0;

    auto fail = [&]() {
        report_status(status, kStatusWaitTimeout);
        *abort_flag = 1;
    };

    if (aborted_at_start) {
        // nothing issued
    } else if (warp == 0 && lane == 0) {
        // ------------------------------------------------------------ producer
        auto load_q = [&](int t, const Item& it) {
            mbar_arrive_expect_tx(&bar.q_full[t], C::kQBytes);
            for (int c = 0; c < HD / 64; ++c)
                tma_load_2d(sQ + t * C::kQBytes + c * (kBM * 128), it.seg ? &tm_q1 : &tm_q0, &bar.q_full[t],
                            p.q_col + it.h * HD + c * 64, it.b * p.nq[it.seg] + it.q0 + t * kBM);
        };
        // S_1 of the steps up to c is done: the ring entries are confirmed in
        // step order, so each parity wait is for the entry's current phase
        int seen = -1;
        auto s1_done_upto = [&](int c) {
            for (; seen < c; ++seen)
                if (!mbar_wait(&bar.s1_ring[(seen + 1) & 3], ((seen + 1) >> 2) & 1)) return false;
            return true;
        };
        Item cur = item_of(0);
        load_q(0, cur);
        load_q(1, cur);
        for (int n = 0, k = 0, j = seg_j0(0); n < 2 * nsteps; ++n) {
            const int s = n % S;
            const int g = n >> 1;                 // global step of this K or V tile: item k, local step j
            // item n - S (group c = (n - S + 1) / 2) leaves slot s once the
            // MMAs of group c are done, i.e. once S_1,c is done (S_1,c is the
            // last MMA of step c - 1, and K_0's only readers are S_0,0 and
            // S_1,0)
            if (n >= S && !s1_done_upto((n - S + 1) >> 1)) { fail(); break; }
            const bool new_item = !(n & 1) && j == seg_j0(k) && k > 0;
            if (new_item) cur = item_of(k);
            uint64_t* fb = &bar.grp_full[((n + 1) >> 1) & 3];
            const int ks = j < nt0 ? 0 : 1;
            const int row = cur.b * p.nkv[ks] + (j - (ks ? nt0 : 0)) * kBN;
            const CUtensorMap* tkv = ks ? &tm_kv1 : &tm_kv0;
            const int col = ((n & 1) ? p.v_col : p.k_col) + cur.h * HD;
            uint8_t* dst = sKV + s * C::kKBytes;
            mbar_arrive_expect_tx(fb, C::kKBytes);
            for (int c = 0; c < HD / 64; ++c)
                tma_load_2d(dst + c * (kBN * 128), tkv, fb, col + c * 64, row);
            if (n == 0 || n == 2 * nsteps - 1) mbar_arrive(fb);   // one-item groups: the second arrival
            if (new_item) {
                // the new item's K_0 is on its way; its query tile t is free
                // once S_t of step g - 1 (the previous item's last) is done.
                // With S_1,g-2 (hence S_0,g-2) seen done, the two-phase
                // s0_full stands at step g - 1, and it cannot pass it: S_0,g
                // needs the tile loaded here.
                if (!s1_done_upto(g - 2) || !mbar_wait(&bar.s0_full, (g - 1) & 1)) { fail(); break; }
                load_q(0, cur);
                if (!s1_done_upto(g - 1)) { fail(); break; }
                load_q(1, cur);
            }
            if (n & 1) {
                if (++j == seg_j1(k)) {
                    ++k;
                    j = seg_j0(k);
                }
            }
        }
    } else if (warp == 1 && lane == 0) {
        // ------------------------------------------------------------ MMA issuer
        // Order per query tile t: S_t,0 ; then for each j: O_t += P_t,j V_j ;
        // S_t,j+1.  The two tiles interleave so one tile's MMAs run while the
        // other tile's softmax works.  tcgen05.mma from one thread executes in
        // issue order, so S_t,j+1 overwrites the columns of P_t,j only after
        // O_t += P_t,j V_j has read them.  Operand group j + 1 (V_j, K_j+1)
        // is awaited once per step, before O_0 += P_0,j V_j.
        constexpr uint32_t idesc_s = idesc_bf16_f32(kBM, kBN);
        constexpr uint32_t idesc_o = idesc_bf16_f32(kBM, HD) | (1u << 16);   // B (V) is MN-major
        bool ok = mbar_wait(&bar.q_full[0], 0) && mbar_wait(&bar.q_full[1], 0);
        if (!ok) fail();
        auto group_ready = [&](int g) {
            if (!mbar_wait(&bar.grp_full[g & 3], (g >> 2) & 1)) return false;
            tc_fence_after();
            return true;
        };
        // Descriptors are built once per operand tile; stepping inside a tile
        // adds the byte offset >> 4 to the start-address field (addresses stay
        // below 256 KB, so the field never carries), which keeps the issue
        // cost per MMA to a few instructions.
        const uint64_t desc_q[2] = {smem_desc_k_sw128(smem_u32(sQ)), smem_desc_k_sw128(smem_u32(sQ + C::kQBytes))};
        // S_t,g for global step g
        auto issue_s = [&](int t, int g) {
            const uint64_t dq = desc_q[t];
            const uint64_t dk = smem_desc_k_sw128(smem_u32(sKV + ((2 * g) % S) * C::kKBytes));
            const uint32_t dS = tmem + t * 256;
#pragma unroll
            for (int k = 0; k < HD / 16; ++k) {
                const uint32_t off_q = ((k / 4) * (kBM * 128) + (k % 4) * 32) >> 4;
                const uint32_t off_k = ((k / 4) * (kBN * 128) + (k % 4) * 32) >> 4;
                tc_mma_bf16(dS, dq + off_q, dk + off_k, idesc_s, k != 0 ? 1u : 0u);
            }
            tc_commit(t == 0 ? &bar.s0_full : &bar.s1_ring[g & 3]);
        };
        // O_t += P_t,g V_g (local step j: the item's first step overwrites O_t)
        auto issue_pv = [&](int t, int g, int j) -> bool {
            // P_0,g's arrival also covers operand group g + 1 (V_g and K_g+1)
            if (!mbar_wait(&bar.p_full[t], g & 1)) return false;
            tc_fence_after();
            const uint64_t dv = smem_desc_mn_sw128(smem_u32(sKV + ((2 * g + 1) % S) * C::kKBytes), kBN * 128);
            const uint32_t dO = tmem + t * 256 + C::kColO;
            const uint32_t aP = tmem + t * 256;
#pragma unroll
            for (int k = 0; k < kBN / 16; ++k)   // 16 tokens = 2048 bytes of V per step
                tc_mma_bf16_ts(dO, aP + k * 8, dv + static_cast<uint64_t>(k * (2048 >> 4)), idesc_o,
                               (j | k) != 0 ? 1u : 0u);
            return true;
        };
        if (ok) {
            if (!group_ready(0)) { fail(); ok = false; }
            else {
                issue_s(0, 0);
                issue_s(1, 0);
            }
        }
        // Across items the order stays PV_t,g ; S_t,g+1: the next item's
        // S_t,0 overwrites P_t of the last step only after PV has read it,
        // and its first PV (which overwrites O_t) waits for P_t,0, which the
        // softmax warps publish only after their epilogue has read O_t.  The
        // item's last step is peeled off, so the per-step loop carries no
        // item bookkeeping.
        // j counts the item's steps from its first (a half item has fewer)
        for (int k = 0, g0 = 0; ok && k < nitems; ++k) {
            const int nk = seg_j1(k) - seg_j0(k);
            for (int j = 0; j + 1 < nk; ++j) {
                for (int t = 0; t < 2; ++t) {
                    if (!issue_pv(t, g0 + j, j)) { fail(); ok = false; break; }
                    issue_s(t, g0 + j + 1);
                }
                if (!ok) break;
            }
            if (!ok) break;
            const int j = nk - 1;   // the item's last step
            const bool more = k + 1 < nitems;
            for (int t = 0; t < 2; ++t) {
                if (!issue_pv(t, g0 + j, j)) { fail(); ok = false; break; }
                tc_commit(&bar.o_last[t]);   // O_t of item k final once this lands
                if (more) {   // query tile t of item k + 1
                    if (!mbar_wait(&bar.q_full[t], (k + 1) & 1)) { fail(); ok = false; break; }
                    tc_fence_after();
                    issue_s(t, g0 + nk);
                }
            }
            g0 += nk;
        }
        tc_commit(&bar.drain);
        if (!mbar_wait(&bar.drain, 0)) report_status(status, kStatusWaitTimeout);
    } else if (warp >= 2) {
        // ------------------------------------------------------------ softmax
        const int t = (warp - 2) >> 2;                   // query tile of this warpgroup
        const int q = warp & 3;                          // TMEM lane quarter of this warp
        const int r = q * 32 + lane;                     // query row within the tile = TMEM lane
        const uint32_t tS = tmem + (static_cast<uint32_t>(q * 32) << 16) + t * 256;
        const uint32_t tO = tS + C::kColO;
        bool ok = true;
        for (int k = 0, g0 = 0; ok && k < nitems; ++k) {
            float m_used = -INFINITY;
            float l = 0.f;
            const int j0 = seg_j0(k), j1 = seg_j1(k);
            for (int j = j0; j < j1; ++j) {
                const int g = g0 + (j - j0);   // global step
                // S_t,g ready; O_t += P_t,g-1 V_g-1 has completed as well
                if (!(t == 0 ? mbar_wait(&bar.s0_full, g & 1) : mbar_wait(&bar.s1_ring[g & 3], (g >> 2) & 1))) {
                    fail();
                    ok = false;
                    break;
                }
                tc_fence_after();
                uint32_t sr[kBN];
                tmem_ld_x128(tS, sr);
                tmem_ld_wait();

                const int ks = j < nt0 ? 0 : 1;
                const int valid = p.nkv[ks] - (j - (ks ? nt0 : 0)) * kBN;   // columns < valid are real tokens
                if (valid < kBN) {
#pragma unroll
                    for (int i = 0; i < kBN; ++i)
                        if (i >= valid) sr[i] = __float_as_uint(-INFINITY);
                }
                auto row_max = [&]() {
                    float mc[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                    for (int i = 0; i < kBN; i += 8) {
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            mc[k] = max3(mc[k], __uint_as_float(sr[i + 2 * k]), __uint_as_float(sr[i + 2 * k + 1]));
                    }
                    return max3(mc[0], mc[1], fmaxf(mc[2], mc[3])) * p.scale_log2;
                };
                // P = exp2(S scale - m) packed over the front of sr; returns the row sum
                auto exps = [&](float m) {
                    const float2 c2 = make_float2(p.scale_log2, p.scale_log2);
                    const float2 nm2 = make_float2(-m, -m);
                    float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                                     make_float2(0.f, 0.f)};
#pragma unroll
                    for (int i = 0; i < kBN; i += 2) {
                        const float2 x = __ffma2_rn(make_float2(__uint_as_float(sr[i]), __uint_as_float(sr[i + 1])), c2, nm2);
                        const float2 e = make_float2(ex2(x.x), ex2(x.y));
                        acc[(i >> 1) & 3] = __fadd2_rn(acc[(i >> 1) & 3], e);
                        sr[i / 2] = pack_bf16x2(e.x, e.y);
                    }
                    const float2 a01 = __fadd2_rn(acc[0], acc[1]);
                    const float2 a23 = __fadd2_rn(acc[2], acc[3]);
                    return (a01.x + a01.y) + (a23.x + a23.y);
                };
                // Softmax is unchanged by the reference m subtracted before the
                // exponentials, so after the first tile the row keeps its first
                // maximum as the reference and skips the max pass.  Later scores
                // may exceed it: P up to 2^40 is exact enough in bf16 / fp32, and
                // a tile whose row sum passes 2^40 (or overflows) is redone with
                // the true maximum, rescaling l and O.
                if (j == j0) m_used = row_max();
                float lt = exps(m_used);
                if (j > j0 && __any_sync(0xffffffffu, !(lt <= 0x1p40f))) {
                    tmem_ld_x128(tS, sr);
                    tmem_ld_wait();
                    if (valid < kBN) {
#pragma unroll
                        for (int i = 0; i < kBN; ++i)
                            if (i >= valid) sr[i] = __float_as_uint(-INFINITY);
                    }
                    const float m_new = fmaxf(m_used, row_max());
                    const float alpha = ex2(m_used - m_new);
                    lt = exps(m_new);
                    l *= alpha;
                    m_used = m_new;
#pragma unroll 1
                    for (int c = 0; c < HD; c += 32) {
                        uint32_t o[32];
                        tmem_ld_x32(tO + c, o);
                        tmem_ld_wait();
#pragma unroll
                        for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
                        tmem_st_x32(tO + c, o);
                    }
                }
                l += lt;
                // P_t,j (bf16 pairs) over the first kBN/2 columns of S_t
#pragma unroll
                for (int c = 0; c < kBN / 2; c += 32) tmem_st_x32(tS + c, &sr[c]);
                tmem_st_wait();
                tc_fence_before();
                // tile 0 also checks operand group g + 1 (V_g, K_g+1): the MMA
                // thread issues O_0 += P_0,g V_g and S_0,g+1 on this arrival alone
                if (!warp_wait(&bar.grp_full[(g + 1) & 3], ((g + 1) >> 2) & 1, t == 0, lane)) {
                    fail();
                    ok = false;
                    break;
                }
                if (lane == 0) mbar_arrive(&bar.p_full[t]);
            }
            if (!ok) break;
            g0 += j1 - j0;
            // ---- epilogue: O / l -> bf16, after the item's last O += P V, and
            // the row's log-sum-exp m + log2(l) (base 2) when it is asked for.
            // The next item's first O += P V waits for this warpgroup's P, so it
            // cannot overwrite O_t before these loads.
            if (!mbar_wait(&bar.o_last[t], k & 1)) {
                fail();
                ok = false;
                break;
            }
            tc_fence_after();
            const Item it = item_of(k);
            const int row = it.q0 + t * kBM + r;
            const bool live = row < p.nq[it.seg];
            const int64_t grow = static_cast<int64_t>(it.b) * p.nq[it.seg] + row;
            __nv_bfloat16* dst = p.out[it.seg] + grow * p.ldo[it.seg] + it.h * HD;
            __nv_bfloat16* dst_lo =
                p.out_lo[it.seg] ? p.out_lo[it.seg] + grow * p.ldo_lo[it.seg] + it.h * HD : nullptr;
            float* lse_at = p.lse && live
                                ? p.lse + (static_cast<int64_t>(it.b) * p.heads + it.h) * p.lse_rows +
                                      p.lse_base[it.seg] + row
                                : nullptr;
            // eight outputs from column c0 as bf16, and what bf16 dropped (itself
            // in bf16) when the low part is asked for
            auto put8 = [&](int c0, const float* f) {
                const uint4 hi = make_uint4(pack_bf16x2(f[0], f[1]), pack_bf16x2(f[2], f[3]),
                                            pack_bf16x2(f[4], f[5]), pack_bf16x2(f[6], f[7]));
                *reinterpret_cast<uint4*>(dst + c0) = hi;
                if (dst_lo) {
                    const uint32_t hw[4] = {hi.x, hi.y, hi.z, hi.w};
                    uint32_t lw[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const float2 rr = unpack_bf16x2(hw[i]);
                        lw[i] = pack_bf16x2(f[2 * i] - rr.x, f[2 * i + 1] - rr.y);
                    }
                    *reinterpret_cast<uint4*>(dst_lo + c0) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
                }
            };
            if (k < nfull) {
                const float inv = 1.f / l;
                if (lse_at) *lse_at = m_used + log2f(l);
#pragma unroll 1
                for (int c = 0; c < HD; c += 32) {
                    uint32_t o[32];
                    tmem_ld_x32(tO + c, o);
                    tmem_ld_wait();
                    if (live) {
#pragma unroll
                        for (int w = 0; w < 4; ++w) {
                            float f[8];
#pragma unroll
                            for (int i = 0; i < 8; ++i) f[i] = __uint_as_float(o[8 * w + i]) * inv;
                            put8(c + 8 * w, f);
                        }
                    }
                }
            } else {
                // half of a split item: publish this half's unnormalised O_t
                // rows with their (m, l); the warp that finds the other half
                // already published merges the two (the partial softmaxes of
                // two key ranges: weights 2^(m_h - max(m_0, m_1)), always in
                // half order, so the result does not depend on which came last)
                const int si = c_ >> 1, hh = c_ & 1;
                const size_t prow = (static_cast<size_t>(si * 2 + hh) * 2 + t) * kBM + r;
                float* mine = p.part + prow * HD;
#pragma unroll 1
                for (int c = 0; c < HD; c += 32) {
                    uint32_t o[32];
                    tmem_ld_x32(tO + c, o);
                    tmem_ld_wait();
#pragma unroll
                    for (int w = 0; w < 8; ++w)
                        *reinterpret_cast<float4*>(mine + c + 4 * w) =
                            make_float4(__uint_as_float(o[4 * w]), __uint_as_float(o[4 * w + 1]),
                                        __uint_as_float(o[4 * w + 2]), __uint_as_float(o[4 * w + 3]));
                }
                p.part_ml[prow] = make_float2(m_used, l);
                __threadfence();
                __syncwarp();
                unsigned prev = 0;
                if (lane == 0) prev = atomicAdd(&p.tickets[(si * 2 + t) * 4 + q], 1u);
                prev = __shfl_sync(0xffffffffu, prev, 0);
                if (prev == 1u) {
                    __threadfence();
                    const size_t orow = (static_cast<size_t>(si * 2 + (hh ^ 1)) * 2 + t) * kBM + r;
                    const float* other = p.part + orow * HD;
                    const float2 mo = __ldcg(p.part_ml + orow);
                    const float m0 = hh ? mo.x : m_used, l0 = hh ? mo.y : l;
                    const float m1 = hh ? m_used : mo.x, l1 = hh ? l : mo.y;
                    const float mm = fmaxf(m0, m1);
                    const float w0 = ex2(m0 - mm), w1 = ex2(m1 - mm);
                    const float lsum = __fmaf_rn(l1, w1, __fmul_rn(l0, w0));
                    const float inv = 1.f / lsum;
                    if (lse_at) *lse_at = mm + log2f(lsum);
#pragma unroll 1
                    for (int c = 0; c < HD; c += 32) {
                        uint32_t o[32];
                        tmem_ld_x32(tO + c, o);
                        tmem_ld_wait();
                        if (live) {
#pragma unroll
                            for (int w = 0; w < 4; ++w) {
                                const float4 a = __ldcg(reinterpret_cast<const float4*>(other + c + 8 * w));
                                const float4 b = __ldcg(reinterpret_cast<const float4*>(other + c + 8 * w + 4));
                                const float ot[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
                                float f[8];
#pragma unroll
                                for (int i = 0; i < 8; ++i) {
                                    const float own = __uint_as_float(o[8 * w + i]);
                                    const float o0 = hh ? ot[i] : own, o1 = hh ? own : ot[i];
                                    f[i] = __fmul_rn(__fmaf_rn(o1, w1, __fmul_rn(o0, w0)), inv);
                                }
                                put8(c + 8 * w, f);
                            }
                        }
                    }
                }
            }
            tmem_ld_wait();
            tc_fence_before();
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

// The launch variant and grid for `items` work items of `steps` K/V steps
// on `sms` SMs (forced: the test override, 0 for the launcher's own choice).
struct LaunchPlan {
    bool persistent;
    int64_t grid;
    int64_t split_first, split_n;   // split_n > 0: items split_first .. items - 1 run as two halves each
};
LaunchPlan launch_plan(int64_t items, int sms, int steps, int forced, bool have_ws) {
    LaunchPlan r{};
    r.persistent = forced ? forced == 1 || forced == 3
                          : items < static_cast<int64_t>(kPersistentItemsPerSm) * sms || steps <= kPersistentMaxSteps;
    r.grid = r.persistent ? (items < sms ? items : sms) : items;
    if (r.persistent && (forced == 0 || forced == 3) && have_ws && steps >= 2) {
        const int64_t rounds = items / sms, rest = items % sms;
        if (rest > 0 && 2 * rest <= sms && rest <= kSplitMaxItems) {
            r.split_first = rounds * sms;
            r.split_n = rest;
            r.grid = rounds > 0 ? sms : 2 * rest;
        }
    }
    return r;
}

// Scratch of a split launch: per split item, both halves' unnormalised O of
// both query tiles (fp32), their (m, l), and 8 tickets.
size_t split_part_bytes(int hd) { return static_cast<size_t>(kSplitMaxItems) * 2 * 2 * kBM * hd * sizeof(float); }
size_t split_ml_bytes() { return static_cast<size_t>(kSplitMaxItems) * 2 * 2 * kBM * sizeof(float2); }

template <int HD>
int launch_attn(const AttnSpec& a, cudaStream_t stream) {
    using C = ACfg<HD>;
    for (auto* f : {attn_tcgen05_kernel<HD, true>, attn_tcgen05_kernel<HD, false>})
        if (cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) != cudaSuccess)
            return set_error(FF_ERR_CUDA, "attention: cannot set shared memory size");
    CUtensorMap tq[2], tkv[2];
    for (int i = 0; i < 2; ++i) {
        // an empty segment still needs a valid map: point it at the other one
        const AttnQuerySeg& q = a.q[i].n > 0 ? a.q[i] : a.q[1 - i];
        int rc = make_tmap_bf16(&tq[i], q.buf, static_cast<int64_t>(a.B) * q.n, q.ld, q.ld, kBM);
        if (rc) return rc;
        const AttnKvSeg& kv = a.kv[i].n > 0 ? a.kv[i] : a.kv[1 - i];
        rc = make_tmap_bf16(&tkv[i], kv.buf, static_cast<int64_t>(a.B) * kv.n, kv.ld, kv.ld, kBN);
        if (rc) return rc;
    }
    AttnParams p;
    for (int i = 0; i < 2; ++i) {
        p.nq[i] = a.q[i].n;
        p.nkv[i] = a.kv[i].n;
        p.out[i] = a.q[i].out;
        p.ldo[i] = a.q[i].ldo;
        p.out_lo[i] = a.q[i].out_lo;
        p.ldo_lo[i] = a.q[i].ldo_lo;
    }
    p.qpairs0 = (a.q[0].n + 2 * kBM - 1) / (2 * kBM);
    p.qpairs = p.qpairs0 + (a.q[1].n + 2 * kBM - 1) / (2 * kBM);
    p.heads = a.heads;
    const int64_t items = static_cast<int64_t>(p.qpairs) * a.heads * a.B;
    if (items >= (int64_t{1} << 31)) return set_error(FF_ERR_INVALID_ARG, "attention: too many query blocks");
    p.items = static_cast<int>(items);
    p.lse = a.lse;
    p.lse_rows = attn_lse_rows(a.q[0].n, a.q[1].n);
    p.lse_base[0] = 0;
    p.lse_base[1] = attn_pad128(a.q[0].n);
    p.q_col = a.q_col;
    p.k_col = a.k_col;
    p.v_col = a.v_col;
    p.scale_log2 = static_cast<float>(1.4426950408889634 / sqrt(static_cast<double>(HD)));
    // Persistent (one CTA per SM, the kernel takes the whole shared memory,
    // each running a strided share of the items) when there are few items per
    // SM or the items are short: the first K/V and query loads and the
    // epilogue of each item then overlap its neighbours (Flux block, 11 items
    // of 36 steps per SM: 731 -> 707 us; 24-block Flux rollout, 30 items of
    // 12 steps per SM: 762 -> 723 us).  With many long items per SM the
    // hardware's block scheduler, which hands the next item to whichever SM
    // frees first, balances the SMs better than a fixed stride and the
    // overlap is worth little (WAN self-attention, 34 items of 256 steps per
    // SM: 13.8 ms one item per CTA, 14.0 ms persistent).
    //
    // A persistent launch whose items do not fill a whole last round (L of
    // the G SMs busy, 2 L <= G) runs those L items as 2 L halves of their K/V
    // steps on 2 L CTAs, given the caller's scratch: Flux block, 1728 items =
    // 11 rounds + 56, so the last round ends after half an item.
    const int steps = (a.kv[0].n + kBN - 1) / kBN + (a.kv[1].n + kBN - 1) / kBN;
    const bool have_ws = a.split_ws && a.split_ws_bytes >= attention_split_ws_bytes(HD);
    const LaunchPlan plan =
        launch_plan(items, num_sms(), steps, g_launch_override.load(std::memory_order_relaxed), have_ws);
    const bool persistent = plan.persistent;
    p.split_first = static_cast<int>(plan.split_first);
    p.split_n = static_cast<int>(plan.split_n);
    p.part = nullptr;
    p.part_ml = nullptr;
    p.tickets = nullptr;
    if (plan.split_n > 0) {
        uint8_t* ws = static_cast<uint8_t*>(a.split_ws);
        p.part = reinterpret_cast<float*>(ws);
        p.part_ml = reinterpret_cast<float2*>(ws + split_part_bytes(HD));
        p.tickets = reinterpret_cast<unsigned*>(ws + split_part_bytes(HD) + split_ml_bytes());
        if (cudaMemsetAsync(p.tickets, 0, static_cast<size_t>(plan.split_n) * 8 * sizeof(unsigned), stream) !=
            cudaSuccess)
            return set_error(FF_ERR_CUDA, "attention: cannot clear the split tickets");
    }
    const int grid = static_cast<int>(plan.grid);
    const double nkv = static_cast<double>(a.kv[0].n + a.kv[1].n);
    const double nq = static_cast<double>(a.q[0].n + a.q[1].n);
    ProfScope prof(stream, "attention", 4.0 * a.B * a.heads * nq * nkv * HD,
                   2.0 * a.B * a.heads * HD * (2.0 * nq + 2.0 * nkv));
    if (persistent)
        attn_tcgen05_kernel<HD, true><<<grid, kThreads, C::kSmemBytes, stream>>>(tq[0], tq[1], tkv[0], tkv[1], p,
                                                                                  device_status_ptr());
    else
        attn_tcgen05_kernel<HD, false><<<grid, kThreads, C::kSmemBytes, stream>>>(tq[0], tq[1], tkv[0], tkv[1], p,
                                                                                   device_status_ptr());
    return check_launch("attn_tcgen05_kernel");
}

}  // namespace

int attention_launch_override(int mode) { return g_launch_override.exchange(mode); }

}  // namespace ff

// The attention launcher's choice for a launch of `items` query blocks of
// `steps` K/V steps on `sms` SMs (host arithmetic only; for tests).
extern "C" int ff_debug_attention_plan(int64_t items, int sms, int steps, int have_ws, int mode, int* persistent,
                                       int64_t* grid, int64_t* split_first, int64_t* split_n) {
    using namespace ff;
    if (items <= 0 || sms <= 0 || steps <= 0 || mode < 0 || mode > 3 || !persistent || !grid || !split_first ||
        !split_n)
        return set_error(FF_ERR_INVALID_ARG, "attention plan: bad arguments");
    const LaunchPlan r = launch_plan(items, sms, steps, mode, have_ws != 0);
    *persistent = r.persistent ? 1 : 0;
    *grid = r.grid;
    *split_first = r.split_first;
    *split_n = r.split_n;
    return FF_OK;
}

namespace ff {

size_t attention_split_ws_bytes(int head_dim) {
    return split_part_bytes(head_dim) + split_ml_bytes() + static_cast<size_t>(kSplitMaxItems) * 8 * sizeof(unsigned);
}

int attention_general(const AttnSpec& a, cudaStream_t stream) {
    if (a.B <= 0 || a.heads <= 0 || a.B > 65535 || a.heads > 65535)
        return set_error(FF_ERR_INVALID_ARG, "attention: bad batch / heads");
    for (int i = 0; i < 2; ++i) {
        if (a.q[i].n < 0 || a.kv[i].n < 0) return set_error(FF_ERR_INVALID_ARG, "attention: negative token count");
        if (a.q[i].n && (!a.q[i].buf || !a.q[i].out || !aligned16(a.q[i].out) || a.q[i].ld % 8 || a.q[i].ldo % 8))
            return set_error(FF_ERR_INVALID_ARG, "attention: bad query segment %d", i);
        if (a.q[i].n && a.q[i].out_lo && (!aligned16(a.q[i].out_lo) || a.q[i].ldo_lo % 8))
            return set_error(FF_ERR_INVALID_ARG, "attention: bad low-part output of query segment %d", i);
        if (a.kv[i].n && (!a.kv[i].buf || a.kv[i].ld % 8))
            return set_error(FF_ERR_INVALID_ARG, "attention: bad key/value segment %d", i);
    }
    if (a.q[0].n + a.q[1].n <= 0 || a.kv[0].n + a.kv[1].n <= 0)
        return set_error(FF_ERR_INVALID_ARG, "attention: no queries or no keys");
    if (a.q_col % 64 || a.k_col % 64 || a.v_col % 64)
        return set_error(FF_ERR_UNSUPPORTED, "attention: column offsets must be multiples of 64");
    const int64_t hd = static_cast<int64_t>(a.heads) * a.head_dim;
    for (int i = 0; i < 2; ++i) {
        if (a.q[i].n && a.q_col + hd > a.q[i].ld) return set_error(FF_ERR_INVALID_ARG, "attention: q columns exceed ld");
        if (a.kv[i].n && (a.k_col + hd > a.kv[i].ld || a.v_col + hd > a.kv[i].ld))
            return set_error(FF_ERR_INVALID_ARG, "attention: k/v columns exceed ld");
    }
    if (a.split_ws && !aligned16(a.split_ws)) return set_error(FF_ERR_INVALID_ARG, "attention: misaligned split scratch");
    if (a.head_dim == 128) return launch_attn<128>(a, stream);
    if (a.head_dim == 64) return launch_attn<64>(a, stream);
    return set_error(FF_ERR_UNSUPPORTED, "attention: head_dim %d", a.head_dim);
}

int attention(const AttnSegment& s0, const AttnSegment& s1, int B, int heads, int head_dim, int H,
              cudaStream_t stream, float* lse, void* split_ws, size_t split_ws_bytes) {
    AttnSpec a;
    a.lse = lse;
    a.split_ws = split_ws;
    a.split_ws_bytes = split_ws_bytes;
    const AttnSegment* seg[2] = {&s0, &s1};
    for (int i = 0; i < 2; ++i) {
        a.q[i] = AttnQuerySeg{seg[i]->qkv, seg[i]->ld, seg[i]->n, seg[i]->out, seg[i]->ldo, seg[i]->out_lo,
                              seg[i]->ldo_lo};
        a.kv[i] = AttnKvSeg{seg[i]->qkv, seg[i]->ld, seg[i]->n};
    }
    a.q_col = 0;
    a.k_col = H;
    a.v_col = 2 * H;
    a.B = B;
    a.heads = heads;
    a.head_dim = head_dim;
    return attention_general(a, stream);
}

}  // namespace ff

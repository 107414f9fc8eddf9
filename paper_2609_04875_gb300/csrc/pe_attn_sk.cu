// Persistent stream-K replay attention on sm_103a (tcgen05 + TMEM + TMA).
//
// Same result as replay_attn_kernel (pe_attn.cu): for the last n_q positions
// of a sequence, query i at position len-n_q+i and q-head h attend the keys
// 0..len-n_q+i of kv-head h / (Hq/Hkv), O = softmax(scale q K^T) V, fp32
// accumulation, bf16 output (Alg. 1 replay loop; Sec. 3.2 re-prefill on the
// cropped cache).  What differs is how the work is laid out on the SMs.
//
// One CTA per SM.  A work unit is (sequence, kv-head, pair of 128-row q-tiles)
// and loads the key tiles [0, n) of its pair; CTA c takes a contiguous
// stretch of (unit, key tile) work, chosen on the host so that every CTA has
// about the same number of key tiles plus per-unit overhead.  A unit cut by a
// stretch boundary is computed in pieces (key ranges) by consecutive CTAs, each
// writing fp32 partials (O / l and the row's log2-sum-exp); per warp of 32 rows
// a ticket counts the parts written, and the warp that writes a unit's last
// part merges the parts into the bf16 output (no combine launch).  Whole units
// write bf16 output directly.  So the last wave of a launch is as full as the
// first, and a CTA's next unit starts loading while its previous unit's last
// tile and epilogue run (no CTA launch, TMEM allocation or barrier set-up
// between units).
//
// Roles (320 threads) as in replay_attn_kernel: softmax warpgroups 0 and 1
// (one per q-tile, thread r owns row r), producer warp 8 (page table -> TMA
// boxes), MMA warp 9 (one thread issues tcgen05.mma).  Every role walks the
// same sequence of pieces, computed from the kernel parameters; barrier phases
// run on across pieces (per q-tile tile counts for S / P / O, a global key
// tile count for the K and V rings, a piece count for Q).  Two more barriers
// than the one-unit kernel: q_empty (the piece's last S GEMMs are done, so the
// next piece's Q may load while its last tile's softmax and P V run) and o_free[t] (the softmax warps have read O_t out of
// TMEM, so the next piece's first P V GEMM may overwrite it).
//
// Key tiles start at logical key 0 (multiples of 128 keys) whatever the
// pieces, so a whole unit's rows are computed exactly as by the one-unit
// kernel.  Every wait is bounded (kWaitNs); on expiry the CTA records a status
// code, all roles leave their loops, copies in flight get a bounded drain, and
// TMEM is freed before exit.
#include <cuda_bf16.h>

#include "dev_common.cuh"
#include "pe_internal.h"
#include "ptx.cuh"

namespace pe {
namespace {

constexpr float kTileSumLimit = 1.8446744e19f;  // 2^64: larger tile sums move the reference
constexpr int kThreads = 320;

template <int HD>
struct SkCfg {
    static constexpr int kRegions = HD / 64;            // 128-byte swizzle atoms along d
    static constexpr int kTileBytes = kBM * HD * 2;     // one Q, K or V tile (128 rows)
    static constexpr int kRegionBytes = kBM * 128;      // 128 rows x 128 bytes
    static constexpr int kStages = (HD == 128) ? 2 : 3; // K ring and V ring depth
    static constexpr int kOffQ = 0;                     // Q_0, Q_1
    static constexpr int kOffK = kOffQ + 2 * kTileBytes;
    static constexpr int kOffV = kOffK + kStages * kTileBytes;
    static constexpr int kOffBar = kOffV + kStages * kTileBytes;
    // q_full, q_empty, k_full[S], k_empty[S], v_full[S], v_empty[S], s_full[2], p_full[2], o_done[2], o_free[2]
    static constexpr int kNumBars = 2 + 4 * kStages + 8;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;  // tmem slot, abort flag
    static constexpr int kSmemBytes = kOffMisc + 16;
    static constexpr int kDynSmem = kSmemBytes + 1024;       // alignment slack
    static constexpr uint32_t kTmemCols = 512;
    static_assert(kDynSmem <= 232448, "shared memory budget");
};

// One piece of a CTA's stretch: unit `u`, key tiles [lo, hi).
struct Piece {
    int u, lo, hi;
    int slot, part;        // slot < 0: the whole unit, bf16 output
};

// Geometry of one q-tile of a piece.
struct QGeo {
    int qt;                // q-tile index within the sequence (-1: absent)
    int q_first, q_last;   // first / last valid query of the tile
    int pos_first;         // absolute position of the first query
    int ntiles;            // key tiles of this piece that the q-tile attends (from the piece's lo)
};

struct UnitGeo {
    int si, kvh, pair;
    int n_all;             // key tiles the unit loads (its heavier q-tile's causal tile count)
};

__device__ __forceinline__ UnitGeo unit_geo(const AttnParams &p, int u)
{
    UnitGeo U;
    int si = 0, hi = p.n_seqs;  // the last sequence whose first unit is at most u
    while (hi - si > 1) {
        const int mid = (si + hi) >> 1;
        if (p.seqs[mid].item0 <= u) si = mid;
        else hi = mid;
    }
    const AttnSeq &sq = p.seqs[si];
    const int local = u - sq.item0;
    U.si = si;
    U.kvh = local % p.hkv;
    U.pair = sq.pair_top - 1 - local / p.hkv;
    const int bmq = kBM / p.group;
    const int qt_last = min(2 * U.pair + 1, sq.n_qtiles - 1);
    const int q_last = min((qt_last + 1) * bmq, sq.n_q) - 1;
    U.n_all = (sq.n_keys - sq.n_q + q_last + 1 + kBN - 1) / kBN;
    return U;
}

__device__ __forceinline__ QGeo q_geo(const AttnParams &p, const AttnSeq &sq, int pair, int t, int lo, int hi)
{
    QGeo G;
    const int bmq = kBM / p.group;
    const int qt = 2 * pair + t;
    if (qt < sq.n_qtiles) {
        G.qt = qt;
        G.q_first = qt * bmq;
        G.q_last = min(G.q_first + bmq, sq.n_q) - 1;
        G.pos_first = sq.n_keys - sq.n_q + G.q_first;
        const int nkt = (sq.n_keys - sq.n_q + G.q_last + 1 + kBN - 1) / kBN;
        G.ntiles = max(0, min(hi, nkt) - lo);
    } else {
        G.qt = -1;
        G.q_first = G.q_last = G.pos_first = 0;
        G.ntiles = 0;
    }
    return G;
}

// The k-th piece of this CTA's work (k from 0): whole units in the lockstep
// rounds, then the pieces of its tail stretch cw; false past the end.
__device__ __forceinline__ bool piece_of(const SkParams &P, const SkCta &cw, int k, Piece &pc, UnitGeo &U)
{
    const AttnParams &p = P.a;
    if (k < P.rounds) {
        const int cta = blockIdx.x;
        pc.u = k * P.n_ctas + ((k & 1) ? P.n_ctas - 1 - cta : cta);
        U = unit_geo(p, pc.u);
        pc.lo = 0;
        pc.hi = U.n_all;
        pc.slot = -1;
        pc.part = 0;
        return true;
    }
    k -= P.rounds;
    const int u = cw.u0 + k;
    if (u > cw.u1 || (u == cw.u1 && cw.t1 == 0 && u != cw.u0)) return false;
    U = unit_geo(p, u);
    pc.u = u;
    pc.lo = (k == 0) ? cw.t0 : 0;
    pc.hi = (u == cw.u1 && cw.t1 > 0) ? cw.t1 : U.n_all;
    if (k == 0) {
        pc.slot = cw.slot0;
        pc.part = cw.part0;
    } else if (u == cw.u1) {
        pc.slot = cw.slot1;
        pc.part = cw.part1;
    } else {
        pc.slot = -1;
        pc.part = 0;
    }
    return pc.hi > pc.lo;
}

// Merge of one row of a cut unit's q-tile t from its n parts (slot `slot`):
// O = sum_p 2^(lse_p - m) O_p / sum_p 2^(lse_p - m), m = max_p lse_p, where
// O_p is part p's O / l and lse_p its log2-sum-exp (-inf: no visible key).
// The parts were written by other CTAs of this grid: read through L2.  Out of
// line (as merge_own_row), so that their accumulators do not add to the
// register pressure of the kernel's tile loop (halves the kernel's spills).
template <int HD>
__device__ __noinline__ void merge_parts_row(const SkParams &P, int slot, int t, int row, int n, uint4 *dst)
{
    const AttnParams &p = P.a;
    constexpr int64_t kStride = 2 * kBM;  // rows from one part to the next
    const int64_t r0 = static_cast<int64_t>(slot) * P.max_parts * kStride + t * kBM + row;
    float mx = -INFINITY;
    for (int q = 0; q < n; ++q) mx = fmaxf(mx, __ldcg(p.part_lse + r0 + q * kStride));
    float den = 0.f;
    for (int q = 0; q < n; ++q) {
        const float lse = __ldcg(p.part_lse + r0 + q * kStride);
        if (lse != -INFINITY) den += ex2(lse - mx);
    }
    const float inv = den > 0.f ? 1.0f / den : 0.f;
    constexpr int kCh = 64;  // columns per pass
#pragma unroll 1
    for (int c0 = 0; c0 < HD; c0 += kCh) {
        float acc[kCh];
#pragma unroll
        for (int i = 0; i < kCh; ++i) acc[i] = 0.f;
#pragma unroll 1
        for (int q = 0; q < n; ++q) {
            const float lse = __ldcg(p.part_lse + r0 + q * kStride);
            if (lse == -INFINITY) continue;
            const float w = ex2(lse - mx);
#pragma unroll
            for (int i = 0; i < kCh / 4; ++i) {
                const float4 v = __ldcg(part_chunk<HD>(p.part_o, r0 + q * kStride, c0 / 4 + i));
                acc[4 * i + 0] += w * v.x;
                acc[4 * i + 1] += w * v.y;
                acc[4 * i + 2] += w * v.z;
                acc[4 * i + 3] += w * v.w;
            }
        }
#pragma unroll
        for (int i = 0; i < kCh / 8; ++i)
            dst[c0 / 8 + i] = make_uint4(pack_bf16(acc[8 * i + 0] * inv, acc[8 * i + 1] * inv),
                                         pack_bf16(acc[8 * i + 2] * inv, acc[8 * i + 3] * inv),
                                         pack_bf16(acc[8 * i + 4] * inv, acc[8 * i + 5] * inv),
                                         pack_bf16(acc[8 * i + 6] * inv, acc[8 * i + 7] * inv));
    }
}

// The same merge by the warp whose part of the unit comes last (n <= 4 parts):
// its own part is still in TMEM (unnormalised O at tO, with l and m_ref) and
// is not written; the other parts are read through L2.  Own values are formed
// exactly as a written part holds them (O * (1 / l), m_ref + log2 l) and the
// parts are summed in index order, so the bits do not depend on which part's
// warp merges.  has_tmem = false: this piece has no key for the q-tile (TMEM
// is not read).  kOwn = false: every part, this warp's too, is read from L2
// (own, tO, l and m_ref unused).  Whole warp.
constexpr int kMaxOwnMergeParts = 4;
template <int HD, bool kOwn>
__device__ __noinline__ void merge_own_row(const SkParams &P, int slot, int t, int row, int n, int own,
                                              bool has_tmem, uint32_t tO, float l, float m_ref, bool valid,
                                              uint4 *dst)
{
    if (!kOwn) own = -1;
    const AttnParams &p = P.a;
    constexpr int64_t kStride = 2 * kBM;
    const int64_t r0 = static_cast<int64_t>(slot) * P.max_parts * kStride + t * kBM + row;
    const float lse_own = (has_tmem && l > 0.f) ? m_ref + __log2f(l) : -INFINITY;
    const float inv_own = l > 0.f ? 1.0f / l : 0.f;
    float lse[kMaxOwnMergeParts];
#pragma unroll
    for (int q = 0; q < kMaxOwnMergeParts; ++q)
        lse[q] = q == own ? lse_own : (valid && q < n) ? __ldcg(p.part_lse + r0 + q * kStride) : -INFINITY;
    float mx = -INFINITY;
#pragma unroll
    for (int q = 0; q < kMaxOwnMergeParts; ++q)
        if (q < n) mx = fmaxf(mx, lse[q]);
    float den = 0.f;
#pragma unroll
    for (int q = 0; q < kMaxOwnMergeParts; ++q)
        if (q < n && lse[q] != -INFINITY) den += ex2(lse[q] - mx);
    const float inv = den > 0.f ? 1.0f / den : 0.f;
    constexpr int kCh = 64;  // columns per pass
#pragma unroll 1
    for (int c0 = 0; c0 < HD; c0 += kCh) {
        float acc[kCh];
#pragma unroll
        for (int i = 0; i < kCh; ++i) acc[i] = 0.f;
#pragma unroll
        for (int q = 0; q < kMaxOwnMergeParts; ++q) {
            if (q >= n) break;
            if (kOwn && q == own) {  // warp-uniform: the TMEM loads are collective
                if (has_tmem) {
#pragma unroll
                    for (int h = 0; h < kCh; h += 32) {
                        float o[32];
                        ptx::tmem_ld32(tO + c0 + h, o);
                        ptx::tmem_wait_ld();
                        if (lse[q] != -INFINITY) {
                            const float w = ex2(lse[q] - mx);
#pragma unroll
                            for (int i = 0; i < 32; ++i) acc[h + i] += w * (o[i] * inv_own);
                        }
                    }
                }
            } else if (valid && lse[q] != -INFINITY) {
                const float w = ex2(lse[q] - mx);
#pragma unroll
                for (int i = 0; i < kCh / 4; ++i) {
                    const float4 v = __ldcg(part_chunk<HD>(p.part_o, r0 + q * kStride, c0 / 4 + i));
                    acc[4 * i + 0] += w * v.x;
                    acc[4 * i + 1] += w * v.y;
                    acc[4 * i + 2] += w * v.z;
                    acc[4 * i + 3] += w * v.w;
                }
            }
        }
        if (valid) {
#pragma unroll
            for (int i = 0; i < kCh / 8; ++i)
                dst[c0 / 8 + i] = make_uint4(pack_bf16(acc[8 * i + 0] * inv, acc[8 * i + 1] * inv),
                                             pack_bf16(acc[8 * i + 2] * inv, acc[8 * i + 3] * inv),
                                             pack_bf16(acc[8 * i + 4] * inv, acc[8 * i + 5] * inv),
                                             pack_bf16(acc[8 * i + 6] * inv, acc[8 * i + 7] * inv));
        }
    }
}

template <int HD>
__global__ void __launch_bounds__(kThreads, 1)
    replay_attn_sk_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                          const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ SkParams P)
{
    using C = SkCfg<HD>;
    const AttnParams &p = P.a;
    const SkCta &cw = P.cta[blockIdx.x];
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = ptx::smem_addr(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;
    uint8_t *smem = smem_raw + (sbase - raw);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int g = p.group;

    const uint32_t q_smem = sbase + C::kOffQ;
    const uint32_t k_smem0 = sbase + C::kOffK;
    const uint32_t v_smem0 = sbase + C::kOffV;
    const uint32_t bar0 = sbase + C::kOffBar;
    const uint32_t b_q_full = bar0;
    const uint32_t b_q_empty = bar0 + 8;
    const uint32_t b_k_full = bar0 + 16;
    const uint32_t b_k_empty = b_k_full + 8 * C::kStages;
    const uint32_t b_v_full = b_k_empty + 8 * C::kStages;
    const uint32_t b_v_empty = b_v_full + 8 * C::kStages;
    const uint32_t b_s_full = b_v_empty + 8 * C::kStages;  // [2]
    const uint32_t b_p_full = b_s_full + 16;               // [2]
    const uint32_t b_o_done = b_p_full + 16;               // [2]
    const uint32_t b_o_free = b_o_done + 16;               // [2]
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + C::kOffMisc);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + C::kOffMisc + 4);
    const WaitCtx wctx{abort_flag, p.status};

    // the next kernel may start its set-up; it waits for this grid before touching memory
    ptx::griddep_launch_dependents();
    if (warp == 8) {
        if (lane == 0) {
            ptx::mbar_init(b_q_full, 1);
            ptx::mbar_init(b_q_empty, 1);
            for (int s = 0; s < C::kStages; ++s) {
                ptx::mbar_init(b_k_full + 8 * s, 1);
                ptx::mbar_init(b_k_empty + 8 * s, 1);
                ptx::mbar_init(b_v_full + 8 * s, 1);
                ptx::mbar_init(b_v_empty + 8 * s, 1);
            }
            for (int t = 0; t < 2; ++t) {
                ptx::mbar_init(b_s_full + 8 * t, 1);
                ptx::mbar_init(b_p_full + 8 * t, 128);
                ptx::mbar_init(b_o_done + 8 * t, 1);
                ptx::mbar_init(b_o_free + 8 * t, 128);
            }
            *abort_flag = 0;
            ptx::fence_barrier_init();
            ptx::fence_proxy_async_smem();
            ptx::prefetch_tensormap(&tm_q);
            ptx::prefetch_tensormap(&tm_k);
            ptx::prefetch_tensormap(&tm_v);
        }
        __syncwarp();
    }
    if (warp == 9) {
        ptx::tmem_alloc(ptx::smem_addr(tmem_slot), C::kTmemCols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 8) {
        // =================================================== producer (TMA)
        ptx::griddep_wait();  // page table, pool and Q were written by earlier kernels
        const int ppt = kBN / p.ps;                 // pages per key tile
        const int n_ops = ppt * C::kRegions;        // TMA boxes per K (or V) tile, <= 32
        const int op_page = lane / C::kRegions;     // this lane's box: page index and half
        const int op_reg = lane % C::kRegions;
        const bool op_on = lane < n_ops;
        const uint32_t op_off = op_reg * C::kRegionBytes + op_page * p.ps * 128;
        int gk = 0;        // key tiles issued so far (K / V ring position)
        int q_issued = 0;  // Q loads issued so far
        bool ok = true;
        Piece pc;
        UnitGeo U;
        for (int k = 0; ok && piece_of(P, cw, k, pc, U); ++k) {
            const AttnSeq &sq = p.seqs[U.si];
            const bool two = 2 * U.pair + 1 < sq.n_qtiles;
            auto page_of = [&](int kt) -> int {  // this lane's page id of key tile kt (or -1)
                const int lp = kt * ppt + lane;
                return (lane < ppt && lp < sq.n_pages) ? p.page_table[sq.table_row + lp] : -1;
            };
            int page_next = page_of(pc.lo);  // read while the previous piece's last S GEMMs run
            // Q of this piece once the previous piece's S GEMMs have read theirs
            if (q_issued > 0 && !wait_bar_warp(b_q_empty, (q_issued - 1) & 1, wctx)) { ok = false; break; }
            if (lane == 0) {
                const int nq = two ? 2 : 1;
                ptx::mbar_arrive_expect_tx(b_q_full, nq * C::kTileBytes);
                for (int t = 0; t < nq; ++t)
                    for (int r = 0; r < C::kRegions; ++r)
                        ptx::tma_load_3d(q_smem + t * C::kTileBytes + r * C::kRegionBytes, &tm_q, r * 64,
                                         U.kvh * g, sq.q_row0 + (2 * U.pair + t) * (kBM / g), b_q_full);
            }
            __syncwarp();
            ++q_issued;
            for (int kt = pc.lo; kt < pc.hi; ++kt, ++gk) {
                const int page = page_next;
                if (kt + 1 < pc.hi) page_next = page_of(kt + 1);
                const int s = gk % C::kStages;
                const int pg = __shfl_sync(0xffffffffu, page, op_page & 31);
                // rows of pages past the sequence read as zeros (out-of-bounds box)
                const int y = pg >= 0 ? ((p.layer * p.num_pages + pg) * p.hkv + U.kvh) * p.ps : p.oob_row;
                if (gk >= C::kStages && !wait_bar_warp(b_k_empty + 8 * s, ((gk / C::kStages) - 1) & 1, wctx)) {
                    ok = false;
                    break;
                }
                if (lane == 0) ptx::mbar_arrive_expect_tx(b_k_full + 8 * s, C::kTileBytes);
                __syncwarp();
                if (op_on)
                    ptx::tma_load_2d(k_smem0 + s * C::kTileBytes + op_off, &tm_k, op_reg * 64, y, b_k_full + 8 * s);
                if (gk >= C::kStages && !wait_bar_warp(b_v_empty + 8 * s, ((gk / C::kStages) - 1) & 1, wctx)) {
                    ok = false;
                    break;
                }
                if (lane == 0) ptx::mbar_arrive_expect_tx(b_v_full + 8 * s, C::kTileBytes);
                __syncwarp();
                if (op_on)
                    ptx::tma_load_2d(v_smem0 + s * C::kTileBytes + op_off, &tm_v, op_reg * 64, y, b_v_full + 8 * s);
            }
        }
        __syncwarp();
        if (!ok && lane == 0) {
            // give copies in flight a bounded chance to land before the CTA exits
            const uint64_t t0 = ptx::globaltimer();
            if (q_issued > 0)
                while (!ptx::mbar_try_wait(b_q_full, (q_issued - 1) & 1) && ptx::globaltimer() - t0 < 2000000ull) {}
            for (int i = max(0, gk - C::kStages); i <= gk && i >= 0; ++i) {
                const int s = i % C::kStages;
                while (!ptx::mbar_try_wait(b_k_full + 8 * s, (i / C::kStages) & 1) &&
                       ptx::globaltimer() - t0 < 4000000ull) {}
                while (!ptx::mbar_try_wait(b_v_full + 8 * s, (i / C::kStages) & 1) &&
                       ptx::globaltimer() - t0 < 6000000ull) {}
            }
        }
    } else if (warp == 9) {
        // =================================================== MMA issuer
        if (lane == 0) {
            constexpr uint32_t kIdescQK = ptx::idesc_bf16_f32(kBM, kBN, false);
            constexpr uint32_t kIdescPV = ptx::idesc_bf16_f32(kBM, HD, true);
            auto issue_s = [&](int t, int s) {
                const uint32_t qa = q_smem + t * C::kTileBytes;
                const uint32_t kb = k_smem0 + s * C::kTileBytes;
#pragma unroll
                for (int kk = 0; kk < HD / 16; ++kk) {
                    const uint32_t off = (kk >> 2) * C::kRegionBytes + (kk & 3) * 32;
                    ptx::mma_bf16(tmem + 128 * t, ptx::smem_desc_sw128(qa + off, 16, 1024),
                                  ptx::smem_desc_sw128(kb + off, 16, 1024), kIdescQK, kk > 0 ? 1u : 0u);
                }
                ptx::mma_commit(b_s_full + 8 * t);
            };
            auto issue_pv = [&](int t, int s, bool acc) {
                const uint32_t vb = v_smem0 + s * C::kTileBytes;
#pragma unroll
                for (int kk = 0; kk < kBN / 16; ++kk)
                    mma_bf16_ts(tmem + 256 + HD * t, tmem + 128 * t + kk * 8,
                                ptx::smem_desc_sw128(vb + kk * 16 * 128, C::kRegionBytes, 1024), kIdescPV,
                                (acc || kk > 0) ? 1u : 0u);
                ptx::mma_commit(b_o_done + 8 * t);
            };
            int gk = 0;              // key tiles consumed so far (ring position)
            int cnt0 = 0, cnt1 = 0;  // tiles of q-tile 0 / 1 in earlier pieces (S, P, O phases)
            int seg0 = 0, seg1 = 0;  // earlier pieces in which q-tile 0 / 1 had tiles (o_free phase)
            bool ok = true;
            Piece pc;
            UnitGeo U;
            for (int k = 0; ok && piece_of(P, cw, k, pc, U); ++k) {
                const AttnSeq &sq = p.seqs[U.si];
                const int n0 = q_geo(p, sq, U.pair, 0, pc.lo, pc.hi).ntiles;
                const int n1 = q_geo(p, sq, U.pair, 1, pc.lo, pc.hi).ntiles;
                const int n_all = pc.hi - pc.lo;
                if (!wait_bar(b_q_full, k & 1, wctx) || !wait_bar(b_k_full + 8 * (gk % C::kStages),
                                                                 (gk / C::kStages) & 1, wctx)) {
                    ok = false;
                    break;
                }
                ptx::tc_fence_after();
                const int n_s = max(n0, n1);  // key tiles with S GEMMs; Q is free after the last one
                if (n0 > 0) issue_s(0, gk % C::kStages);
                if (n1 > 0) issue_s(1, gk % C::kStages);
                ptx::mma_commit(b_k_empty + 8 * (gk % C::kStages));
                if (n_s <= 1) ptx::mma_commit(b_q_empty);
                for (int j = 0; j < n_all; ++j) {
                    const int gj = gk + j;
                    const int s = gj % C::kStages;
                    const int s1 = (gj + 1) % C::kStages;
                    const bool more = j + 1 < n_all;
                    if (!wait_bar(b_v_full + 8 * s, (gj / C::kStages) & 1, wctx)) { ok = false; break; }
                    if (j < n0) {
                        // the first P V GEMM of a piece overwrites O_0: the previous piece's epilogue read it
                        if (j == 0 && seg0 > 0 && !wait_bar(b_o_free, (seg0 - 1) & 1, wctx)) { ok = false; break; }
                        if (!wait_bar(b_p_full, (cnt0 + j) & 1, wctx)) { ok = false; break; }
                        ptx::tc_fence_after();
                        issue_pv(0, s, j > 0);
                    }
                    if (more && !wait_bar(b_k_full + 8 * s1, ((gj + 1) / C::kStages) & 1, wctx)) { ok = false; break; }
                    ptx::tc_fence_after();
                    if (j + 1 < n0) issue_s(0, s1);
                    if (j < n1) {
                        if (j == 0 && seg1 > 0 && !wait_bar(b_o_free + 8, (seg1 - 1) & 1, wctx)) { ok = false; break; }
                        if (!wait_bar(b_p_full + 8, (cnt1 + j) & 1, wctx)) { ok = false; break; }
                        ptx::tc_fence_after();
                        issue_pv(1, s, j > 0);
                    }
                    if (j + 1 < n1) issue_s(1, s1);
                    if (j + 2 == n_s) ptx::mma_commit(b_q_empty);    // the piece's last S GEMMs read Q
                    if (more) ptx::mma_commit(b_k_empty + 8 * s1);  // K of tile j+1 consumed by its S GEMMs
                    ptx::mma_commit(b_v_empty + 8 * s);              // V of tile j consumed by its P V GEMMs
                }
                gk += n_all;
                cnt0 += n0;
                cnt1 += n1;
                seg0 += n0 > 0 ? 1 : 0;
                seg1 += n1 > 0 ? 1 : 0;
            }
        }
        __syncwarp();
    } else {
        // =================================================== softmax / epilogue (warps 0-7)
        ptx::griddep_wait();                     // before this role's first global write
        const int t = warp >> 2;                 // q-tile of this warpgroup
        const int row = threadIdx.x & 127;       // TMEM lane
        const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
        const uint32_t tS = tmem + 128 * t + lane_off;
        const uint32_t tO = tmem + 256 + HD * t + lane_off;
        const uint32_t b_s = b_s_full + 8 * t, b_p = b_p_full + 8 * t, b_o = b_o_done + 8 * t;
        const uint32_t b_f = b_o_free + 8 * t;
        const float sl2 = p.scale_log2;
        const float2 sl2x2 = make_float2(sl2, sl2);
        int cnt = 0;  // tiles of this q-tile in earlier pieces (S, P, O phases)
        bool ok = true;
        Piece pc;
        UnitGeo U;
        for (int k = 0; ok && piece_of(P, cw, k, pc, U); ++k) {
            const AttnSeq &sq = p.seqs[U.si];
            const QGeo G = q_geo(p, sq, U.pair, t, pc.lo, pc.hi);
            const int qi = G.q_first + row / g;
            const bool valid = G.qt >= 0 && qi <= G.q_last;
            const int pos = sq.n_keys - sq.n_q + qi;
            float m_ref = -INFINITY;
            float l = 0.f;
            for (int j = 0; j < G.ntiles; ++j) {
                const int kbase = (pc.lo + j) * kBN;
                if (!wait_bar_warp(b_s, (cnt + j) & 1, wctx)) { ok = false; break; }
                ptx::tc_fence_after();
                float s[kBN];
                {
                    float (&s0)[32] = *reinterpret_cast<float (*)[32]>(&s[0]);
                    float (&s1)[32] = *reinterpret_cast<float (*)[32]>(&s[32]);
                    float (&s2)[32] = *reinterpret_cast<float (*)[32]>(&s[64]);
                    float (&s3)[32] = *reinterpret_cast<float (*)[32]>(&s[96]);
                    ptx::tmem_ld32(tS + 0, s0);
                    ptx::tmem_ld32(tS + 32, s1);
                    ptx::tmem_ld32(tS + 64, s2);
                    ptx::tmem_ld32(tS + 96, s3);
                    ptx::tmem_wait_ld();
                }
                if (kbase + kBN - 1 > G.pos_first) {  // tile crosses the causal diagonal of some row
#pragma unroll
                    for (int c = 0; c < kBN; ++c)
                        if (kbase + c > pos) s[c] = -INFINITY;
                }
                // Exponentials against the row's reference m_ref (see replay_attn_kernel): the
                // exact tile max only on the piece's first tile, or when the tile sum passes 2^64.
                auto exp_tile = [&](float ref) -> float {
                    const float2 nref = make_float2(-ref, -ref);
                    float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                                     make_float2(0.f, 0.f)};
#pragma unroll
                    for (int ch = 0; ch < kBN / 32; ++ch) {
                        uint32_t pk[16];
#pragma unroll
                        for (int q = 0; q < 16; ++q) {
                            const int c = ch * 32 + 2 * q;
                            const float2 x = fma2(make_float2(s[c], s[c + 1]), sl2x2, nref);
                            const float2 e = make_float2(ex2(x.x), ex2(x.y));
                            acc[q & 3] = add2(acc[q & 3], e);
                            pk[q] = pack_bf16(e.x, e.y);
                        }
                        tmem_st16(tS + ch * 16, pk);
                    }
                    const float2 a = add2(add2(acc[0], acc[1]), add2(acc[2], acc[3]));
                    return a.x + a.y;
                };
                float rs = 0.f;
                bool need = j == 0;
                if (j > 0) {
                    rs = exp_tile(m_ref);
                    need = !(rs <= kTileSumLimit);
                }
                if (__any_sync(0xffffffffu, need)) {
                    float mx[8];
#pragma unroll
                    for (int q = 0; q < 8; ++q) mx[q] = fmaxf(s[q], s[8 + q]);
#pragma unroll
                    for (int c = 16; c < kBN; c += 16)
#pragma unroll
                        for (int q = 0; q < 8; ++q) mx[q] = max3(mx[q], s[c + q], s[c + 8 + q]);
                    const float mt =
                        fmaxf(max3(mx[0], mx[1], mx[2]), max3(max3(mx[3], mx[4], mx[5]), mx[6], mx[7]));
                    const float m_new = fmaxf(m_ref, mt * sl2);
                    if (j == 0) {
                        m_ref = (m_new == -INFINITY) ? 0.f : m_new;
                    } else {
                        // O holds P V of this piece's tiles < j once P V(j-1) completed
                        if (!wait_bar_warp(b_o, (cnt + j - 1) & 1, wctx)) { ok = false; break; }
                        ptx::tc_fence_after();
                        const float alpha = need ? ex2(m_ref - m_new) : 1.0f;
#pragma unroll 1
                        for (int ch = 0; ch < HD / 16; ++ch) {
                            uint32_t o[16];
                            tmem_ld16(tO + ch * 16, o);
                            ptx::tmem_wait_ld();
#pragma unroll
                            for (int q = 0; q < 16; ++q) o[q] = __float_as_uint(__uint_as_float(o[q]) * alpha);
                            tmem_st16(tO + ch * 16, o);
                        }
                        if (need) {
                            l *= alpha;
                            m_ref = m_new;
                        }
                    }
                    ptx::tmem_wait_st();
                    rs = exp_tile(m_ref);
                }
                l += rs;
                ptx::tmem_wait_st();
                ptx::tc_fence_before();
                ptx::mbar_arrive(b_p);
            }
            if (!ok) break;
            if (pc.slot >= P.n_slots || pc.part >= P.max_parts) {  // a plan outside the workspace: never write
                atomicCAS(p.status, 0, kStatusBadPlan);
                pc.slot = -2;
            }
            const int head = U.kvh * g + (row % g);
            const int64_t prow = pc.slot >= 0
                ? (static_cast<int64_t>(pc.slot) * P.max_parts + pc.part) * (2 * kBM) + t * kBM + row
                : 0;
            uint4 *out_row = reinterpret_cast<uint4 *>(reinterpret_cast<__nv_bfloat16 *>(p.out) +
                                                       (static_cast<int64_t>(sq.q_row0 + qi) * p.hq + head) * HD);
            // A part of a cut unit: per warp of 32 rows a ticket counts the parts written.  When
            // every other part is in already, this warp merges them with its own part straight
            // from TMEM; else it writes its part and counts it.
            int *ticket = P.tickets + (max(pc.slot, 0) * 2 + t) * 4 + (warp & 3);
            const int n_parts = pc.slot >= 0 ? P.slots[pc.slot].n_parts : 0;
            int seen = 0;
            if (pc.slot >= 0 && lane == 0) seen = *reinterpret_cast<volatile int *>(ticket);
            const bool last = pc.slot >= 0 && n_parts <= kMaxOwnMergeParts &&
                              __shfl_sync(0xffffffffu, seen, 0) == n_parts - 1;
            if (last) __threadfence();  // the other parts' rows, written before their tickets
            if (last && lane == 0) {
                // the other parts were written long before (often back in DRAM by now): start bringing
                // this warp's 32-row blocks of them into L2 while the last P V GEMM completes
                for (int q = 0; q < n_parts; ++q) {
                    if (q == pc.part) continue;
                    const int64_t rq = (static_cast<int64_t>(pc.slot) * P.max_parts + q) * (2 * kBM) + t * kBM +
                                       (warp & 3) * 32;
                    ptx::prefetch_l2_bulk(p.part_o + rq * HD, 32 * HD * 4);
                    ptx::prefetch_l2_bulk(p.part_lse + rq, 32 * 4);
                }
            }
            if (G.ntiles > 0) {
                // ---- epilogue: O / l, bf16 output or fp32 partial
                if (!wait_bar_warp(b_o, (cnt + G.ntiles - 1) & 1, wctx)) { ok = false; break; }
                ptx::tc_fence_after();
                const float inv = l > 0.f ? 1.0f / l : 0.f;
                if (pc.slot == -1) {
                    __nv_bfloat16 *dst = reinterpret_cast<__nv_bfloat16 *>(p.out) +
                                         (static_cast<int64_t>(sq.q_row0 + qi) * p.hq + head) * HD;
#pragma unroll
                    for (int ch = 0; ch < HD / 32; ++ch) {
                        float o[32];
                        ptx::tmem_ld32(tO + ch * 32, o);
                        ptx::tmem_wait_ld();
                        if (valid) {
                            uint4 *d4 = reinterpret_cast<uint4 *>(dst + ch * 32);
#pragma unroll
                            for (int q = 0; q < 4; ++q)
                                d4[q] = make_uint4(pack_bf16(o[8 * q + 0] * inv, o[8 * q + 1] * inv),
                                                   pack_bf16(o[8 * q + 2] * inv, o[8 * q + 3] * inv),
                                                   pack_bf16(o[8 * q + 4] * inv, o[8 * q + 5] * inv),
                                                   pack_bf16(o[8 * q + 6] * inv, o[8 * q + 7] * inv));
                        }
                    }
                } else if (last) {
                    merge_own_row<HD, true>(P, pc.slot, t, row, n_parts, pc.part, true, tO, l, m_ref, valid,
                                            out_row);
                } else if (pc.slot >= 0) {
#pragma unroll
                    for (int ch = 0; ch < HD / 32; ++ch) {
                        float o[32];
                        ptx::tmem_ld32(tO + ch * 32, o);
                        ptx::tmem_wait_ld();
                        if (valid && l > 0.f) {
#pragma unroll
                            for (int q = 0; q < 8; ++q)
                                *part_chunk<HD>(p.part_o, prow, ch * 8 + q) =
                                    make_float4(o[4 * q] * inv, o[4 * q + 1] * inv, o[4 * q + 2] * inv,
                                                o[4 * q + 3] * inv);
                        }
                    }
                    if (valid) p.part_lse[prow] = l > 0.f ? m_ref + __log2f(l) : -INFINITY;
                }
                // O_t has been read: the next piece's first P V GEMM may overwrite it
                ptx::tc_fence_before();
                ptx::mbar_arrive(b_f);
            } else if (last) {
                merge_own_row<HD, true>(P, pc.slot, t, row, n_parts, pc.part, false, tO, 0.f, 0.f, valid, out_row);
            } else if (pc.slot >= 0 && valid) {
                p.part_lse[prow] = -INFINITY;  // no key of this piece is visible to these rows
            }
            if (last) {
                if (lane == 0) *ticket = 0;  // zero again for the next launch
            } else if (pc.slot >= 0) {
                // this warp's 32 rows of the part are written: count them; the warp that brings
                // the count to the part count (another part finished meanwhile) merges from L2
                __threadfence();
                __syncwarp();
                int arrived = 0;
                if (lane == 0) arrived = atomicAdd(ticket, 1);
                if (__shfl_sync(0xffffffffu, arrived, 0) == n_parts - 1) {
                    __threadfence();
                    if (n_parts <= kMaxOwnMergeParts)
                        merge_own_row<HD, false>(P, pc.slot, t, row, n_parts, -1, false, tO, 0.f, 0.f, valid,
                                                 out_row);
                    else if (valid)
                        merge_parts_row<HD>(P, pc.slot, t, row, n_parts, out_row);
                    if (lane == 0) *ticket = 0;
                }
            }
            cnt += G.ntiles;
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, C::kTmemCols);
    }
}

template <int HD>
cudaError_t launch_sk_t(const CUtensorMap &q, const CUtensorMap &k, const CUtensorMap &v, const SkParams &p,
                        cudaStream_t st)
{
    using C = SkCfg<HD>;
    static std::atomic<uint64_t> configured{0};
    cudaError_t e = set_dyn_smem_once(replay_attn_sk_kernel<HD>, C::kDynSmem, configured);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(p.n_ctas));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = C::kDynSmem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, replay_attn_sk_kernel<HD>, q, k, v, p);
}

}  // namespace

cudaError_t launch_replay_attn_sk(int head_dim, const CUtensorMap &tm_q, const CUtensorMap &tm_k,
                                  const CUtensorMap &tm_v, const SkParams &p, cudaStream_t st)
{
    if (p.n_ctas <= 0) return cudaSuccess;
    if (p.n_ctas > kMaxSkCtas) return cudaErrorInvalidValue;
    if (head_dim == 128) return launch_sk_t<128>(tm_q, tm_k, tm_v, p, st);
    if (head_dim == 64) return launch_sk_t<64>(tm_q, tm_k, tm_v, p, st);
    return cudaErrorInvalidValue;
}

}  // namespace pe

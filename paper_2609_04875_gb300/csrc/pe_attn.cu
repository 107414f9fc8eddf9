// Replay attention over a paged KV cache on sm_103a (tcgen05 + TMEM + TMA).
//
// What it computes (Alg. 1 replay loop; the sanitized suffix is re-prefilled
// on the cropped cache, Sec. 3.2 / Sec. 4.5): for the last n_q positions of a
// sequence, query i at position len-n_q+i and q-head h attend the keys
// 0..len-n_q+i of kv-head h / (Hq/Hkv):
//     O = softmax(scale * q K^T) V      (bf16 in, fp32 accumulate, bf16 out)
//
// One CTA computes one work item: (sequence, kv-head, pair of q-tiles[, key
// split]).  A q-tile packs 128 rows = (128/g queries) x (g q-heads of one
// kv-head), so each K/V tile brought into shared memory serves 2 x 128 rows.
// Roles (320 threads):
//   warps 0-3, 4-7  softmax of q-tile 0 / q-tile 1: thread r owns row r
//                   (TMEM lane r); masks, online softmax in fp32 (exp2),
//                   writes P (bf16) back into TMEM (d = 128: over its S
//                   columns; d = 64: into its own P columns), rescales O in
//                   TMEM when needed, epilogue (a full q-tile's O goes to
//                   shared memory, then out by one TMA store per 64 columns).
//   warp 8          producer: reads the page table; its lanes issue one TMA
//                   box per (page, 64-column half) into K and V stage rings.
//   warp 9          MMA: allocates TMEM; one thread issues tcgen05.mma for
//                   S_t = Q_t K^T (A, B from shared memory) and
//                   O_t += P_t V (A = P from TMEM, B = V from shared memory).
// Tensor-core order per key tile j (d = 128):  PV_0(j), S_0(j+1), PV_1(j),
// S_1(j+1), so one softmax group works while the tensor core runs the other
// group's GEMMs; S_t(j+1) waits for PV_t(j), which reads P_t(j) over S_t.
// TMEM columns: S_0 [0,128), S_1 [128,256), O_0 and O_1 (HD each) from 256.
// At d = 64 the last 128 columns hold P_0 and P_1, so S_t(j+1) is issued as
// soon as the softmax has copied S_t(j) into registers (barrier s_free) and
// runs during the softmax of tile j; the softmax writes P_t(j) once
// PV_t(j-1) has read P_t(j-1).  Same arithmetic, so the same bits.
//
// Key tiles always start at logical key 0 (multiples of 128 keys), whatever
// the physical pages, so a row's arithmetic depends only on its own keys.
//
// Online softmax with a lazily moved reference: a row's reference m_ref is the
// first tile's max (log2 units) and only moves when a later tile's weights
// exp2(x - m_ref) sum beyond 2^64 (a logit more than ~64 above m_ref, or
// inf/NaN); then the tile max is taken, O and l are rescaled in place and the
// tile's weights recomputed.  Any fixed reference gives the same O / l, and
// weights up to 2^64 stay far inside fp32/bf16 range, so the tile max is
// skipped on all other tiles.  Rows decide independently.
//
// Every wait is bounded (kWaitNs); on expiry the CTA records a status code,
// all roles leave their loops, and TMEM is freed before exit.
#include <cuda_bf16.h>

#include <mutex>

#include "dev_common.cuh"
#include "pe_internal.h"
#include "ptx.cuh"

namespace pe {

constexpr float kTileSumLimit = 1.8446744e19f;  // 2^64: larger tile sums move the reference
constexpr int kThreads = 320;

template <int HD>
struct AttnCfg {
    static constexpr int kRegions = HD / 64;            // 128-byte swizzle atoms along d
    static constexpr int kTileBytes = kBM * HD * 2;     // one Q, K or V tile (128 rows)
    static constexpr int kRegionBytes = kBM * 128;      // 128 rows x 128 bytes
    static constexpr int kStages = (HD == 128) ? 2 : 3; // K ring and V ring depth
    static constexpr int kOffQ = 0;                     // Q_0, Q_1
    static constexpr int kOffK = kOffQ + 2 * kTileBytes;
    static constexpr int kOffV = kOffK + kStages * kTileBytes;
    static constexpr int kOffBar = kOffV + kStages * kTileBytes;
    // barriers: q_full, k_full[S], k_empty[S], v_full[S], v_empty[S], s_full[2], p_full[2], o_done[2],
    // s_free[2], o_staged[2]
    static constexpr int kNumBars = 1 + 4 * kStages + 10;
    // TMEM columns: S_0, S_1 (128 each), O_0, O_1 (HD each); for d = 64 the 128 left over hold P_0 and
    // P_1 (64 each), so S(j+1) need not wait for the P V GEMM of tile j (P(j) lives apart from S)
    static constexpr bool kSepP = HD == 64;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;  // tmem slot, abort flag
    static constexpr int kSmemBytes = kOffMisc + 16;
    static constexpr int kDynSmem = kSmemBytes + 1024;       // alignment slack
    static constexpr uint32_t kTmemCols = 512;
    static_assert(kDynSmem <= 232448, "shared memory budget");
};

// Per q-tile geometry of a work item.
struct TileGeo {
    int qt;          // q-tile index within the sequence (-1: absent)
    int q_first;     // first query of the tile
    int q_last;      // last valid query of the tile
    int pos_first;   // absolute position of the first query
    int ntiles;      // key tiles this q-tile processes (from kt0)
};

template <int HD, bool SPLIT>
__global__ void __launch_bounds__(kThreads, 1)
    replay_attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                       const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_o,
                       const __grid_constant__ AttnParams p)
{
    using C = AttnCfg<HD>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = ptx::smem_addr(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;
    uint8_t *smem = smem_raw + (sbase - raw);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    // ---- work item -> (sequence, kv-head, split, q-tile pair); heaviest pairs first.  Within a
    // sequence the kv-heads run fastest (every head's heaviest pairs first), or, when p.pairs_fastest
    // is set (launches of many waves), the pairs: then the CTAs resident at once work on one or two
    // kv-heads' keys, which stay in L2 while Q and O stream through.
    auto decode_item = [&](int item, int &si, int &kvh, int &split, int &pair) {
        si = 0;
        int si_hi = p.n_seqs;  // the last sequence whose first item is at most `item` (binary search)
        while (si_hi - si > 1) {
            const int mid = (si + si_hi) >> 1;
            if (p.seqs[mid].item0 <= item) si = mid;
            else si_hi = mid;
        }
        const AttnSeq &q = p.seqs[si];
        int local = item - q.item0;
        if (p.pairs_fastest) {
            const int seq_items = (si + 1 < p.n_seqs ? p.seqs[si + 1].item0 : p.total_items) - q.item0;
            const int n_pairs = seq_items / (p.hkv * q.n_splits);  // pairs of this sequence in the launch
            pair = q.pair_top - 1 - local % n_pairs;
            local /= n_pairs;
            split = local % q.n_splits;
            kvh = local / q.n_splits;
        } else {
            kvh = local % p.hkv;
            local /= p.hkv;
            split = local % q.n_splits;
            pair = q.pair_top - 1 - local / q.n_splits;
        }
    };
    int si, kvh, split, pair;
    decode_item(blockIdx.x, si, kvh, split, pair);
    const AttnSeq &sq = p.seqs[si];
    const int g = p.group;
    const int bmq = kBM / g;
    const int kt0 = SPLIT ? split * p.split_tiles : 0;
    TileGeo geo[2];
#pragma unroll
    for (int t = 0; t < 2; ++t) {
        const int qt = 2 * pair + t;
        TileGeo &G = geo[t];
        if (qt < sq.n_qtiles) {
            G.qt = qt;
            G.q_first = qt * bmq;
            G.q_last = min(G.q_first + bmq, sq.n_q) - 1;
            G.pos_first = sq.n_keys - sq.n_q + G.q_first;
            const int k_end = sq.n_keys - sq.n_q + G.q_last + 1;
            const int nkt = (k_end + kBN - 1) / kBN;
            const int kt1 = SPLIT ? min(nkt, kt0 + p.split_tiles) : nkt;
            G.ntiles = max(0, kt1 - kt0);
        } else {
            G.qt = -1;
            G.q_first = G.q_last = G.pos_first = 0;
            G.ntiles = 0;
        }
    }
    const int n_all = max(geo[0].ntiles, geo[1].ntiles);  // key tiles loaded for the pair

    // ---- shared memory carve-up
    const uint32_t q_smem = sbase + C::kOffQ;
    const uint32_t k_smem0 = sbase + C::kOffK;
    const uint32_t v_smem0 = sbase + C::kOffV;
    const uint32_t bar0 = sbase + C::kOffBar;
    const uint32_t b_q_full = bar0;
    const uint32_t b_k_full = bar0 + 8;
    const uint32_t b_k_empty = b_k_full + 8 * C::kStages;
    const uint32_t b_v_full = b_k_empty + 8 * C::kStages;
    const uint32_t b_v_empty = b_v_full + 8 * C::kStages;
    const uint32_t b_s_full = b_v_empty + 8 * C::kStages;  // [2]
    const uint32_t b_p_full = b_s_full + 16;               // [2]
    const uint32_t b_o_done = b_p_full + 16;               // [2]
    const uint32_t b_s_free = b_o_done + 16;               // [2] (d = 64) S_t has been read into registers
    const uint32_t b_o_staged = b_s_free + 16;             // [2] O_t (bf16) is in Q_t's shared memory
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + C::kOffMisc);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + C::kOffMisc + 4);
    const WaitCtx wctx{abort_flag, p.status};

    // The producer warp initialises the barriers and starts the Q loads and the
    // first key tile's loads before the CTA-wide sync, while the MMA warp
    // allocates TMEM; no other thread touches a barrier before the sync.
    const int ppt = kBN / p.ps;                 // pages per key tile
    const int n_ops = ppt * C::kRegions;        // TMA boxes per K (or V) tile, <= 32
    const int op_page = lane / C::kRegions;     // this lane's box: page index and half
    const int op_reg = lane % C::kRegions;
    const bool op_on = lane < n_ops;
    const uint32_t op_off = op_reg * C::kRegionBytes + op_page * p.ps * 128;
    auto page_of = [&](int i) -> int {          // this lane's page id of key tile i (or -1)
        const int lp = (kt0 + i) * ppt + lane;
        return (lane < ppt && lp < sq.n_pages) ? p.page_table[sq.table_row + lp] : -1;
    };
    auto issue_kv = [&](int i, int page) {      // all lanes: TMA boxes of key tile i into stage i % S
        const int s = i % C::kStages;
        const int pg = __shfl_sync(0xffffffffu, page, op_page & 31);
        // rows of pages past the sequence read as zeros (out-of-bounds box)
        const int y = pg >= 0 ? ((p.layer * p.num_pages + pg) * p.hkv + kvh) * p.ps : p.oob_row;
        if (i >= C::kStages && !wait_bar_warp(b_k_empty + 8 * s, ((i / C::kStages) - 1) & 1, wctx)) return false;
        if (lane == 0) ptx::mbar_arrive_expect_tx(b_k_full + 8 * s, C::kTileBytes);
        __syncwarp();
        if (op_on) ptx::tma_load_2d(k_smem0 + s * C::kTileBytes + op_off, &tm_k, op_reg * 64, y, b_k_full + 8 * s);
        if (i >= C::kStages && !wait_bar_warp(b_v_empty + 8 * s, ((i / C::kStages) - 1) & 1, wctx)) return false;
        if (lane == 0) ptx::mbar_arrive_expect_tx(b_v_full + 8 * s, C::kTileBytes);
        __syncwarp();
        if (op_on) ptx::tma_load_2d(v_smem0 + s * C::kTileBytes + op_off, &tm_v, op_reg * 64, y, b_v_full + 8 * s);
        return true;
    };
    // Launched with programmatic serialization: the next kernel in the stream may
    // start its set-up once every CTA of this grid has started (it waits for this
    // grid's completion before touching memory), and this grid's set-up overlaps
    // the previous kernel; griddepcontrol.wait comes before the first read of
    // memory an earlier kernel wrote (page table, pool, Q) and before any write.
    ptx::griddep_launch_dependents();
    int page_next = -1;
    if (warp == 8) {
        if (lane == 0) {
            ptx::mbar_init(b_q_full, 1);
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
                ptx::mbar_init(b_s_free + 8 * t, 128);
                ptx::mbar_init(b_o_staged + 8 * t, 128);
            }
            *abort_flag = 0;
            ptx::fence_barrier_init();
            ptx::fence_proxy_async_smem();
            ptx::prefetch_tensormap(&tm_q);
            ptx::prefetch_tensormap(&tm_k);
            ptx::prefetch_tensormap(&tm_v);
            if (!SPLIT) ptx::prefetch_tensormap(&tm_o);
        }
        ptx::griddep_wait();
        if (n_all > 0) page_next = page_of(0);
        if (lane == 0) {
            if (n_all > 0) {
                const int nq = geo[1].qt >= 0 ? 2 : 1;
                ptx::mbar_arrive_expect_tx(b_q_full, nq * C::kTileBytes);
                for (int t = 0; t < nq; ++t)
                    for (int r = 0; r < C::kRegions; ++r)
                        ptx::tma_load_3d(q_smem + t * C::kTileBytes + r * C::kRegionBytes, &tm_q, r * 64, kvh * g,
                                         sq.q_row0 + (2 * pair + t) * bmq, b_q_full);
            }
        }
        __syncwarp();
        if (n_all > 0) {
            const int page = page_next;
            if (n_all > 1) page_next = page_of(1);
            issue_kv(0, page);  // tile 0 never waits (its stage is fresh)
        }
    }
    if (warp == 9) {
        ptx::tmem_alloc(ptx::smem_addr(tmem_slot), C::kTmemCols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 8 && n_all > 0) {
        // =================================================== producer (TMA), tiles 1..
        for (int i = 1; i < n_all; ++i) {
            const int page = page_next;
            if (i + 1 < n_all) page_next = page_of(i + 1);  // prefetch the next tile's page ids
            if (!issue_kv(i, page)) break;
        }
        // With one CTA per SM, the CTA that starts on this SM next is about blockIdx.x + next_stride:
        // bring its Q tiles (read once, from DRAM) into L2 now, so that its first S GEMMs wait less.
        const int nxt = blockIdx.x + p.next_stride;
        if (p.next_stride > 0 && nxt < p.total_items && lane == 0 && !*abort_flag) {
            int nsi, nkvh, nsplit, npair;
            decode_item(nxt, nsi, nkvh, nsplit, npair);
            const AttnSeq &nq = p.seqs[nsi];
            for (int t = 0; t < 2; ++t) {
                const int qt = 2 * npair + t;
                if (qt >= nq.n_qtiles) break;
                for (int r = 0; r < C::kRegions; ++r)
                    ptx::tma_prefetch_3d(&tm_q, r * 64, nkvh * g, nq.q_row0 + qt * (kBM / g));
            }
        }
        __syncwarp();
        if (*abort_flag && lane == 0) {
            // give copies in flight a bounded chance to land before the CTA exits
            const uint64_t t0 = ptx::globaltimer();
            for (int i = max(0, n_all - C::kStages); i < n_all; ++i) {
                const int s = i % C::kStages;
                while (!ptx::mbar_try_wait(b_k_full + 8 * s, (i / C::kStages) & 1) &&
                       ptx::globaltimer() - t0 < 2000000ull) {}
                while (!ptx::mbar_try_wait(b_v_full + 8 * s, (i / C::kStages) & 1) &&
                       ptx::globaltimer() - t0 < 4000000ull) {}
            }
        }
    } else if (warp == 9 && n_all > 0) {
        // =================================================== MMA issuer
        if (lane == 0) {
            constexpr uint32_t kIdescQK = ptx::idesc_bf16_f32(kBM, kBN, false);
            constexpr uint32_t kIdescPV = ptx::idesc_bf16_f32(kBM, HD, true);
            const int n0 = geo[0].ntiles, n1 = geo[1].ntiles;
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
                const uint32_t tp = C::kSepP ? tmem + 256 + 2 * HD + 64 * t : tmem + 128 * t;  // P_t
#pragma unroll
                for (int kk = 0; kk < kBN / 16; ++kk)
                    mma_bf16_ts(tmem + 256 + HD * t, tp + kk * 8,
                                ptx::smem_desc_sw128(vb + kk * 16 * 128, C::kRegionBytes, 1024), kIdescPV,
                                (acc || kk > 0) ? 1u : 0u);
                ptx::mma_commit(b_o_done + 8 * t);
            };
            bool ok = wait_bar(b_q_full, 0, wctx) && wait_bar(b_k_full, 0, wctx);
            if (ok) {
                ptx::tc_fence_after();
                if (n0 > 0) issue_s(0, 0);
                if (n1 > 0) issue_s(1, 0);
                if (n0 > 0 || n1 > 0) ptx::mma_commit(b_k_empty);
            }
            for (int j = 0; ok && C::kSepP && j < n_all; ++j) {
                // d = 64: S_t(j+1) once the softmax holds S_t(j) in registers, P V_t(j) once P_t(j) is in
                const int s = j % C::kStages;
                const int s1 = (j + 1) % C::kStages;
                const bool more = j + 1 < n_all;
                if (more && !wait_bar(b_k_full + 8 * s1, ((j + 1) / C::kStages) & 1, wctx)) { ok = false; break; }
#pragma unroll
                for (int t = 0; t < 2; ++t) {
                    if (j + 1 >= (t ? n1 : n0)) continue;
                    if (!wait_bar(b_s_free + 8 * t, j & 1, wctx)) { ok = false; break; }
                    ptx::tc_fence_after();
                    issue_s(t, s1);
                }
                if (!ok) break;
                if (more) ptx::mma_commit(b_k_empty + 8 * s1);  // K of tile j+1 consumed by its S GEMMs
                if (!wait_bar(b_v_full + 8 * s, (j / C::kStages) & 1, wctx)) { ok = false; break; }
#pragma unroll
                for (int t = 0; t < 2; ++t) {
                    if (j >= (t ? n1 : n0)) continue;
                    if (!wait_bar(b_p_full + 8 * t, j & 1, wctx)) { ok = false; break; }
                    ptx::tc_fence_after();
                    issue_pv(t, s, j > 0);
                }
                if (!ok) break;
                ptx::mma_commit(b_v_empty + 8 * s);              // V of tile j consumed by its PV GEMMs
            }
            for (int j = 0; ok && !C::kSepP && j < n_all; ++j) {
                const int s = j % C::kStages;
                const int s1 = (j + 1) % C::kStages;
                const bool more = j + 1 < n_all;
                if (!wait_bar(b_v_full + 8 * s, (j / C::kStages) & 1, wctx)) { ok = false; break; }
                if (j < n0) {
                    if (!wait_bar(b_p_full, j & 1, wctx)) { ok = false; break; }
                    ptx::tc_fence_after();
                    issue_pv(0, s, j > 0);
                }
                if (more && !wait_bar(b_k_full + 8 * s1, ((j + 1) / C::kStages) & 1, wctx)) { ok = false; break; }
                ptx::tc_fence_after();
                if (j + 1 < n0) issue_s(0, s1);
                if (j < n1) {
                    if (!wait_bar(b_p_full + 8, j & 1, wctx)) { ok = false; break; }
                    ptx::tc_fence_after();
                    issue_pv(1, s, j > 0);
                }
                if (j + 1 < n1) issue_s(1, s1);
                if (more) ptx::mma_commit(b_k_empty + 8 * s1);  // K of tile j+1 consumed by its S GEMMs
                ptx::mma_commit(b_v_empty + 8 * s);              // V of tile j consumed by its PV GEMMs
            }
        }
        __syncwarp();
    } else if (warp < 8) {
        // =================================================== softmax / epilogue
        ptx::griddep_wait();                     // before this role's first global write
        const int t = warp >> 2;                 // q-tile of this warpgroup
        const TileGeo G = t ? geo[1] : geo[0];   // by value: no run-time index into geo (local memory)
        const int row = threadIdx.x & 127;       // TMEM lane
        const int qi = G.q_first + row / g;
        const bool valid = G.qt >= 0 && qi <= G.q_last;
        const int pos = sq.n_keys - sq.n_q + qi;
        const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
        const uint32_t tS = tmem + 128 * t + lane_off;
        const uint32_t tO = tmem + 256 + HD * t + lane_off;
        const uint32_t b_s = b_s_full + 8 * t, b_p = b_p_full + 8 * t, b_o = b_o_done + 8 * t;
        const uint32_t tP = C::kSepP ? tmem + 256 + 2 * HD + 64 * t + lane_off : tS;  // P_t (over S_t for d = 128)
        const float sl2 = p.scale_log2;
        const float2 sl2x2 = make_float2(sl2, sl2);
        float m_ref = -INFINITY;
        float l = 0.f;
        bool ok = true;
        for (int j = 0; j < G.ntiles; ++j) {
            const int kbase = (kt0 + j) * kBN;
            if (!wait_bar_warp(b_s, j & 1, wctx)) { ok = false; break; }
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
            if (C::kSepP) {
                // S_t(j) is in registers: the next tile's S GEMM may overwrite it
                ptx::tc_fence_before();
                ptx::mbar_arrive(b_s_free + 8 * t);
            }
            if (kbase + kBN - 1 > G.pos_first) {  // tile crosses the causal diagonal of some row
#pragma unroll
                for (int c = 0; c < kBN; ++c)
                    if (kbase + c > pos) s[c] = -INFINITY;
            }
            // Exponentials against the row's current reference m_ref; the exact tile
            // max is needed only on the first tile, or when the tile's sum exceeds
            // 2^64 (some logit above m_ref + ~64, or inf/NaN): then m_ref moves, O
            // and l are rescaled, and the tile is recomputed.
            auto exp_tile = [&](float ref) -> float {
                const float2 nref = make_float2(-ref, -ref);
                float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                                 make_float2(0.f, 0.f)};
#pragma unroll
                for (int ch = 0; ch < kBN / 32; ++ch) {
                    uint32_t pk[16];
#pragma unroll
                    for (int k = 0; k < 16; ++k) {
                        const int c = ch * 32 + 2 * k;
                        const float2 x = fma2(make_float2(s[c], s[c + 1]), sl2x2, nref);
                        const float2 e = make_float2(ex2(x.x), ex2(x.y));
                        acc[k & 3] = add2(acc[k & 3], e);
                        pk[k] = pack_bf16(e.x, e.y);
                    }
                    if (C::kSepP && ch == 0 && j > 0) {
                        // P_t(j) goes to P_t's own columns once P V_t(j-1) has read P_t(j-1)
                        if (!wait_bar_warp(b_o, (j - 1) & 1, wctx)) ok = false;
                        ptx::tc_fence_after();
                    }
                    tmem_st16(tP + ch * 16, pk);
                }
                const float2 a = add2(add2(acc[0], acc[1]), add2(acc[2], acc[3]));
                return a.x + a.y;
            };
            float rs = 0.f;
            bool need = j == 0;
            if (j > 0) {
                rs = exp_tile(m_ref);
                if (!ok) break;
                need = !(rs <= kTileSumLimit);
            }
            if (__any_sync(0xffffffffu, need)) {
                float mx[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) mx[k] = fmaxf(s[k], s[8 + k]);
#pragma unroll
                for (int c = 16; c < kBN; c += 16)
#pragma unroll
                    for (int k = 0; k < 8; ++k) mx[k] = max3(mx[k], s[c + k], s[c + 8 + k]);
                const float mt = fmaxf(max3(mx[0], mx[1], mx[2]), max3(max3(mx[3], mx[4], mx[5]), mx[6], mx[7]));
                const float m_new = fmaxf(m_ref, mt * sl2);
                if (j == 0) {
                    m_ref = (m_new == -INFINITY) ? 0.f : m_new;
                } else {
                    // O holds PV of tiles < j once PV(j-1) completed; PV(j) waits for our P
                    if (!wait_bar_warp(b_o, (j - 1) & 1, wctx)) { ok = false; break; }
                    ptx::tc_fence_after();
                    const float alpha = need ? ex2(m_ref - m_new) : 1.0f;
#pragma unroll 1
                    for (int ch = 0; ch < HD / 16; ++ch) {
                        uint32_t o[16];
                        tmem_ld16(tO + ch * 16, o);
                        ptx::tmem_wait_ld();
#pragma unroll
                        for (int k = 0; k < 16; ++k) o[k] = __float_as_uint(__uint_as_float(o[k]) * alpha);
                        tmem_st16(tO + ch * 16, o);
                    }
                    if (need) {
                        l *= alpha;
                        m_ref = m_new;
                    }
                }
                ptx::tmem_wait_st();
                rs = exp_tile(m_ref);
                if (!ok) break;
            }
            l += rs;
            ptx::tmem_wait_st();
            ptx::tc_fence_before();
            ptx::mbar_arrive(b_p);
        }
        // ---- epilogue: O / l
        if (ok && G.ntiles > 0) {
            ok = wait_bar_warp(b_o, (G.ntiles - 1) & 1, wctx);
            if (ok) {
                ptx::tc_fence_after();
                const float inv = l > 0.f ? 1.0f / l : 0.f;
                const int head = kvh * g + (row % g);
                if (!SPLIT && (G.q_last - G.q_first + 1) * g == kBM) {
                    // a full q-tile: O in bf16 into Q_t's shared memory (its S GEMMs are long done), laid
                    // out as the Q box was loaded (128-byte rows, 16-byte chunks swizzled by row & 7), then
                    // one TMA store per 64-column region; a ragged tile (other sequences' rows follow its
                    // last query) takes the plain stores below
                    const uint32_t qt_smem = q_smem + t * C::kTileBytes;
#pragma unroll
                    for (int ch = 0; ch < HD / 32; ++ch) {
                        float o[32];
                        ptx::tmem_ld32(tO + ch * 32, o);
                        ptx::tmem_wait_ld();
                        const uint32_t rbase = qt_smem + (ch >> 1) * C::kRegionBytes + row * 128;
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const int c = (ch & 1) * 4 + k;  // 16-byte chunk within the 128-byte row
                            const uint32_t a = rbase + ((c ^ (row & 7)) << 4);
                            asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(a),
                                         "r"(pack_bf16(o[8 * k + 0] * inv, o[8 * k + 1] * inv)),
                                         "r"(pack_bf16(o[8 * k + 2] * inv, o[8 * k + 3] * inv)),
                                         "r"(pack_bf16(o[8 * k + 4] * inv, o[8 * k + 5] * inv)),
                                         "r"(pack_bf16(o[8 * k + 6] * inv, o[8 * k + 7] * inv))
                                         : "memory");
                        }
                    }
                    ptx::fence_proxy_async_smem();  // the stores above, seen by the TMA store
                    ptx::mbar_arrive(b_o_staged + 8 * t);
                    if (row == 0) {
                        if (wait_bar(b_o_staged + 8 * t, 0, wctx)) {
#pragma unroll
                            for (int r = 0; r < C::kRegions; ++r)
                                ptx::tma_store_3d(&tm_o, r * 64, kvh * g, sq.q_row0 + G.q_first,
                                                  qt_smem + r * C::kRegionBytes);
                            ptx::bulk_commit_group();
                            ptx::bulk_wait_read_all();  // shared memory stays until the copies have read it
                        }
                    }
                } else if (!SPLIT) {
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
                            for (int k = 0; k < 4; ++k)
                                d4[k] = make_uint4(pack_bf16(o[8 * k + 0] * inv, o[8 * k + 1] * inv),
                                                   pack_bf16(o[8 * k + 2] * inv, o[8 * k + 3] * inv),
                                                   pack_bf16(o[8 * k + 4] * inv, o[8 * k + 5] * inv),
                                                   pack_bf16(o[8 * k + 6] * inv, o[8 * k + 7] * inv));
                        }
                    }
                } else {
                    const int64_t prow = sq.part_row0 +
                                         (static_cast<int64_t>(G.qt * p.hkv + kvh) * sq.n_splits + split) * kBM + row;
#pragma unroll
                    for (int ch = 0; ch < HD / 32; ++ch) {
                        float o[32];
                        ptx::tmem_ld32(tO + ch * 32, o);
                        ptx::tmem_wait_ld();
                        if (valid && l > 0.f) {
#pragma unroll
                            for (int k = 0; k < 8; ++k)
                                *part_chunk<HD>(p.part_o, prow, ch * 8 + k) =
                                    make_float4(o[4 * k] * inv, o[4 * k + 1] * inv, o[4 * k + 2] * inv,
                                                o[4 * k + 3] * inv);
                        }
                    }
                    if (valid) p.part_lse[prow] = l > 0.f ? m_ref + __log2f(l) : -INFINITY;
                }
            }
        }
        if (SPLIT && G.ntiles == 0 && valid) {
            // empty key range: this split contributes nothing to these rows
            const int64_t prow = sq.part_row0 +
                                 (static_cast<int64_t>(G.qt * p.hkv + kvh) * sq.n_splits + split) * kBM + row;
            p.part_lse[prow] = -INFINITY;
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, C::kTmemCols);
    }
}

// Exercises the bounded wait on its own: one thread waits on an mbarrier that
// nothing arrives at; after limit_ns the wait gives up, records the status code
// and the kernel returns normally, leaving the context usable.
__global__ void bounded_wait_selftest_kernel(int32_t *status, uint64_t limit_ns)
{
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x != 0) return;
    const uint32_t b = ptx::smem_addr(&bar);
    ptx::mbar_init(b, 1);
    abort_flag = 0;
    ptx::fence_barrier_init();
    const WaitCtx w{&abort_flag, status};
    (void)wait_bar(b, 0, w, limit_ns);
}

cudaError_t launch_bounded_wait_selftest(int32_t *status, uint64_t limit_ns, cudaStream_t st)
{
    bounded_wait_selftest_kernel<<<1, 32, 0, st>>>(status, limit_ns);
    return cudaGetLastError();
}

// LSE-weighted merge of the split partials: one warp per 32 rows (a row block of the partials) and 32
// columns, lane i on row 32 w + i, so every load of a split's chunk is 512 contiguous bytes.  For each
// row, in split order: w_s = 2^(lse_s - max lse), den += w_s, acc += w_s O_s.
template <int HD>
__global__ void __launch_bounds__(256) splitkv_combine_kernel(const __grid_constant__ AttnParams p)
{
    // launched with programmatic serialization after the attention grid: wait
    // for its partials; the next kernel may start its own set-up meanwhile
    ptx::griddep_launch_dependents();
    ptx::griddep_wait();
    constexpr int kGroups = HD / 32;  // column groups of 32 (8 chunks of 16 bytes)
    const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    const int blk = gw / kGroups, cg = gw % kGroups;
    const int rbase = blk * 32;  // first combine row of this warp's block
    if (rbase >= p.total_comb) return;
    int si = 0;
    while (si + 1 < p.n_seqs && rbase >= p.seqs[si + 1].comb0) ++si;
    const AttnSeq &sq = p.seqs[si];
    const int local = rbase + lane - sq.comb0;
    const int row = local % kBM;
    const int unit = local / kBM;  // qt * hkv + kvh (the same for the whole block)
    const int kvh = unit % p.hkv;
    const int qt = unit / p.hkv;
    const int g = p.group;
    const int qi = qt * (kBM / g) + row / g;
    const int64_t base = sq.part_row0 + static_cast<int64_t>(unit) * sq.n_splits * kBM + row;
    const int ns = sq.n_splits;
    float mx = -INFINITY;
    for (int s = 0; s < ns; ++s) mx = fmaxf(mx, p.part_lse[base + static_cast<int64_t>(s) * kBM]);
    float acc[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) acc[i] = 0.f;
    float den = 0.f;
    if (mx != -INFINITY) {
#pragma unroll 2
        for (int s = 0; s < ns; ++s) {
            const int64_t r = base + static_cast<int64_t>(s) * kBM;
            const float lse = p.part_lse[r];
            if (lse == -INFINITY) continue;
            const float w = ex2(lse - mx);
            den += w;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const float4 v = *part_chunk<HD>(p.part_o, r, cg * 8 + k);
                acc[4 * k + 0] += w * v.x;
                acc[4 * k + 1] += w * v.y;
                acc[4 * k + 2] += w * v.z;
                acc[4 * k + 3] += w * v.w;
            }
        }
    }
    if (qi >= sq.n_q) return;
    const float inv = den > 0.f ? 1.0f / den : 0.f;
    const int head = kvh * g + (row % g);
    uint4 *dst = reinterpret_cast<uint4 *>(reinterpret_cast<__nv_bfloat16 *>(p.out) +
                                           (static_cast<int64_t>(sq.q_row0 + qi) * p.hq + head) * HD + cg * 32);
#pragma unroll
    for (int k = 0; k < 4; ++k)
        dst[k] = make_uint4(pack_bf16(acc[8 * k + 0] * inv, acc[8 * k + 1] * inv),
                            pack_bf16(acc[8 * k + 2] * inv, acc[8 * k + 3] * inv),
                            pack_bf16(acc[8 * k + 4] * inv, acc[8 * k + 5] * inv),
                            pack_bf16(acc[8 * k + 6] * inv, acc[8 * k + 7] * inv));
}

// Split-KV partials of pe_replay_attn_static_scratch: a fixed 16 MiB array that
// every GPU loading the library holds until the process exits.  Host code must
// not pass the symbol itself to a kernel (on the host it names a stand-in, not
// device memory); static_scratch() looks up its device address instead.
static __device__ __align__(256) float g_static_splitkv_scratch[kStaticScratchBytes / sizeof(float)];

cudaError_t static_scratch(float **ptr)
{
    constexpr int kMaxDevices = 64;
    static std::mutex mu;
    static float *addr[kMaxDevices] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[dev]) {  // once per device, with that device current
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_splitkv_scratch);
        if (e != cudaSuccess) return e;
        addr[dev] = static_cast<float *>(p);
    }
    *ptr = addr[dev];
    return cudaSuccess;
}

template <int HD, bool SPLIT>
static cudaError_t launch_attn_t(const CUtensorMap &q, const CUtensorMap &k, const CUtensorMap &v,
                                 const CUtensorMap &o, const AttnParams &p, cudaStream_t st)
{
    using C = AttnCfg<HD>;
    static std::atomic<uint64_t> configured{0};
    cudaError_t e = set_dyn_smem_once(replay_attn_kernel<HD, SPLIT>, C::kDynSmem, configured);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(p.total_items));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = C::kDynSmem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, replay_attn_kernel<HD, SPLIT>, q, k, v, o, p);
}

cudaError_t launch_replay_attn(int head_dim, bool split, const CUtensorMap &tm_q, const CUtensorMap &tm_k,
                               const CUtensorMap &tm_v, const CUtensorMap &tm_o, const AttnParams &p, cudaStream_t st)
{
    if (p.total_items <= 0) return cudaSuccess;
    if (head_dim == 128)
        return split ? launch_attn_t<128, true>(tm_q, tm_k, tm_v, tm_o, p, st)
                     : launch_attn_t<128, false>(tm_q, tm_k, tm_v, tm_o, p, st);
    if (head_dim == 64)
        return split ? launch_attn_t<64, true>(tm_q, tm_k, tm_v, tm_o, p, st)
                     : launch_attn_t<64, false>(tm_q, tm_k, tm_v, tm_o, p, st);
    return cudaErrorInvalidValue;
}

cudaError_t launch_splitkv_combine(int head_dim, const AttnParams &p, cudaStream_t st)
{
    if (p.total_comb <= 0) return cudaSuccess;
    if (head_dim != 64 && head_dim != 128) return cudaErrorInvalidValue;
    const int warps_per_block = 8;
    const int64_t warps = static_cast<int64_t>(p.total_comb + 31) / 32 * (head_dim / 32);  // row blocks x column groups
    const int blocks = static_cast<int>((warps + warps_per_block - 1) / warps_per_block);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(blocks));
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (head_dim == 128) return cudaLaunchKernelEx(&cfg, splitkv_combine_kernel<128>, p);
    if (head_dim == 64) return cudaLaunchKernelEx(&cfg, splitkv_combine_kernel<64>, p);
    return cudaErrorInvalidValue;
}

}  // namespace pe

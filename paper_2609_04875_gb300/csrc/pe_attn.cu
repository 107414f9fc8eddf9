// Replay attention over a paged KV cache on sm_103a (tcgen05 + TMEM + TMA).
//
// What it computes (Alg. 1 replay loop; the sanitized suffix is re-prefilled
// on the cropped cache, Sec. 3.2 / Sec. 4.5): for the last n_q positions of a
// sequence, query i at position len-n_q+i and q-head h attend the keys
// 0..len-n_q+i of kv-head h / (Hq/Hkv):
//     O = softmax(scale * q K^T) V      (bf16 in, fp32 accumulate, bf16 out)
//
// One CTA computes one work item: (sequence, kv-head, q-tile[, key split]).
// A q-tile packs 128 rows = (128/g queries) x (g q-heads of one kv-head), so K
// and V tiles are read once for the whole GQA group.  Roles (192 threads):
//   warps 0-3  softmax: thread r owns row r (TMEM lane r); masks, online
//              softmax in fp32 (exp2), writes P (bf16) to shared memory,
//              rescales O in TMEM when needed, epilogue.
//   warp 4     producer: reads the page table and issues one TMA box per
//              (page, 64-column half) into a K/V stage ring.
//   warp 5     MMA: allocates TMEM; one thread issues tcgen05.mma for
//              S = Q K^T (TMEM, double-buffered) and O += P V (TMEM).
// Key tiles always start at logical key 0 (multiples of 128 keys), whatever
// the physical pages, so a row's arithmetic depends only on its own keys.
//
// Online softmax with a lazily moved reference: a row's reference max m_ref
// only moves when a new tile's max exceeds it by more than 2^8 (then O and l
// are rescaled in place); otherwise exp2(x - m_ref) <= 256, exact in the final
// O / l.  Rows decide independently.
//
// Every wait is bounded (kWaitNs); on expiry the CTA records a status code,
// all roles leave their loops, and TMEM is freed before exit.
#include <cuda_bf16.h>

#include "pe_internal.h"
#include "ptx.cuh"

namespace pe {

constexpr uint64_t kWaitNs = 1000000000ull;  // 1 s
constexpr float kRescaleThreshold = 8.0f;    // log2 units

template <int HD>
struct AttnCfg {
    static constexpr int kRegions = HD / 64;            // 128-byte swizzle atoms along d
    static constexpr int kTileBytes = kBM * HD * 2;     // one Q, K or V tile (128 rows)
    static constexpr int kRegionBytes = kBM * 128;      // 128 rows x 128 bytes
    static constexpr int kStages = (HD == 128) ? 2 : 4;
    static constexpr int kPBytes = kBM * kBN * 2;       // P tile: 128 rows x 128 keys bf16
    static constexpr int kOffQ = 0;
    static constexpr int kOffK = kOffQ + kTileBytes;
    static constexpr int kOffV = kOffK + kStages * kTileBytes;
    static constexpr int kOffP = kOffV + kStages * kTileBytes;
    static constexpr int kOffBar = kOffP + 2 * kPBytes;
    // barriers: q_full, k_full[S], v_full[S], kv_empty[S], s_full[2], s_free[2], p_full[2], pv_done[2]
    static constexpr int kNumBars = 1 + 3 * kStages + 8;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;  // tmem slot, abort flag
    static constexpr int kSmemBytes = kOffMisc + 16;
    static constexpr int kDynSmem = kSmemBytes + 1024;       // alignment slack
    static constexpr uint32_t kTmemCols = 512;               // S0 | S1 | O
    static_assert(kDynSmem <= 232448, "shared memory budget");
};

struct Bars {
    uint32_t q_full, k_full0, v_full0, kv_empty0, s_full0, s_free0, p_full0, pv_done0;
};

struct WaitCtx {
    volatile int *abort;
    int32_t *status;
};

// Bounded mbarrier wait.  Returns false (and stops the CTA's pipeline) when the
// wait ran out or another role already gave up.
__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, const WaitCtx &w)
{
    if (ptx::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = ptx::globaltimer();
    for (;;) {
        if (ptx::mbar_try_wait(bar, parity)) return true;
        if (*w.abort) return false;
        if (ptx::globaltimer() - t0 > kWaitNs) {
            *w.abort = 1;
            atomicCAS(w.status, 0, kStatusWaitTimeout);
            return false;
        }
    }
}

// Warp-collective form: every lane waits, and the warp proceeds only if all
// lanes saw the phase complete, so no lane reaches a .sync.aligned tcgen05
// instruction without its warp-mates.
__device__ __forceinline__ bool wait_bar_warp(uint32_t bar, uint32_t parity, const WaitCtx &w)
{
    const bool ok = wait_bar(bar, parity, w);
    return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&h);
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d)
{
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d)
                 : "memory");
}

template <int HD, bool SPLIT>
__global__ void __launch_bounds__(192, 1)
    replay_attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                       const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ AttnParams p)
{
    using C = AttnCfg<HD>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = ptx::smem_addr(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;
    uint8_t *smem = smem_raw + (sbase - raw);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    // ---- work item -> (sequence, kv-head, split, q-tile); heaviest q-tiles first
    const int item = blockIdx.x;
    int si = 0;
    while (si + 1 < p.n_seqs && item >= p.seqs[si + 1].item0) ++si;
    const AttnSeq &sq = p.seqs[si];
    int local = item - sq.item0;
    const int kvh = local % p.hkv;
    local /= p.hkv;
    const int split = local % sq.n_splits;
    local /= sq.n_splits;
    const int qt = sq.n_qtiles - 1 - local;
    const int g = p.group;
    const int bmq = kBM / g;
    const int q_first = qt * bmq;
    const int q_last = min(q_first + bmq, sq.n_q) - 1;
    const int pos_first = sq.n_keys - sq.n_q + q_first;   // position of the tile's first query
    const int k_end = sq.n_keys - sq.n_q + q_last + 1;    // keys needed by the tile's last query
    const int nkt = (k_end + kBN - 1) / kBN;
    int kt0 = 0, kt1 = nkt;
    if (SPLIT) {
        kt0 = split * p.split_tiles;
        kt1 = min(nkt, kt0 + p.split_tiles);
    }
    const int ntiles = max(0, kt1 - kt0);

    // ---- shared memory carve-up
    const uint32_t q_smem = sbase + C::kOffQ;
    const uint32_t k_smem0 = sbase + C::kOffK;
    const uint32_t v_smem0 = sbase + C::kOffV;
    const uint32_t p_smem0 = sbase + C::kOffP;
    const uint32_t bar0 = sbase + C::kOffBar;
    Bars B;
    B.q_full = bar0;
    B.k_full0 = bar0 + 8;
    B.v_full0 = B.k_full0 + 8 * C::kStages;
    B.kv_empty0 = B.v_full0 + 8 * C::kStages;
    B.s_full0 = B.kv_empty0 + 8 * C::kStages;
    B.s_free0 = B.s_full0 + 16;
    B.p_full0 = B.s_free0 + 16;
    B.pv_done0 = B.p_full0 + 16;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + C::kOffMisc);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + C::kOffMisc + 4);
    const WaitCtx wctx{abort_flag, p.status};

    if (threadIdx.x == 0) {
        ptx::mbar_init(B.q_full, 1);
        for (int s = 0; s < C::kStages; ++s) {
            ptx::mbar_init(B.k_full0 + 8 * s, 1);
            ptx::mbar_init(B.v_full0 + 8 * s, 1);
            ptx::mbar_init(B.kv_empty0 + 8 * s, 1);
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(B.s_full0 + 8 * b, 1);
            ptx::mbar_init(B.s_free0 + 8 * b, 128);
            ptx::mbar_init(B.p_full0 + 8 * b, 128);
            ptx::mbar_init(B.pv_done0 + 8 * b, 1);
        }
        *abort_flag = 0;
        ptx::fence_barrier_init();
        ptx::fence_proxy_async_smem();
    }
    if (warp == 4 && lane == 0) {
        ptx::prefetch_tensormap(&tm_q);
        ptx::prefetch_tensormap(&tm_k);
        ptx::prefetch_tensormap(&tm_v);
    }
    if (warp == 5) {
        ptx::tmem_alloc(ptx::smem_addr(tmem_slot), C::kTmemCols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const uint32_t tS0 = tmem;          // S buffer b at column 128*b
    const uint32_t tO = tmem + 256;     // O accumulator: HD columns

    if (ntiles > 0 && warp == 4) {
        // =================================================== producer (TMA)
        if (lane == 0) {
            ptx::mbar_arrive_expect_tx(B.q_full, C::kTileBytes);
            for (int r = 0; r < C::kRegions; ++r)
                ptx::tma_load_3d(q_smem + r * C::kRegionBytes, &tm_q, r * 64, kvh * g, sq.q_row0 + q_first,
                                 B.q_full);
        }
        const int ppt = kBN / p.ps;  // pages per key tile
        for (int i = 0; i < ntiles; ++i) {
            const int s = i % C::kStages;
            if (i >= C::kStages && !wait_bar_warp(B.kv_empty0 + 8 * s, ((i / C::kStages) - 1) & 1, wctx)) break;
            const int lp = (kt0 + i) * ppt + lane;
            int page = -1;
            if (lane < ppt && lp < sq.n_pages) page = p.page_table[sq.table_row + lp];
            const uint32_t kdst = k_smem0 + s * C::kTileBytes;
            const uint32_t vdst = v_smem0 + s * C::kTileBytes;
            if (lane == 0) {
                ptx::mbar_arrive_expect_tx(B.k_full0 + 8 * s, C::kTileBytes);
                ptx::mbar_arrive_expect_tx(B.v_full0 + 8 * s, C::kTileBytes);
            }
            for (int j = 0; j < ppt; ++j) {
                const int pg = __shfl_sync(0xffffffffu, page, j);
                if (lane == 0) {
                    // rows of pages past the sequence read as zeros (out-of-bounds box)
                    const int y = pg >= 0 ? ((p.layer * p.num_pages + pg) * p.hkv + kvh) * p.ps : p.oob_row;
                    for (int r = 0; r < C::kRegions; ++r) {
                        const uint32_t off = r * C::kRegionBytes + j * p.ps * 128;
                        ptx::tma_load_2d(kdst + off, &tm_k, r * 64, y, B.k_full0 + 8 * s);
                        ptx::tma_load_2d(vdst + off, &tm_v, r * 64, y, B.v_full0 + 8 * s);
                    }
                }
            }
        }
        __syncwarp();
        if (*abort_flag && lane == 0) {
            // give copies in flight a bounded chance to land before the CTA exits
            const int first = max(0, ntiles - C::kStages);
            for (int i = first; i < ntiles; ++i) {
                const int s = i % C::kStages;
                const uint64_t t0 = ptx::globaltimer();
                while (!ptx::mbar_try_wait(B.k_full0 + 8 * s, (i / C::kStages) & 1) &&
                       ptx::globaltimer() - t0 < 1000000ull) {}
                while (!ptx::mbar_try_wait(B.v_full0 + 8 * s, (i / C::kStages) & 1) &&
                       ptx::globaltimer() - t0 < 2000000ull) {}
            }
        }
    } else if (ntiles > 0 && warp == 5) {
        // =================================================== MMA issuer
        if (lane == 0) {
            constexpr uint32_t kIdescQK = ptx::idesc_bf16_f32(kBM, kBN, false);
            constexpr uint32_t kIdescPV = ptx::idesc_bf16_f32(kBM, HD, true);
            bool ok = wait_bar(B.q_full, 0, wctx);
            auto issue_pv = [&](int i) -> bool {
                const int s = i % C::kStages;
                const int b = i & 1;
                if (!wait_bar(B.p_full0 + 8 * b, (i >> 1) & 1, wctx)) return false;
                if (!wait_bar(B.v_full0 + 8 * s, (i / C::kStages) & 1, wctx)) return false;
                ptx::tc_fence_after();
                const uint32_t pa = p_smem0 + b * C::kPBytes;
                const uint32_t vb = v_smem0 + s * C::kTileBytes;
#pragma unroll
                for (int kk = 0; kk < kBN / 16; ++kk) {
                    const uint64_t da = ptx::smem_desc_sw128(pa + (kk >> 2) * C::kRegionBytes + (kk & 3) * 32, 16, 1024);
                    const uint64_t db = ptx::smem_desc_sw128(vb + kk * 16 * 128, C::kRegionBytes, 1024);
                    ptx::mma_bf16(tO, da, db, kIdescPV, (i > 0 || kk > 0) ? 1u : 0u);
                }
                ptx::mma_commit(B.kv_empty0 + 8 * s);
                ptx::mma_commit(B.pv_done0 + 8 * b);
                return true;
            };
            for (int i = 0; ok && i < ntiles; ++i) {
                const int s = i % C::kStages;
                const int b = i & 1;
                if (!wait_bar(B.k_full0 + 8 * s, (i / C::kStages) & 1, wctx)) { ok = false; break; }
                if (i >= 2 && !wait_bar(B.s_free0 + 8 * b, ((i >> 1) - 1) & 1, wctx)) { ok = false; break; }
                ptx::tc_fence_after();
                const uint32_t kb = k_smem0 + s * C::kTileBytes;
#pragma unroll
                for (int kk = 0; kk < HD / 16; ++kk) {
                    const uint32_t off = (kk >> 2) * C::kRegionBytes + (kk & 3) * 32;
                    const uint64_t da = ptx::smem_desc_sw128(q_smem + off, 16, 1024);
                    const uint64_t db = ptx::smem_desc_sw128(kb + off, 16, 1024);
                    ptx::mma_bf16(tS0 + 128 * b, da, db, kIdescQK, kk > 0 ? 1u : 0u);
                }
                ptx::mma_commit(B.s_full0 + 8 * b);
                if (i >= 1 && !issue_pv(i - 1)) { ok = false; break; }
            }
            if (ok) issue_pv(ntiles - 1);
        }
        __syncwarp();
    } else if (warp < 4) {
        // =================================================== softmax / epilogue
        const int row = threadIdx.x;  // TMEM lane
        const int qi = q_first + row / g;
        const bool valid = qi <= q_last;
        const int pos = sq.n_keys - sq.n_q + qi;
        const uint32_t lane_off = static_cast<uint32_t>(warp * 32) << 16;
        const float sl2 = p.scale_log2;
        float m_ref = -INFINITY;
        float l = 0.f;
        bool ok = true;
        for (int i = 0; i < ntiles; ++i) {
            const int b = i & 1;
            const int kbase = (kt0 + i) * kBN;
            if (!wait_bar_warp(B.s_full0 + 8 * b, (i >> 1) & 1, wctx)) { ok = false; break; }
            ptx::tc_fence_after();
            __syncwarp();
            float s[kBN];
            {
                float (&s0)[32] = *reinterpret_cast<float (*)[32]>(&s[0]);
                float (&s1)[32] = *reinterpret_cast<float (*)[32]>(&s[32]);
                float (&s2)[32] = *reinterpret_cast<float (*)[32]>(&s[64]);
                float (&s3)[32] = *reinterpret_cast<float (*)[32]>(&s[96]);
                const uint32_t ts = tS0 + 128 * b + lane_off;
                ptx::tmem_ld32(ts + 0, s0);
                ptx::tmem_ld32(ts + 32, s1);
                ptx::tmem_ld32(ts + 64, s2);
                ptx::tmem_ld32(ts + 96, s3);
                ptx::tmem_wait_ld();
            }
            ptx::tc_fence_before();
            ptx::mbar_arrive(B.s_free0 + 8 * b);
            if (kbase + kBN - 1 > pos_first) {  // tile crosses the causal diagonal of some row
#pragma unroll
                for (int c = 0; c < kBN; ++c)
                    if (kbase + c > pos) s[c] = -INFINITY;
            }
            float mx = -INFINITY;
#pragma unroll
            for (int c = 0; c < kBN; ++c) mx = fmaxf(mx, s[c]);
            const float m_new = fmaxf(m_ref, mx * sl2);
            if (i == 0) {
                m_ref = (m_new == -INFINITY) ? 0.f : m_new;
            } else {
                const bool need = m_new > m_ref + kRescaleThreshold;
                if (__any_sync(0xffffffffu, need)) {
                    // O holds PV of tiles < i once PV_{i-1} completed; PV_i waits for our P
                    if (!wait_bar_warp(B.pv_done0 + 8 * ((i - 1) & 1), ((i - 1) >> 1) & 1, wctx)) { ok = false; break; }
                    ptx::tc_fence_after();
                    __syncwarp();
                    const float alpha = need ? ex2(m_ref - m_new) : 1.0f;
#pragma unroll
                    for (int ch = 0; ch < HD / 32; ++ch) {
                        float o[32];
                        ptx::tmem_ld32(tO + lane_off + ch * 32, o);
                        ptx::tmem_wait_ld();
#pragma unroll
                        for (int j = 0; j < 32; ++j) o[j] *= alpha;
                        ptx::tmem_st32(tO + lane_off + ch * 32, o);
                    }
                    ptx::tmem_wait_st();
                    if (need) {
                        l *= alpha;
                        m_ref = m_new;
                    }
                }
            }
            // P buffer b is free once PV_{i-2} completed
            if (i >= 2 && !wait_bar_warp(B.pv_done0 + 8 * b, ((i >> 1) - 1) & 1, wctx)) { ok = false; break; }
            const float neg_ref = -m_ref;
            float rs = 0.f;
            const uint32_t prow = p_smem0 + b * C::kPBytes + row * 128;
#pragma unroll
            for (int cidx = 0; cidx < kBN / 8; ++cidx) {
                float e[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    e[j] = ex2(fmaf(s[cidx * 8 + j], sl2, neg_ref));
                    rs += e[j];
                }
                const uint32_t addr = prow + (cidx >> 3) * C::kRegionBytes + ((((cidx & 7) ^ (row & 7))) << 4);
                st_shared_v4(addr, pack_bf16(e[0], e[1]), pack_bf16(e[2], e[3]), pack_bf16(e[4], e[5]),
                             pack_bf16(e[6], e[7]));
            }
            l += rs;
            ptx::fence_proxy_async_smem();
            ptx::tc_fence_before();
            ptx::mbar_arrive(B.p_full0 + 8 * b);
        }
        // ---- epilogue: O / l
        if (ok && ntiles > 0) {
            const int last = ntiles - 1;
            ok = wait_bar_warp(B.pv_done0 + 8 * (last & 1), (last >> 1) & 1, wctx);
        }
        if (ok && ntiles > 0) {
            ptx::tc_fence_after();
            __syncwarp();
            const float inv = l > 0.f ? 1.0f / l : 0.f;
            const int head = kvh * g + (row % g);
            if (!SPLIT) {
                __nv_bfloat16 *dst = reinterpret_cast<__nv_bfloat16 *>(p.out) +
                                     (static_cast<int64_t>(sq.q_row0 + qi) * p.hq + head) * HD;
#pragma unroll
                for (int ch = 0; ch < HD / 32; ++ch) {
                    float o[32];
                    ptx::tmem_ld32(tO + lane_off + ch * 32, o);
                    ptx::tmem_wait_ld();
                    if (valid) {
                        uint4 *d4 = reinterpret_cast<uint4 *>(dst + ch * 32);
#pragma unroll
                        for (int j = 0; j < 4; ++j)
                            d4[j] = make_uint4(pack_bf16(o[8 * j + 0] * inv, o[8 * j + 1] * inv),
                                               pack_bf16(o[8 * j + 2] * inv, o[8 * j + 3] * inv),
                                               pack_bf16(o[8 * j + 4] * inv, o[8 * j + 5] * inv),
                                               pack_bf16(o[8 * j + 6] * inv, o[8 * j + 7] * inv));
                    }
                }
            } else {
                const int64_t prow_idx =
                    sq.part_row0 + (static_cast<int64_t>(qt * p.hkv + kvh) * sq.n_splits + split) * kBM + row;
                float *dst = p.part_o + prow_idx * HD;
#pragma unroll
                for (int ch = 0; ch < HD / 32; ++ch) {
                    float o[32];
                    ptx::tmem_ld32(tO + lane_off + ch * 32, o);
                    ptx::tmem_wait_ld();
                    if (valid && l > 0.f) {
                        float4 *d4 = reinterpret_cast<float4 *>(dst + ch * 32);
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            d4[j] = make_float4(o[4 * j] * inv, o[4 * j + 1] * inv, o[4 * j + 2] * inv,
                                                o[4 * j + 3] * inv);
                    }
                }
                if (valid) p.part_lse[prow_idx] = l > 0.f ? m_ref + __log2f(l) : -INFINITY;
            }
        }
    }
    if (SPLIT && ntiles == 0 && warp < 4) {
        // empty key range: this split contributes nothing to its rows
        const int row = threadIdx.x;
        const int qi = q_first + row / g;
        if (qi <= q_last) {
            const int64_t prow_idx =
                sq.part_row0 + (static_cast<int64_t>(qt * p.hkv + kvh) * sq.n_splits + split) * kBM + row;
            p.part_lse[prow_idx] = -INFINITY;
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 5) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, C::kTmemCols);
    }
}

// One warp per output row: LSE-weighted merge of the split partials.
template <int HD>
__global__ void __launch_bounds__(256) splitkv_combine_kernel(const __grid_constant__ AttnParams p)
{
    const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (gw >= p.total_comb) return;
    int si = 0;
    while (si + 1 < p.n_seqs && gw >= p.seqs[si + 1].comb0) ++si;
    const AttnSeq &sq = p.seqs[si];
    const int local = gw - sq.comb0;
    const int row = local % kBM;
    const int unit = local / kBM;  // qt * hkv + kvh
    const int kvh = unit % p.hkv;
    const int qt = unit / p.hkv;
    const int g = p.group;
    const int qi = qt * (kBM / g) + row / g;
    if (qi >= sq.n_q) return;
    const int64_t base = sq.part_row0 + static_cast<int64_t>(unit) * sq.n_splits * kBM + row;
    float mx = -INFINITY;
    for (int s = 0; s < sq.n_splits; ++s) mx = fmaxf(mx, p.part_lse[base + static_cast<int64_t>(s) * kBM]);
    constexpr int kPer = HD / 32;
    float acc[kPer];
#pragma unroll
    for (int j = 0; j < kPer; ++j) acc[j] = 0.f;
    float den = 0.f;
    if (mx != -INFINITY) {
        for (int s = 0; s < sq.n_splits; ++s) {
            const int64_t r = base + static_cast<int64_t>(s) * kBM;
            const float lse = p.part_lse[r];
            if (lse == -INFINITY) continue;
            const float w = ex2(lse - mx);
            den += w;
            const float *src = p.part_o + r * HD + lane * kPer;
#pragma unroll
            for (int j = 0; j < kPer; ++j) acc[j] += w * src[j];
        }
    }
    const float inv = den > 0.f ? 1.0f / den : 0.f;
    const int head = kvh * g + (row % g);
    __nv_bfloat16 *dst = reinterpret_cast<__nv_bfloat16 *>(p.out) +
                         (static_cast<int64_t>(sq.q_row0 + qi) * p.hq + head) * HD + lane * kPer;
    if (kPer == 4) {
        uint2 v = make_uint2(pack_bf16(acc[0] * inv, acc[1] * inv), pack_bf16(acc[2] * inv, acc[3] * inv));
        *reinterpret_cast<uint2 *>(dst) = v;
    } else {
        *reinterpret_cast<uint32_t *>(dst) = pack_bf16(acc[0] * inv, acc[kPer - 1] * inv);
    }
}

template <int HD, bool SPLIT>
static cudaError_t launch_attn_t(const CUtensorMap &q, const CUtensorMap &k, const CUtensorMap &v,
                                 const AttnParams &p, cudaStream_t st)
{
    using C = AttnCfg<HD>;
    static bool configured = false;
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(replay_attn_kernel<HD, SPLIT>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, C::kDynSmem);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    replay_attn_kernel<HD, SPLIT><<<p.total_items, 192, C::kDynSmem, st>>>(q, k, v, p);
    return cudaGetLastError();
}

cudaError_t launch_replay_attn(int head_dim, bool split, const CUtensorMap &tm_q, const CUtensorMap &tm_k,
                               const CUtensorMap &tm_v, const AttnParams &p, cudaStream_t st)
{
    if (p.total_items <= 0) return cudaSuccess;
    if (head_dim == 128)
        return split ? launch_attn_t<128, true>(tm_q, tm_k, tm_v, p, st)
                     : launch_attn_t<128, false>(tm_q, tm_k, tm_v, p, st);
    if (head_dim == 64)
        return split ? launch_attn_t<64, true>(tm_q, tm_k, tm_v, p, st)
                     : launch_attn_t<64, false>(tm_q, tm_k, tm_v, p, st);
    return cudaErrorInvalidValue;
}

cudaError_t launch_splitkv_combine(int head_dim, const AttnParams &p, cudaStream_t st)
{
    if (p.total_comb <= 0) return cudaSuccess;
    const int warps_per_block = 8;
    const int blocks = (p.total_comb + warps_per_block - 1) / warps_per_block;
    if (head_dim == 128)
        splitkv_combine_kernel<128><<<blocks, 256, 0, st>>>(p);
    else if (head_dim == 64)
        splitkv_combine_kernel<64><<<blocks, 256, 0, st>>>(p);
    else
        return cudaErrorInvalidValue;
    return cudaGetLastError();
}

}  // namespace pe

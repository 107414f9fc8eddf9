// Decode attention over a paged KV cache on sm_103a.
//
// What it computes (Alg. 1 replay loop for positions that are generated again
// one per pass; Sec. 4.5: target-dependent turns are re-decoded): the n_q x g
// query rows of one kv-head -- at most 16, e.g. one new position of a GQA
// group -- attend the sequence's keys, query i at position len-n_q+i seeing
// keys 0..len-n_q+i:
//     O = softmax(scale * q K^T) V      (bf16 in, fp32 accumulate, bf16 out)
//
// With so few rows per key this is a stream over the sequence's K/V, bound by
// HBM, not by a contraction: CUDA cores do the arithmetic and the design keeps
// HBM busy.  One CTA = (sequence, kv-head, key split):
//   warp 8       producer: reads page ids one tile ahead; its lanes issue one
//                TMA box per (page, 64-column half) of K and of V into a
//                3-stage ring of 64-key tiles (128-byte swizzle, so that
//                reads along a key and along a column are both conflict-free).
//                Boxes past the sequence read zeros.
//   warps 0-7    consumers, each an independent online-softmax worker over
//                its own keys [8w, 8w+8) of every tile (no CTA barrier per
//                tile):
//     1. scores: lane l takes key 8w + l/4 and the d-quarter l%4; its partial
//        dots with the RB query rows (fp32, shared memory) are summed over the
//        key's four lanes by a reduce-scatter, leaving each lane RB/4 rows;
//     2. softmax over the warp's 8 keys per row: running max m and sum l in
//        registers, weights P (exp2) to a warp-private shared buffer;
//     3. O[r][cols] = alpha_r O[r][cols] + sum_k P[k][r] V[k][cols], lane l
//        taking the columns [l*d/32, (l+1)*d/32).
//   After the last tile the 8 warps' (m, l, O) are merged through shared
//   memory.  With one split the rows are normalised and written.  With several,
//   each split writes (O, m, l) to the workspace and the last split of a
//   (sequence, kv-head) to finish -- a ticket counter -- merges them, so no
//   second launch is needed; it resets the counter for the next launch.
// Keys past the sequence or past a row's query position get weight 0.  Every
// wait is bounded.
#include "dev_common.cuh"

namespace pe {
namespace {

constexpr int kDecWarps = 8;                       // consumer warps
constexpr int kConsumers = 32 * kDecWarps;
constexpr int kDecThreads = kConsumers + 32;       // + producer warp
constexpr int kDecStages = 3;
constexpr int kBarConsumers = 1;                   // named barrier of the consumer warps
constexpr int kStatusBadPage = 2;                  // device status: page id outside the pool

// Every split of a (sequence, kv-head) has written its partial (O, m, l) for
// the RB rows: O unnormalised [RB][HD], m the running max (log2 units), l the
// sum of exp2(x - m).  Each split takes a ticket (also after an abort, so the
// counter returns to 0); the last one merges the partials into the bf16
// output, O = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s, and resets the
// counter for the next launch.  Called by `nthreads` threads (whole warps,
// thread ids 0..nthreads-1) that share named barrier `bar`.
template <int RB, int HD>
__device__ __forceinline__ void split_merge(const DecodeParams &p, const DecodeSeq &sq, int si, int kvh, int n_rows,
                                            int tid, int nthreads, int bar, int *s_ticket)
{
    const float *pm = p.part + static_cast<int64_t>(p.total_ctas) * RB * HD;
    const float *pl = pm + static_cast<int64_t>(p.total_ctas) * RB;
    const int g = p.group;
    __threadfence();
    ptx::bar_sync(bar, nthreads);
    int32_t *ticket = p.tickets + si * p.hkv + kvh;
    if (tid == 0) *s_ticket = atomicAdd(ticket, 1);
    ptx::bar_sync(bar, nthreads);
    if (*s_ticket != sq.n_splits - 1) return;
    __threadfence();
    const int64_t c0 = sq.cta0 + static_cast<int64_t>(kvh) * sq.n_splits;
    for (int e = tid; e < RB * HD / 2; e += nthreads) {
        const int r = (2 * e) / HD;
        const int col = (2 * e) % HD;
        if (r >= n_rows) continue;
        float mx = -INFINITY;
        for (int sp = 0; sp < sq.n_splits; ++sp) mx = fmaxf(mx, __ldcg(pm + (c0 + sp) * RB + r));
        float den = 0.f, o0 = 0.f, o1 = 0.f;
        if (mx != -INFINITY) {
            for (int sp = 0; sp < sq.n_splits; ++sp) {
                const float ms = __ldcg(pm + (c0 + sp) * RB + r);
                if (ms == -INFINITY) continue;
                const float w = ex2(ms - mx);
                den += w * __ldcg(pl + (c0 + sp) * RB + r);
                const float2 x =
                    __ldcg(reinterpret_cast<const float2 *>(p.part + ((c0 + sp) * RB + r) * HD + col));
                o0 += w * x.x;
                o1 += w * x.y;
            }
        }
        const float inv = den > 0.f ? 1.0f / den : 0.f;
        __nv_bfloat16 *dst = static_cast<__nv_bfloat16 *>(p.out) +
                             (static_cast<int64_t>(sq.q_row0 + r / g) * p.hq + kvh * g + r % g) * HD + col;
        *reinterpret_cast<uint32_t *>(dst) = pack_bf16(o0 * inv, o1 * inv);
    }
    if (tid == 0) *ticket = 0;
}

template <int HD, int RB>
struct DecCfg {
    static constexpr int kRegions = HD / 64;                 // 128-byte swizzle atoms along d
    static constexpr int kRegionBytes = kDecKeys * 128;      // 64 keys x 64 columns (bf16)
    static constexpr int kTileBytes = kRegions * kRegionBytes;
    static constexpr int kStageBytes = 2 * kTileBytes;       // K then V
    static constexpr int kQuarter = HD / 4;                  // d-columns per scoring lane
    static constexpr int kQChunks = kQuarter / 8;            // 16-byte chunks per quarter row
    static constexpr int kQStride = kQuarter + 4;            // floats per (row, quarter) of q: spreads banks
    static constexpr int kRPL = RB / 4;                      // score rows per lane
    static constexpr int kCW = HD / 32;                      // d-columns per lane in P V
    static constexpr int kOffQ = kDecStages * kStageBytes;   // q [RB][4][kQStride] fp32, log2 units
    static constexpr int kOffPw = kOffQ + RB * 4 * kQStride * 4;   // per warp: P [8 keys][RB], alpha [RB]
    static constexpr int kPwFloats = 8 * RB + RB;
    static constexpr int kOffML = kOffPw + kDecWarps * kPwFloats * 4;  // merge: m, l [8 warps][RB]
    static constexpr int kOffBar = kOffML + 2 * kDecWarps * RB * 4;    // full[S], empty[S]
    static constexpr int kOffMisc = kOffBar + 2 * kDecStages * 8;  // abort flag, ticket, tiles issued
    static constexpr int kSmem = kOffMisc + 16;
    static constexpr int kDynSmem = kSmem + 1024;            // the stages start 1024-byte aligned
    static constexpr int kMinBlocks = RB <= 8 ? 2 : 1;
    static_assert(RB == 4 || RB == 8 || RB == 16, "row capacity");
    static_assert(kDecWarps * RB * HD * 4 <= kDecStages * kStageBytes, "the O merge reuses the stages");
    static_assert(kOffBar % 8 == 0, "mbarrier alignment");
};

template <int HD, int RB>
__global__ void __launch_bounds__(kDecThreads, DecCfg<HD, RB>::kMinBlocks)
    decode_attn_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                       const __grid_constant__ DecodeParams p)
{
    using C = DecCfg<HD, RB>;
    constexpr int CW = C::kCW;
    constexpr int RPL = C::kRPL;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    int si = 0;
    while (si + 1 < p.n_seqs && static_cast<int>(blockIdx.x) >= p.seqs[si + 1].cta0) ++si;
    const DecodeSeq &sq = p.seqs[si];
    const int local = static_cast<int>(blockIdx.x) - sq.cta0;
    const int kvh = local / sq.n_splits;
    const int split = local - kvh * sq.n_splits;
    const int g = p.group;
    const int n_rows = sq.n_q * g;
    const int n_tiles_all = (sq.n_keys + kDecKeys - 1) / kDecKeys;
    const int t0 = split * p.split_tiles;
    const int nt = max(0, min(t0 + p.split_tiles, n_tiles_all) - t0);
    const int qpos0 = sq.n_keys - sq.n_q;  // position of query 0

    float *s_q = reinterpret_cast<float *>(smem + C::kOffQ);
    float *s_ml = reinterpret_cast<float *>(smem + C::kOffML);
    const uint32_t bar0 = ptx::smem_addr(smem + C::kOffBar);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + C::kOffMisc);
    int *s_ticket = reinterpret_cast<int *>(smem + C::kOffMisc + 4);
    volatile int *s_issued = reinterpret_cast<volatile int *>(smem + C::kOffMisc + 8);
    const WaitCtx wctx{abort_flag, p.status};
    auto full = [&](int s) { return bar0 + 8u * s; };
    auto empty = [&](int s) { return bar0 + 8u * (kDecStages + s); };

    if (threadIdx.x == kConsumers) {
        for (int s = 0; s < kDecStages; ++s) {
            ptx::mbar_init(full(s), 1);
            ptx::mbar_init(empty(s), kDecWarps);
        }
        *abort_flag = 0;
        *s_issued = 0;
        ptx::fence_barrier_init();
        ptx::fence_proxy_async_smem();
        ptx::prefetch_tensormap(&tm_k);
        ptx::prefetch_tensormap(&tm_v);
    }
    // this kv-head's query rows, scaled to log2 units (rows past n_q x g are zero)
    for (int e = threadIdx.x; e < RB * HD; e += kDecThreads) {
        const int r = e / HD;
        const int col = e % HD;
        float x = 0.f;
        if (r < n_rows) {
            const __nv_bfloat16 *src = static_cast<const __nv_bfloat16 *>(p.q) +
                                       (static_cast<int64_t>(sq.q_row0 + r / g) * p.hq + kvh * g + r % g) * HD;
            x = __bfloat162float(src[col]) * p.scale_log2;
        }
        s_q[(r * 4 + col / C::kQuarter) * C::kQStride + col % C::kQuarter] = x;
    }
    __syncthreads();

    if (warp == kDecWarps) {
        // ============================================================ producer
        const int kpc = p.ps < kDecKeys ? p.ps : kDecKeys;  // keys per box (the tensor maps' box height)
        const int n_ops = (kDecKeys / kpc) * C::kRegions;   // boxes per tile and operand, <= 16
        const int op_slot = lane / C::kRegions;             // this lane's page slot in the tile
        const int op_reg = lane % C::kRegions;              // and 64-column half
        const bool op_on = lane < n_ops;
        // this lane's raw page id of tile t (checked where it is used), -1 past the sequence
        auto page_of = [&](int t) -> int {
            const int key0 = t * kDecKeys + op_slot * kpc;
            if (!op_on || key0 >= sq.n_keys) return -1;
            return p.page_table[sq.table_row + key0 / p.ps];
        };
        int page_next = nt > 0 ? page_of(t0) : -1;
        for (int i = 0; i < nt; ++i) {
            const int t = t0 + i;
            const int s = i % kDecStages;
            const int page = page_next;
            if (i + 1 < nt) page_next = page_of(t + 1);
            if (i >= kDecStages && !wait_bar_warp(empty(s), ((i / kDecStages) - 1) & 1, wctx)) break;
            if (lane == 0) ptx::mbar_arrive_expect_tx(full(s), 2u * C::kTileBytes);
            __syncwarp();
            if (op_on) {
                const int key0 = t * kDecKeys + op_slot * kpc;
                const bool ok_page = page >= 0 && page < p.num_pages;
                if (!ok_page && key0 < sq.n_keys) atomicCAS(p.status, 0, kStatusBadPage);
                const int y = ok_page ? ((p.layer * p.num_pages + page) * p.hkv + kvh) * p.ps + (key0 % p.ps)
                                      : p.oob_row;  // past the sequence (or a bad id): zeros
                const uint32_t dst =
                    ptx::smem_addr(smem + s * C::kStageBytes) + op_reg * C::kRegionBytes + op_slot * kpc * 128;
                ptx::tma_load_2d(dst, &tm_k, op_reg * 64, y, full(s));
                ptx::tma_load_2d(dst + C::kTileBytes, &tm_v, op_reg * 64, y, full(s));
            }
            __syncwarp();
            if (lane == 0) *s_issued = i + 1;
        }
    } else {
        // ============================================================ consumers
        float *s_pw = reinterpret_cast<float *>(smem + C::kOffPw) + warp * C::kPwFloats;  // P [8][RB], alpha [RB]
        const int kl = lane >> 2;                  // this lane's key among the warp's 8
        const int quarter = lane & 3;              // and d-quarter while scoring
        const int col0 = quarter * C::kQuarter;
        const int reg1 = col0 / 64;
        const int lc0 = (col0 % 64) / 8;           // first 16-byte chunk of the quarter in its row
        const int row0 = ((lane >> 1) & 1) * (RB / 2) + (lane & 1) * (RB / 4);  // rows [row0, row0 + RPL) after the reduce
        const float *qbase = s_q + quarter * C::kQStride;
        float m_run[RPL], l_run[RPL];
#pragma unroll
        for (int j = 0; j < RPL; ++j) {
            m_run[j] = -INFINITY;
            l_run[j] = 0.f;
        }
        float2 acc[RB][CW / 2];
#pragma unroll
        for (int r = 0; r < RB; ++r)
#pragma unroll
            for (int c = 0; c < CW / 2; ++c) acc[r][c] = make_float2(0.f, 0.f);

        for (int i = 0; i < nt; ++i) {
            const int s = i % kDecStages;
            if (!wait_bar_warp(full(s), (i / kDecStages) & 1, wctx)) break;
            const uint8_t *Ks = smem + s * C::kStageBytes;
            const uint8_t *Vs = Ks + C::kTileBytes;
            const int key = (t0 + i) * kDecKeys + warp * 8 + kl;

            // 1. partial scores of this lane's key over its quarter, all RB rows
            float v[RB];
            {
                float2 sa[RB], sb[RB];
#pragma unroll
                for (int r = 0; r < RB; ++r) {
                    sa[r] = make_float2(0.f, 0.f);
                    sb[r] = make_float2(0.f, 0.f);
                }
                const int krow = warp * 8 + kl;
                const uint8_t *kp = Ks + reg1 * C::kRegionBytes + krow * 128;
#pragma unroll
                for (int c = 0; c < C::kQChunks; ++c) {
                    const uint4 u = *reinterpret_cast<const uint4 *>(kp + (((lc0 + c) ^ (krow & 7)) << 4));
                    const float2 k0 = make_float2(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u));
                    const float2 k1 = make_float2(__uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
                    const float2 k2 = make_float2(__uint_as_float(u.z << 16), __uint_as_float(u.z & 0xffff0000u));
                    const float2 k3 = make_float2(__uint_as_float(u.w << 16), __uint_as_float(u.w & 0xffff0000u));
#pragma unroll
                    for (int r = 0; r < RB; ++r) {
                        const float4 qa = *reinterpret_cast<const float4 *>(qbase + r * 4 * C::kQStride + c * 8);
                        const float4 qb = *reinterpret_cast<const float4 *>(qbase + r * 4 * C::kQStride + c * 8 + 4);
                        sa[r] = fma2(make_float2(qa.x, qa.y), k0, sa[r]);
                        sb[r] = fma2(make_float2(qa.z, qa.w), k1, sb[r]);
                        sa[r] = fma2(make_float2(qb.x, qb.y), k2, sa[r]);
                        sb[r] = fma2(make_float2(qb.z, qb.w), k3, sb[r]);
                    }
                }
#pragma unroll
                for (int r = 0; r < RB; ++r) v[r] = (sa[r].x + sa[r].y) + (sb[r].x + sb[r].y);
            }
            // sum over the key's four lanes: reduce-scatter on lane bits 1 then 0
#pragma unroll
            for (int lvl = 0; lvl < 2; ++lvl) {
                const int n = RB >> lvl;
                const int off = 2 >> lvl;
                const bool upper = (lane & off) != 0;
#pragma unroll
                for (int j = 0; j < n / 2; ++j) {
                    const float send = upper ? v[j] : v[j + n / 2];
                    const float keep = upper ? v[j + n / 2] : v[j];
                    v[j] = keep + __shfl_xor_sync(0xffffffffu, send, off);
                }
            }
            // 2. online softmax over the warp's 8 keys (lanes with equal lane % 4 share rows)
            float alpha[RPL];
#pragma unroll
            for (int j = 0; j < RPL; ++j) {
                const int r = row0 + j;
                const int qpos = r < n_rows ? qpos0 + r / g : sq.n_keys - 1;
                const float x = (key < sq.n_keys && key <= qpos) ? v[j] : -INFINITY;
                float tm = x;
#pragma unroll
                for (int off = 4; off <= 16; off <<= 1) tm = fmaxf(tm, __shfl_xor_sync(0xffffffffu, tm, off));
                const float m_new = fmaxf(m_run[j], tm);
                float pj = 0.f;
                alpha[j] = 1.f;
                if (m_new != -INFINITY) {
                    alpha[j] = ex2(m_run[j] - m_new);
                    pj = ex2(x - m_new);
                }
                float sum = pj;
#pragma unroll
                for (int off = 4; off <= 16; off <<= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
                m_run[j] = m_new;
                l_run[j] = alpha[j] * l_run[j] + sum;
                s_pw[kl * RB + r] = pj;
                if (kl == 0) s_pw[8 * RB + r] = alpha[j];
            }
            __syncwarp();

            // 3. O = alpha O + P V over the warp's 8 keys
#pragma unroll
            for (int r4 = 0; r4 < RB / 4; ++r4) {
                const float4 a4 = *reinterpret_cast<const float4 *>(s_pw + 8 * RB + 4 * r4);
                const float al[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
                for (int h = 0; h < 4; ++h)
#pragma unroll
                    for (int c = 0; c < CW / 2; ++c)
                        acc[4 * r4 + h][c] = make_float2(acc[4 * r4 + h][c].x * al[h], acc[4 * r4 + h][c].y * al[h]);
            }
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                const int k = warp * 8 + kk;
                float2 vf[CW / 2];
                if constexpr (CW == 4) {
                    // lane: columns 4l..4l+3 = half (l & 1) of chunk ((l & 15) >> 1) in region (l >> 4)
                    const uint8_t *row = Vs + (lane >> 4) * C::kRegionBytes + k * 128;
                    const uint2 u =
                        *reinterpret_cast<const uint2 *>(row + ((((lane & 15) >> 1) ^ (k & 7)) << 4) + (lane & 1) * 8);
                    vf[0] = make_float2(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u));
                    vf[1] = make_float2(__uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
                } else {
                    // lane: columns 2l, 2l+1 = quarter (l & 3) of chunk (l >> 2)
                    const uint8_t *row = Vs + k * 128;
                    const uint32_t u =
                        *reinterpret_cast<const uint32_t *>(row + (((lane >> 2) ^ (k & 7)) << 4) + (lane & 3) * 4);
                    vf[0] = make_float2(__uint_as_float(u << 16), __uint_as_float(u & 0xffff0000u));
                }
                const float4 *pk = reinterpret_cast<const float4 *>(s_pw + kk * RB);
#pragma unroll
                for (int r4 = 0; r4 < RB / 4; ++r4) {
                    const float4 w = pk[r4];
                    const float wr[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                    for (int h = 0; h < 4; ++h)
#pragma unroll
                        for (int c = 0; c < CW / 2; ++c)
                            acc[4 * r4 + h][c] = fma2(make_float2(wr[h], wr[h]), vf[c], acc[4 * r4 + h][c]);
                }
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(empty(s));
        }

        // ---------------------------------------------------------- epilogue
        // merge the 8 warps: O = sum_w 2^(m_w - M) O_w, l = sum_w 2^(m_w - M) l_w
        const bool stopped = ptx::bar_sync_or(kBarConsumers, kConsumers, *abort_flag != 0);  // stages are free
        float *red = reinterpret_cast<float *>(smem);  // [8][RB][HD]
        if (kl == 0) {
#pragma unroll
            for (int j = 0; j < RPL; ++j) {
                s_ml[warp * RB + row0 + j] = m_run[j];
                s_ml[kDecWarps * RB + warp * RB + row0 + j] = l_run[j];
            }
        }
#pragma unroll
        for (int r = 0; r < RB; ++r) {
            float *dst = red + (warp * RB + r) * HD + lane * CW;
            if constexpr (CW == 4) {
                *reinterpret_cast<float4 *>(dst) = make_float4(acc[r][0].x, acc[r][0].y, acc[r][1].x, acc[r][1].y);
            } else {
                *reinterpret_cast<float2 *>(dst) = acc[r][0];
            }
        }
        ptx::bar_sync(kBarConsumers, kConsumers);
        const bool single = sq.n_splits == 1;
        float *po = nullptr, *pm = nullptr, *pl = nullptr;
        if (!single) {
            po = p.part + static_cast<int64_t>(blockIdx.x) * RB * HD;
            pm = p.part + static_cast<int64_t>(p.total_ctas) * RB * HD;
            pl = pm + static_cast<int64_t>(p.total_ctas) * RB;
        }
        for (int e = threadIdx.x; e < RB * HD / 2; e += kConsumers) {
            const int r = (2 * e) / HD;
            const int col = (2 * e) % HD;
            float mx = -INFINITY;
#pragma unroll
            for (int w = 0; w < kDecWarps; ++w) mx = fmaxf(mx, s_ml[w * RB + r]);
            float o0 = 0.f, o1 = 0.f, den = 0.f;
            if (mx != -INFINITY) {
#pragma unroll
                for (int w = 0; w < kDecWarps; ++w) {
                    const float mw = s_ml[w * RB + r];
                    if (mw == -INFINITY) continue;
                    const float wgt = ex2(mw - mx);
                    const float2 x = *reinterpret_cast<const float2 *>(red + (w * RB + r) * HD + col);
                    o0 += wgt * x.x;
                    o1 += wgt * x.y;
                    den += wgt * s_ml[kDecWarps * RB + w * RB + r];
                }
            }
            if (single) {
                if (r < n_rows && !stopped) {
                    const float inv = den > 0.f ? 1.0f / den : 0.f;
                    __nv_bfloat16 *dst = static_cast<__nv_bfloat16 *>(p.out) +
                                         (static_cast<int64_t>(sq.q_row0 + r / g) * p.hq + kvh * g + r % g) * HD + col;
                    *reinterpret_cast<uint32_t *>(dst) = pack_bf16(o0 * inv, o1 * inv);
                }
            } else {
                *reinterpret_cast<float2 *>(po + r * HD + col) = make_float2(o0, o1);
                if (col == 0) {
                    pm[static_cast<int64_t>(blockIdx.x) * RB + r] = mx;
                    pl[static_cast<int64_t>(blockIdx.x) * RB + r] = den;
                }
            }
        }
        if (!single) split_merge<RB, HD>(p, sq, si, kvh, n_rows, threadIdx.x, kConsumers, kBarConsumers, s_ticket);
    }

    __syncthreads();
    // After an abort, copies may still be in flight: wait (bounded) for the
    // last tile issued on every stage before the CTA's shared memory goes away.
    if (threadIdx.x == 0 && *abort_flag) {
        const int issued = *s_issued;
        const uint64_t start = ptx::globaltimer();
        for (int i = max(0, issued - kDecStages); i < issued; ++i)
            while (!ptx::mbar_try_wait(full(i % kDecStages), (i / kDecStages) & 1) &&
                   ptx::globaltimer() - start < 4000000ull) {
            }
    }
}

// ============================================================================
// Tensor-core form (d = 128 and d = 64).  With keys on the M side of the MMA
// the few query rows become N = 16 (rows padded):
//     S^T [128 keys x 16] = K [128 x d] . Q^T          (A = K tile, B = Q; K-major)
//     O^T [d x 16]       += V^T [d x 128 keys] . P^T   (A = V tile, MN-major; B = P^T, K-major)
// both accumulated in TMEM (lane = key for S^T, lane = d-column for O^T), so a
// softmax thread owns one key and touches only its RB valid row values per
// 128-key tile.  For d = 64 the O^T GEMM keeps M = 128: the A operand's second
// 64-row half (d-columns 64..127) is a zero-filled shared-memory region beside
// each V stage, so O^T rows 64..127 stay zero and only the first 64 are read.
//
// Persistent, dynamically scheduled: every (sequence, kv-head) item's 128-key
// tiles are cut into chunks of at most 8 tiles (the host picks about three
// chunks per SM); one CTA per SM takes chunk after chunk from a global
// counter, so a slower SM simply takes fewer.  Chunks are numbered longest
// first (every full chunk, then the items' shorter remainders by decreasing
// length), so the chunks taken last are the short ones and the CTAs finish
// close together.  A chunk that is a whole item is written directly; otherwise
// each chunk writes a partial (O, m, l) and a combine launch that follows
// (programmatic serialization, so its launch overlaps this grid's end) merges
// an item's partials in the item's chunk order.  The last CTA to stop taking chunks resets the
// chunk counter for the next launch.
//
// Roles (384 threads):
//   warps 0-3  softmax: thread t = key t of the tile (TMEM lane t); masks,
//              exp2 against a per-row reference, P^T (bf16) to shared memory,
//              per-thread partial row sums; per chunk, the row statistics
//              (m, l) for the epilogue.
//   warps 7-10 epilogue: thread = d-column (TMEM lane); per chunk, reads O^T
//              (double-buffered in TMEM, so the next chunk accumulates into
//              the other buffer meanwhile), writes the output or the chunk's
//              partial.
//   warp 11    scheduler + page-id loader: takes chunk ids (one chunk ahead of
//              the producers) into a ring that the MMA issuer and the softmax
//              warps read, turns each chunk's page ids into TMA row
//              coordinates in a descriptor ring for the producers, and stages
//              each chunk's Q rows (double-buffered), so that no role on the
//              streaming path ever waits on a global load.
//   warp 4     K producer: issues TMA boxes of K into a ring of 128-key tiles,
//              a stage freeing as soon as its S^T MMA completes.
//   warp 6     V producer: the same for V (a V stage is held until
//              O^T += V^T P^T, after the tile's softmax).
//   warp 5     MMA: TMEM allocation; one thread issues each S^T and each
//              O^T += V^T P^T as soon as its operands are in place (S^T up to
//              two tiles ahead), so loads, softmax and MMAs overlap.
// The row reference m is a chunk's first tile max (log2 units) and only moves
// when a tile's weight would pass 2^64 (or a row saw no key yet); then the
// tile max is taken and O^T and the partial sums are rescaled in place.
constexpr int kTcKeys = 128;
constexpr int kTcKStages = 3;                      // K ring (32 KB stages)
constexpr int kTcVStages = 3;                      // V ring
constexpr int kTcThreads = 384;
constexpr int kChunkRing = 4;                      // chunk ids in flight between the roles
constexpr int kDescRing = 2;                       // chunk descriptors (TMA rows) for the producers
constexpr int kDescInts = 8 + 8 * 16;              // header, then the row of box (tile k, slot j) at 8 + 16 k + j
constexpr int kBarSoftmax = 2;                     // named barrier of the softmax warps
constexpr float kTcWeightLimit = 1.8446744e19f;    // 2^64

template <int HD, int RB>
struct TcCfg {
    static constexpr int kRegs = HD / 64;                   // 64-column halves of a K, V or Q row
    static constexpr int kRegionBytes = kTcKeys * 128;      // 128 keys x 64 columns (bf16), 128-byte swizzle
    static constexpr int kTileBytes = 2 * kRegionBytes;     // one K or V stage (d = 64: V's second half is zeros)
    static constexpr int kLoadBytes = kTcKeys * HD * 2;     // bytes the TMA boxes of one tile deliver
    static constexpr int kOffV = kTcKStages * kTileBytes;   // K ring, then V ring
    static constexpr int kOffQ = (kTcKStages + kTcVStages) * kTileBytes;  // Q x2: [16 rows][128] bf16, 2 x 2 KB each
    static constexpr int kOffP = kOffQ + 2 * 4096;          // P^T x2: [16 rows][128 keys] bf16, 2 regions x 2 KB each
    static constexpr int kOffRed = kOffP + 2 * 4096;        // float [4 warps][16]
    static constexpr int kOffBar = kOffRed + 4 * 16 * 4;
    // k_full[KS], k_empty[KS], v_full[VS], v_empty[VS], s_full[2], p_full[2], o_done[2], q_ready[2], drain,
    // ch_full[R], ch_empty[R], o_item[2], o_free[2], stats[2], desc_full[D], desc_empty[D], q_free[2]
    static constexpr int kNumBars = 2 * (kTcKStages + kTcVStages) + 9 + 2 * kChunkRing + 8 + 2 * kDescRing;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;  // tmem slot, abort, K / V tiles issued, chunk ring
    static constexpr int kOffStats = kOffMisc + 32 + 4 * kChunkRing;  // [2][id, m[RB], l[RB]] per chunk parity
    static constexpr int kStatsFloats = 1 + 2 * RB;
    static constexpr int kOffSeqs = kOffStats + 2 * kStatsFloats * 4;  // the launch's sequence table
    static constexpr int kOffDesc = kOffSeqs + kMaxSegs * static_cast<int>(sizeof(DecodeSeq) + 4);  // + rem_seq
    static constexpr int kSmem = kOffDesc + kDescRing * kDescInts * 4;
    static constexpr int kDynSmem = kSmem + 1024;
    static constexpr uint32_t kTmemCols = 64;               // S^T buffers at 0 and 16, O^T buffers at 32 and 48
    static_assert(kDynSmem <= 232448, "shared memory budget");
    static_assert(RB == 4 || RB == 8 || RB == 16, "row capacity");
    static_assert(HD == 64 || HD == 128, "head dim");
};

// A chunk: tiles [t0, t1) of item (sequence si, kv-head kvh).  An item has
// nfull full chunks (ids first .. first + nfull - 1) and, when its tile count
// is not a multiple of the chunk size, one shorter remainder chunk (id rem);
// cpi chunks in all.
struct ChunkInfo {
    int si, kvh, t0, t1, cpi, first, nfull, rem;
};

__device__ __forceinline__ int tc_tiles(const DecodeSeq &sq) { return (sq.n_keys + kTcKeys - 1) / kTcKeys; }

// seqs, rem_seq: shared-memory copies of the launch's sequence table and remainder order
__device__ __forceinline__ ChunkInfo tc_chunk(const DecodeParams &p, const DecodeSeq *seqs, const int32_t *rem_seq,
                                              int c)
{
    int si = 0;
    if (c < p.full_chunks) {
        // the last sequence whose first full chunk id (tile0, non-decreasing) is at most c: a sequence
        // without full chunks shares tile0 with the next one, which then wins
        int hi = p.n_seqs;
        while (hi - si > 1) {
            const int mid = (si + hi) >> 1;
            if (seqs[mid].tile0 <= c) si = mid;
            else hi = mid;
        }
    } else {
        si = rem_seq[(c - p.full_chunks) / p.hkv];
    }
    const DecodeSeq &sq = seqs[si];
    const int nt = tc_tiles(sq);
    const int ct = sq.cta0;  // tiles per full chunk
    ChunkInfo ci;
    ci.si = si;
    ci.nfull = nt / ct;
    if (c < p.full_chunks) {
        const int off = c - sq.tile0;
        ci.kvh = off / ci.nfull;
        ci.t0 = (off - ci.kvh * ci.nfull) * ct;
        ci.t1 = ci.t0 + ct;
    } else {
        ci.kvh = c - sq.rem0;
        ci.t0 = ci.nfull * ct;
        ci.t1 = nt;
    }
    ci.first = sq.tile0 + ci.kvh * ci.nfull;
    ci.rem = sq.rem0 >= 0 ? sq.rem0 + ci.kvh : -1;
    ci.cpi = ci.nfull + (sq.rem0 >= 0 ? 1 : 0);
    return ci;
}

template <int HD, int RB>
__global__ void __launch_bounds__(kTcThreads, 1)
    decode_tc_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                     const __grid_constant__ DecodeParams p)
{
    using C = TcCfg<HD, RB>;
    constexpr int R = kChunkRing;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int g = p.group;

    const uint32_t sbase = ptx::smem_addr(smem);
    const uint32_t q_smem = sbase + C::kOffQ;
    const uint32_t p_smem = sbase + C::kOffP;
    float *s_red = reinterpret_cast<float *>(smem + C::kOffRed);
    const uint32_t bar0 = sbase + C::kOffBar;
    auto k_full = [&](int s) { return bar0 + 8u * s; };
    auto k_empty = [&](int s) { return bar0 + 8u * (kTcKStages + s); };
    auto v_full = [&](int s) { return bar0 + 8u * (2 * kTcKStages + s); };
    auto v_empty = [&](int s) { return bar0 + 8u * (2 * kTcKStages + kTcVStages + s); };
    const uint32_t b_s_full = bar0 + 8u * (2 * (kTcKStages + kTcVStages));  // [2]
    const uint32_t b_p_full = b_s_full + 16;                     // [2]
    const uint32_t b_o_done = b_p_full + 16;                     // [2]
    const uint32_t b_q_ready = b_o_done + 16;                    // [2]
    const uint32_t b_drain = b_q_ready + 16;
    const uint32_t b_ch_full = b_drain + 8;                      // [R]
    const uint32_t b_ch_empty = b_ch_full + 8 * R;               // [R]
    const uint32_t b_o_item = b_ch_empty + 8 * R;                // [2] a chunk's O^T is complete
    const uint32_t b_o_free = b_o_item + 16;                     // [2] the epilogue has read that O^T buffer
    const uint32_t b_stats = b_o_free + 16;                      // [2] a chunk's id, m and l are in s_stats
    const uint32_t b_desc_full = b_stats + 16;                   // [D] a chunk's TMA rows are in s_desc
    const uint32_t b_desc_empty = b_desc_full + 8 * kDescRing;   // [D] both producers have issued that chunk
    const uint32_t b_q_free = b_desc_empty + 8 * kDescRing;      // [2] every S^T reading that Q buffer is done
    float *s_stats = reinterpret_cast<float *>(smem + C::kOffStats);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + C::kOffMisc);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + C::kOffMisc + 4);
    volatile int *s_issued = reinterpret_cast<volatile int *>(smem + C::kOffMisc + 12);  // [2]: K, V
    volatile int *s_chunk = reinterpret_cast<volatile int *>(smem + C::kOffMisc + 32);  // [R]
    DecodeSeq *s_seqs = reinterpret_cast<DecodeSeq *>(smem + C::kOffSeqs);
    int32_t *s_rem_seq = reinterpret_cast<int32_t *>(smem + C::kOffSeqs + kMaxSegs * sizeof(DecodeSeq));
    int *s_desc = reinterpret_cast<int *>(smem + C::kOffDesc);  // [D][kDescInts]
    const WaitCtx wctx{abort_flag, p.status};

    // reads chunk ordinal n from the ring (every reader arrives once); -1 = no more chunks
    auto read_chunk = [&](int n) -> int {
        if (!wait_bar(b_ch_full + 8 * (n % R), (n / R) & 1, wctx)) return -1;
        return s_chunk[n % R];
    };
    if (threadIdx.x == 128) {  // K producer warp, lane 0
        for (int s = 0; s < kTcKStages; ++s) {
            ptx::mbar_init(k_full(s), 1);
            ptx::mbar_init(k_empty(s), 1);
        }
        for (int s = 0; s < kTcVStages; ++s) {
            ptx::mbar_init(v_full(s), 1);
            ptx::mbar_init(v_empty(s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(b_s_full + 8 * b, 1);
            ptx::mbar_init(b_p_full + 8 * b, 128);
            ptx::mbar_init(b_o_done + 8 * b, 1);
            ptx::mbar_init(b_q_ready + 8 * b, 1);
            ptx::mbar_init(b_q_free + 8 * b, 1);
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(b_o_item + 8 * b, 1);
            ptx::mbar_init(b_o_free + 8 * b, 128);
            ptx::mbar_init(b_stats + 8 * b, 1);
        }
        ptx::mbar_init(b_drain, 1);
        for (int r = 0; r < R; ++r) {
            ptx::mbar_init(b_ch_full + 8 * r, 1);
            ptx::mbar_init(b_ch_empty + 8 * r, 1 + 128);  // MMA, softmax threads
        }
        for (int d = 0; d < kDescRing; ++d) {
            ptx::mbar_init(b_desc_full + 8 * d, 1);
            ptx::mbar_init(b_desc_empty + 8 * d, 2);      // K and V producers
        }
        *abort_flag = 0;
        s_issued[0] = 0;
        s_issued[1] = 0;
        ptx::fence_barrier_init();
        ptx::prefetch_tensormap(&tm_k);
        ptx::prefetch_tensormap(&tm_v);
    }
    if (warp == 5) {
        ptx::tmem_alloc(ptx::smem_addr(tmem_slot), C::kTmemCols);
        ptx::tmem_relinquish();
    }
    if (warp < 4) {
        // both P^T buffers start at zero (rows past RB stay zero)
        for (int e = threadIdx.x; e < 2 * 4096 / 16; e += 128)
            reinterpret_cast<uint4 *>(smem + C::kOffP)[e] = make_uint4(0u, 0u, 0u, 0u);
        if (HD == 64) {  // the zero second half of every V stage (d-columns 64..127 of the O^T GEMM's A)
            for (int s = 0; s < kTcVStages; ++s)
                for (int e = threadIdx.x; e < C::kRegionBytes / 16; e += 128)
                    reinterpret_cast<uint4 *>(smem + C::kOffV + s * C::kTileBytes + C::kRegionBytes)[e] =
                        make_uint4(0u, 0u, 0u, 0u);
        }
        ptx::fence_proxy_async_smem();
    } else if (warp >= 7) {
        // the sequence table and the remainder order, read at every chunk by every role
        constexpr int kWords = static_cast<int>(sizeof(DecodeSeq) / 4);
        const int n_words = p.n_seqs * kWords;
        const int32_t *src = reinterpret_cast<const int32_t *>(p.seqs);
        for (int e = threadIdx.x - 224; e < n_words + p.n_seqs; e += kTcThreads - 224) {
            if (e < n_words) reinterpret_cast<int32_t *>(s_seqs)[e] = src[e];
            else s_rem_seq[e - n_words] = p.rem_seq[e - n_words];
        }
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    // Launched with programmatic serialization: the set-up above overlapped the previous kernel (the
    // append of the new positions); nothing written by earlier kernels is read before this point.
    ptx::griddep_wait();
    const uint32_t tmem = *tmem_slot;
    const uint32_t t_s = tmem;         // S^T buffers: columns 0 and 16
    const uint32_t t_o = tmem + 32;    // O^T buffers: columns 32..47 (even chunks) and 48..63 (odd)

    if (warp == 4 || warp == 6) {
        // ============================================================ producers (warp 4: K, warp 6: V)
        // Each chunk's TMA rows come ready from the loader warp; lane kRegs j + h issues box j (keys
        // [j kpc, (j + 1) kpc) of the tile) of 64-column half h.
        const bool is_v = warp == 6;
        const CUtensorMap *map = is_v ? &tm_v : &tm_k;
        const int n_stages = is_v ? kTcVStages : kTcKStages;
        const int kpc = p.ps < kDecKeys ? p.ps : kDecKeys;  // keys per box (<= 64)
        const int n_ops = (kTcKeys / kpc) * C::kRegs;       // boxes per tile, <= 32
        const int op_slot = lane / C::kRegs;
        const int op_reg = lane % C::kRegs;
        const bool op_on = lane < n_ops;
        int i = 0;  // tile ordinal in this CTA
        for (int n = 0;; ++n) {
            const int d = n % kDescRing;
            if (!wait_bar_warp(b_desc_full + 8 * d, (n / kDescRing) & 1, wctx)) break;
            const int *desc = s_desc + d * kDescInts;
            if (desc[0] < 0) break;  // no more chunks
            const int nt = desc[1];
            bool ok = true;
            for (int k = 0; k < nt; ++k) {
                const int s = i % n_stages;
                const uint32_t b_empty = is_v ? v_empty(s) : k_empty(s);
                const uint32_t b_full = is_v ? v_full(s) : k_full(s);
                if (i >= n_stages && !wait_bar_warp(b_empty, ((i / n_stages) - 1) & 1, wctx)) {
                    ok = false;
                    break;
                }
                if (lane == 0) ptx::mbar_arrive_expect_tx(b_full, C::kLoadBytes);
                __syncwarp();
                if (op_on) {
                    const uint32_t dst = sbase + (is_v ? C::kOffV : 0) + s * C::kTileBytes +
                                         op_reg * C::kRegionBytes + op_slot * kpc * 128;
                    ptx::tma_load_2d(dst, map, op_reg * 64, desc[8 + 16 * k + op_slot], b_full);
                }
                __syncwarp();
                ++i;
                if (lane == 0) s_issued[is_v ? 1 : 0] = i;
            }
            if (!ok) break;
            if (lane == 0) ptx::mbar_arrive(b_desc_empty + 8 * d);  // the descriptor slot may be refilled
        }
    } else if (warp == 11) {
        // ============================================================ scheduler + page-id loader
        // Takes the chunk ids (the first two fixed: CTA b takes b and N + b; later ones from the
        // launch's counter), publishes them to the MMA issuer and the softmax warps, and turns each
        // chunk's page ids into the producers' TMA rows.  Ordinal n is taken once the producers are
        // done with ordinal n - kDescRing, so a CTA holds at most kDescRing - 1 chunks it has not
        // started; the page-id loads wait here, not in the producers.
        const int kpc = p.ps < kDecKeys ? p.ps : kDecKeys;
        const int n_slots = kTcKeys / kpc;  // boxes per 64-column half, <= 16
        constexpr int kMaxCT = 8;           // the host keeps chunks at most 8 tiles
        for (int n = 0;; ++n) {
            const int d = n % kDescRing;
            const bool ok = n < kDescRing || wait_bar_warp(b_desc_empty + 8 * d, ((n / kDescRing) - 1) & 1, wctx);
            int c = -1;
            if (ok && lane == 0) {
                c = n < 2 ? n * static_cast<int>(gridDim.x) + static_cast<int>(blockIdx.x)
                          : 2 * static_cast<int>(gridDim.x) + atomicAdd(p.sched, 1);
                if (c >= p.total_tiles) c = -1;  // total_tiles: the launch's chunk count
            }
            c = __shfl_sync(0xffffffffu, c, 0);
            if (lane == 0) {
                if (n >= R) (void)wait_bar(b_ch_empty + 8 * (n % R), ((n / R) - 1) & 1, wctx);
                s_chunk[n % R] = c;
                ptx::mbar_arrive(b_ch_full + 8 * (n % R));  // release: the MMA issuer and softmax read the id
            }
            int *desc = s_desc + d * kDescInts;
            if (c >= 0) {
                const ChunkInfo ci = tc_chunk(p, s_seqs, s_rem_seq, c);
                const DecodeSeq &sq = s_seqs[ci.si];
                constexpr int kPer = kMaxCT * 16 / 32;
                int pg[kPer];
                bool in[kPer];
#pragma unroll
                for (int u = 0; u < kPer; ++u) {  // entry e = 32 u + lane: tile e / 16, box e % 16
                    const int e = 32 * u + lane;
                    const int key0 = (ci.t0 + (e >> 4)) * kTcKeys + (e & 15) * kpc;
                    in[u] = ci.t0 + (e >> 4) < ci.t1 && (e & 15) < n_slots && key0 < sq.n_keys;
                    pg[u] = in[u] ? p.page_table[sq.table_row + key0 / p.ps] : -1;
                }
#pragma unroll
                for (int u = 0; u < kPer; ++u) {
                    const int e = 32 * u + lane;
                    const int key0 = (ci.t0 + (e >> 4)) * kTcKeys + (e & 15) * kpc;
                    const bool ok_page = pg[u] >= 0 && pg[u] < p.num_pages;
                    if (!ok_page && in[u]) atomicCAS(p.status, 0, kStatusBadPage);
                    desc[8 + e] = ok_page ? ((p.layer * p.num_pages + pg[u]) * p.hkv + ci.kvh) * p.ps + key0 % p.ps
                                          : p.oob_row;  // past the sequence (or a bad id): zeros
                }
                if (lane == 0) {
                    desc[0] = c;
                    desc[1] = ci.t1 - ci.t0;
                }
            } else if (lane == 0) {
                desc[0] = -1;
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(b_desc_full + 8 * d);  // release: the producers read the rows
            if (c < 0) break;
            // the chunk's Q rows into buffer n & 1 as [16 rows][d] bf16 (128-byte swizzle, 64-column
            // halves 2 KB apart), rows past n_q x g zero; the buffer's previous chunk (n - 2) must be
            // done with it
            {
                const ChunkInfo ci = tc_chunk(p, s_seqs, s_rem_seq, c);
                const DecodeSeq &sq = s_seqs[ci.si];
                const int n_rows = sq.n_q * g;
                constexpr int kCols = HD / 8;     // 16-byte columns of a row
                constexpr int kQj = 16 * kCols / 32;
                uint4 qv[kQj];
#pragma unroll
                for (int j = 0; j < kQj; ++j) {  // piece e = 32 j + lane: row e / kCols, 16-byte column e % kCols
                    const int e = 32 * j + lane;
                    const int r = e / kCols;
                    qv[j] = make_uint4(0u, 0u, 0u, 0u);
                    if (r < n_rows)
                        qv[j] = *reinterpret_cast<const uint4 *>(
                            static_cast<const __nv_bfloat16 *>(p.q) +
                            (static_cast<int64_t>(sq.q_row0 + r / g) * p.hq + ci.kvh * g + r % g) * HD +
                            (e % kCols) * 8);
                }
                if (n >= 2 && !wait_bar_warp(b_q_free + 8 * (n & 1), ((n - 2) >> 1) & 1, wctx)) break;
#pragma unroll
                for (int j = 0; j < kQj; ++j) {
                    const int e = 32 * j + lane;
                    const int r = e / kCols;
                    const int cc = e % kCols;
                    *reinterpret_cast<uint4 *>(smem + C::kOffQ + (n & 1) * 4096 + (cc >> 3) * 2048 + r * 128 +
                                               (((cc & 7) ^ (r & 7)) << 4)) = qv[j];
                }
                ptx::fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(b_q_ready + 8 * (n & 1));  // release: S^T of chunk n may read it
            }
        }
        // this CTA takes no more ids: the last loader to stop resets the counter for the next launch
        // (every other CTA has made its last atomicAdd on it by then)
        if (lane == 0) {
            __threadfence();
            if (atomicAdd(p.sched + 1, 1) == static_cast<int>(gridDim.x) - 1) {
                p.sched[0] = 0;
                p.sched[1] = 0;
                __threadfence();
            }
        }
    } else if (warp == 5) {
        // ============================================================ MMA issuer
        if (lane == 0) {
            constexpr uint32_t kIdS = ptx::idesc_bf16_f32(128, 16, false, false);
            constexpr uint32_t kIdPV = ptx::idesc_bf16_f32(128, 16, false, true);
            // S^T cursor: chunk ordinal ns_chunk, tile k_s within it; P V cursor: tiles left in its chunk
            int ns = 0, np = 0;                    // next S^T tile, next P V tile (ordinals in this CTA)
            int ns_chunk = 0;                      // chunk ordinal of tile ns
            int s_left = 0;                        // tiles of chunk ns_chunk not yet given an S^T
            int pv_tiles[4] = {0, 0, 0, 0};        // tile counts of chunks the S^T cursor has read
            int np_chunk = 0, p_done = 0;          // P V cursor: chunk ordinal, tiles done in it
            bool more = true;                      // the S^T cursor may read another chunk
            int c0 = read_chunk(0);
            if (c0 >= 0) {
                const ChunkInfo ci = tc_chunk(p, s_seqs, s_rem_seq, c0);
                s_left = ci.t1 - ci.t0;
                pv_tiles[0] = s_left;
            } else {
                more = false;
            }
            ptx::mbar_arrive(b_ch_empty);
            uint64_t t_last = ptx::globaltimer();
            while (s_left > 0 || np < ns) {
                bool progress = false;
                // S^T(ns): K landed, S buffer free (P V(ns - 2) issued), Q of its chunk ready
                if (s_left > 0 && ns <= np + 1) {
                    const int s = ns % kTcKStages;
                    const int tile_in = pv_tiles[ns_chunk & 3] - s_left;
                    if ((tile_in > 0 || ptx::mbar_test_wait(b_q_ready + 8 * (ns_chunk & 1), (ns_chunk >> 1) & 1)) &&
                        ptx::mbar_test_wait(k_full(s), (ns / kTcKStages) & 1)) {
                        ptx::tc_fence_after();
                        const uint32_t ka = sbase + s * C::kTileBytes;
                        const uint32_t qa = q_smem + (ns_chunk & 1) * 4096;
#pragma unroll
                        for (int kk = 0; kk < HD / 16; ++kk) {
                            const uint32_t off = (kk >> 2) * C::kRegionBytes + (kk & 3) * 32;
                            const uint32_t qoff = (kk >> 2) * 2048 + (kk & 3) * 32;
                            ptx::mma_bf16(t_s + 16 * (ns & 1), ptx::smem_desc_sw128(ka + off, 16, 1024),
                                          ptx::smem_desc_sw128(qa + qoff, 16, 1024), kIdS, kk > 0 ? 1u : 0u);
                        }
                        ptx::mma_commit(b_s_full + 8 * (ns & 1));
                        ptx::mma_commit(k_empty(s));  // the K stage is free once S^T(ns) is done
                        if (s_left == 1) ptx::mma_commit(b_q_free + 8 * (ns_chunk & 1));  // the chunk's last S^T
                        ++ns;
                        if (--s_left == 0 && more) {
                            // next chunk (the ring entry is read once, then released)
                            const int c = read_chunk(ns_chunk + 1);
                            ptx::mbar_arrive(b_ch_empty + 8 * ((ns_chunk + 1) % R));
                            if (c >= 0) {
                                ++ns_chunk;
                                const ChunkInfo ci = tc_chunk(p, s_seqs, s_rem_seq, c);
                                s_left = ci.t1 - ci.t0;
                                pv_tiles[ns_chunk & 3] = s_left;
                            } else {
                                more = false;
                            }
                        }
                        progress = true;
                    }
                }
                // O^T += V^T P^T(np): V landed, P^T(np) written, and at a chunk's first tile the epilogue
                // has read the O^T buffer's previous chunk
                if (np < ns && ptx::mbar_test_wait(v_full(np % kTcVStages), (np / kTcVStages) & 1) &&
                    ptx::mbar_test_wait(b_p_full + 8 * (np & 1), (np >> 1) & 1) &&
                    (p_done > 0 || np_chunk < 2 ||
                     ptx::mbar_test_wait(b_o_free + 8 * (np_chunk & 1), ((np_chunk - 2) >> 1) & 1))) {
                    ptx::tc_fence_after();
                    const uint32_t vb = sbase + C::kOffV + (np % kTcVStages) * C::kTileBytes;
                    const uint32_t pb = p_smem + (np & 1) * 4096;
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        ptx::mma_bf16(t_o + 16 * (np_chunk & 1),
                                      ptx::smem_desc_sw128(vb + kk * 16 * 128, C::kRegionBytes, 1024),
                                      ptx::smem_desc_sw128(pb + (kk >> 2) * 2048 + (kk & 3) * 32, 16, 1024), kIdPV,
                                      (p_done > 0 || kk > 0) ? 1u : 0u);
                    }
                    ptx::mma_commit(v_empty(np % kTcVStages));
                    ptx::mma_commit(b_o_done + 8 * (np & 1));
                    ++np;
                    if (++p_done == pv_tiles[np_chunk & 3]) {
                        ptx::mma_commit(b_o_item + 8 * (np_chunk & 1));  // the chunk's O^T is complete
                        ++np_chunk;
                        p_done = 0;
                    }
                    progress = true;
                }
                if (progress) {
                    t_last = ptx::globaltimer();
                } else {
                    if (*abort_flag) break;
                    if (ptx::globaltimer() - t_last > kWaitNs) {  // bounded: give up, record, let every role leave
                        *abort_flag = 1;
                        atomicCAS(p.status, 0, kStatusWaitTimeout);
                        break;
                    }
                }
            }
        }
        // every tcgen05 op of this CTA completes before TMEM is released
        if (lane == 0) {
            ptx::mma_commit(b_drain);
            const uint64_t start = ptx::globaltimer();
            while (!ptx::mbar_try_wait(b_drain, 0) && ptx::globaltimer() - start < 4000000ull) {
            }
        }
        __syncwarp();
    } else if (warp < 4) {
        // ============================================================ softmax (thread = key of the tile)
        const int t = threadIdx.x;              // TMEM lane
        const uint32_t lane_off = static_cast<uint32_t>(warp * 32) << 16;
        float mref[RB], lpart[RB];
        auto tile_max = [&](const float (&x)[RB], float (&m)[RB]) {
#pragma unroll
            for (int r = 0; r < RB; ++r) {
                float v = x[r];
#pragma unroll
                for (int off = 16; off >= 1; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
                if (lane == 0) s_red[warp * 16 + r] = v;
            }
            ptx::bar_sync(kBarSoftmax, 128);
#pragma unroll
            for (int r = 0; r < RB; ++r)
                m[r] = fmaxf(fmaxf(s_red[r], s_red[16 + r]), fmaxf(s_red[32 + r], s_red[48 + r]));
            ptx::bar_sync(kBarSoftmax, 128);  // s_red is reused
        };
        int c_cur = read_chunk(0);
        ptx::mbar_arrive(b_ch_empty);
        ChunkInfo ci{};
        if (c_cur >= 0) ci = tc_chunk(p, s_seqs, s_rem_seq, c_cur);
        int n = 0;   // chunk ordinal
        int i = 0;   // tile ordinal in this CTA
        bool stopped = false;
        while (c_cur >= 0 && !stopped) {
            const DecodeSeq &sq = s_seqs[ci.si];
            const int n_rows = sq.n_q * g;
            const int qpos0 = sq.n_keys - sq.n_q;
            // the next chunk's id
            const int c_next = read_chunk(n + 1);
            ptx::mbar_arrive(b_ch_empty + 8 * ((n + 1) % R));
            ChunkInfo cn{};
            if (c_next >= 0) cn = tc_chunk(p, s_seqs, s_rem_seq, c_next);
#pragma unroll
            for (int r = 0; r < RB; ++r) {
                mref[r] = -INFINITY;
                lpart[r] = 0.f;
            }
            for (int lt = ci.t0; lt < ci.t1; ++lt, ++i) {
                const int j = lt - ci.t0;
                const bool ok = wait_bar_warp(b_s_full + 8 * (i & 1), (i >> 1) & 1, wctx);
                if (ptx::bar_sync_or(kBarSoftmax, 128, !ok || *abort_flag)) {
                    stopped = true;
                    break;
                }
                ptx::tc_fence_after();
                float x[RB];
                ptx::tmem_ld_n<RB>(t_s + 16 * (i & 1) + lane_off, x);
                ptx::tmem_wait_ld();
                const int key = lt * kTcKeys + t;
#pragma unroll
                for (int r = 0; r < RB; ++r) {
                    const int qpos = r < n_rows ? qpos0 + r / g : sq.n_keys - 1;
                    x[r] = (key < sq.n_keys && key <= qpos) ? x[r] * p.scale_log2 : -INFINITY;
                }
                if (j == 0) tile_max(x, mref);
                float pr[RB];
                bool big = false;
#pragma unroll
                for (int r = 0; r < RB; ++r) {
                    pr[r] = mref[r] == -INFINITY ? (x[r] == -INFINITY ? 0.f : INFINITY) : ex2(x[r] - mref[r]);
                    big = big || !(pr[r] <= kTcWeightLimit);
                }
                if (ptx::bar_sync_or(kBarSoftmax, 128, big)) {
                    // rare: move the reference to the running max, rescale O^T and the partial sums
                    float tm[RB], f[RB];
                    tile_max(x, tm);
#pragma unroll
                    for (int r = 0; r < RB; ++r) {
                        const float mn = fmaxf(mref[r], tm[r]);
                        f[r] = mn == -INFINITY ? 1.f : ex2(mref[r] - mn);
                        mref[r] = mn;
                        lpart[r] *= f[r];
                        pr[r] = mn == -INFINITY ? 0.f : ex2(x[r] - mn);
                    }
                    if (j > 0) {  // every earlier O^T update of this chunk has landed
                        const bool done = wait_bar_warp(b_o_done + 8 * ((i - 1) & 1), ((i - 1) >> 1) & 1, wctx);
                        if (done) {
                            ptx::tc_fence_after();
                            float o[RB];
                            ptx::tmem_ld_n<RB>(t_o + 16 * (n & 1) + lane_off, o);
                            ptx::tmem_wait_ld();
#pragma unroll
                            for (int r = 0; r < RB; ++r) o[r] *= f[r];
                            ptx::tmem_st_n<RB>(t_o + 16 * (n & 1) + lane_off, o);
                            ptx::tmem_wait_st();
                        }
                    }
                }
#pragma unroll
                for (int r = 0; r < RB; ++r) lpart[r] += pr[r];
                // P^T(i) into buffer i & 1 once O^T += V^T P^T(i - 2) has read it
                if (i >= 2) (void)wait_bar_warp(b_o_done + 8 * (i & 1), ((i - 2) >> 1) & 1, wctx);
                uint8_t *pt = smem + C::kOffP + (i & 1) * 4096 + (t >> 6) * 2048;
                const int chunk = (t & 63) >> 3;
#pragma unroll
                for (int r = 0; r < RB; ++r)
                    *reinterpret_cast<__nv_bfloat16 *>(pt + r * 128 + ((chunk ^ (r & 7)) << 4) + (t & 7) * 2) =
                        __float2bfloat16_rn(pr[r]);
                ptx::fence_proxy_async_smem();
                ptx::tc_fence_before();
                ptx::mbar_arrive(b_p_full + 8 * (i & 1));
            }
            if (stopped) break;

            // ---------------------------------------------------- row statistics for the epilogue warps
            float lsum[RB];
#pragma unroll
            for (int r = 0; r < RB; ++r) {
                float v = lpart[r];
#pragma unroll
                for (int off = 16; off >= 1; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
                if (lane == 0) s_red[warp * 16 + r] = v;
            }
            ptx::bar_sync(kBarSoftmax, 128);
#pragma unroll
            for (int r = 0; r < RB; ++r) lsum[r] = (s_red[r] + s_red[16 + r]) + (s_red[32 + r] + s_red[48 + r]);
            ptx::bar_sync(kBarSoftmax, 128);  // s_red is reused
            if (t == 0) {
                // the stats slot of chunk n - 2 must have been read
                if (n >= 2) (void)wait_bar(b_o_free + 8 * (n & 1), ((n - 2) >> 1) & 1, wctx);
                float *st = s_stats + (n & 1) * C::kStatsFloats;
                st[0] = __int_as_float(c_cur);
#pragma unroll
                for (int r = 0; r < RB; ++r) {
                    st[1 + r] = mref[r];
                    st[1 + RB + r] = lsum[r];
                }
                ptx::mbar_arrive(b_stats + 8 * (n & 1));  // release: the epilogue reads the slot
            }
            ci = cn;
            c_cur = c_next;
            ++n;
        }
        if (t == 0) {  // no more chunks: the epilogue warps stop at ordinal n
            if (n >= 2) (void)wait_bar(b_o_free + 8 * (n & 1), ((n - 2) >> 1) & 1, wctx);
            s_stats[(n & 1) * C::kStatsFloats] = __int_as_float(-1);
            ptx::mbar_arrive(b_stats + 8 * (n & 1));
        }
    } else if (warp >= 7 && warp < 11) {
        // ============================================================ epilogue (thread = d-column = TMEM lane)
        const int q4 = warp & 3;                       // TMEM lane quarter this warp may access
        const int t = q4 * 32 + lane;                  // d-column
        const int et = (warp - 7) * 32 + lane;         // thread index within the epilogue group
        const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
        for (int n = 0;; ++n) {
            if (!wait_bar_warp(b_stats + 8 * (n & 1), (n >> 1) & 1, wctx)) break;
            const float *st = s_stats + (n & 1) * C::kStatsFloats;
            const int c = __float_as_int(st[0]);
            if (c < 0) break;
            float o[RB], mref[RB], lsum[RB];
#pragma unroll
            for (int r = 0; r < RB; ++r) {
                mref[r] = st[1 + r];
                lsum[r] = st[1 + RB + r];
                o[r] = 0.f;
            }
            if (wait_bar_warp(b_o_item + 8 * (n & 1), (n >> 1) & 1, wctx)) {
                ptx::tc_fence_after();
                ptx::tmem_ld_n<RB>(t_o + 16 * (n & 1) + lane_off, o);
                ptx::tmem_wait_ld();
            }
            ptx::tc_fence_before();
            ptx::mbar_arrive(b_o_free + 8 * (n & 1));  // O^T buffer and stats slot may be reused
            const ChunkInfo ci = tc_chunk(p, s_seqs, s_rem_seq, c);
            const DecodeSeq &sq = s_seqs[ci.si];
            const int n_rows = sq.n_q * g;
            if (ci.cpi == 1) {
#pragma unroll
                for (int r = 0; r < RB; ++r) {
                    if (r < n_rows && t < HD) {  // d = 64: O^T rows 64..127 are the zero half
                        const float inv = lsum[r] > 0.f ? 1.0f / lsum[r] : 0.f;
                        static_cast<__nv_bfloat16 *>(p.out)[(static_cast<int64_t>(sq.q_row0 + r / g) * p.hq +
                                                             ci.kvh * g + r % g) * HD + t] = __float2bfloat16_rn(o[r] * inv);
                    }
                }
                continue;
            }
            // partial of chunk c (O / l unnormalised, with its reference m and sum l); the combine
            // launch that follows merges an item's partials
            float *po = p.part + static_cast<int64_t>(c) * RB * HD;
            float *pm = p.part + static_cast<int64_t>(p.total_tiles) * RB * HD;
            float *pl = pm + static_cast<int64_t>(p.total_tiles) * RB;
            if (t < HD) {
#pragma unroll
                for (int r = 0; r < RB; ++r) po[r * HD + t] = o[r];
            }
            if (et < RB) {
                float mv = -INFINITY, lv = 0.f;
#pragma unroll
                for (int r = 0; r < RB; ++r)
                    if (r == et) {
                        mv = mref[r];
                        lv = lsum[r];
                    }
                pm[static_cast<int64_t>(c) * RB + et] = mv;
                pl[static_cast<int64_t>(c) * RB + et] = lv;
            }
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0) {
        if (*abort_flag) {
            // after an abort, copies may still be in flight: bounded wait for the last ones issued
            const uint64_t start = ptx::globaltimer();
            for (int ring = 0; ring < 2; ++ring) {
                const int issued = s_issued[ring];
                const int n_stages = ring ? kTcVStages : kTcKStages;
                for (int i = max(0, issued - n_stages); i < issued; ++i) {
                    const uint32_t b = ring ? v_full(i % n_stages) : k_full(i % n_stages);
                    while (!ptx::mbar_try_wait(b, (i / n_stages) & 1) && ptx::globaltimer() - start < 4000000ull) {
                    }
                }
            }
        }
    }
    if (warp == 5) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, C::kTmemCols);
    }
}

// Merge of an item's chunk partials (one block per (sequence, kv-head), thread = d-column), after
// the decode kernel: M = max_k m_k, O = sum_k 2^(m_k - M) O_k / sum_k 2^(m_k - M) l_k over the item's
// chunks in its chunk order.  Items held in one chunk were written by the decode kernel itself.
template <int HD, int RB>
__global__ void __launch_bounds__(128) decode_tc_combine_kernel(const __grid_constant__ DecodeParams p)
{
    ptx::griddep_wait();  // launched with programmatic serialization: the decode kernel's partials
    if (static_cast<int>(threadIdx.x) >= HD) return;
    const int si = static_cast<int>(blockIdx.x) / p.hkv;
    const int kvh = static_cast<int>(blockIdx.x) - si * p.hkv;
    if (si >= p.n_seqs) return;
    const DecodeSeq &sq = p.seqs[si];
    const int nt = tc_tiles(sq);
    const int nfull = nt / sq.cta0;
    const int first = sq.tile0 + kvh * nfull;
    const int rem = sq.rem0 >= 0 ? sq.rem0 + kvh : -1;
    const int cpi = nfull + (rem >= 0 ? 1 : 0);
    if (cpi <= 1) return;
    const int g = p.group;
    const int n_rows = sq.n_q * g;
    const int t = static_cast<int>(threadIdx.x);
    const float *pm = p.part + static_cast<int64_t>(p.total_tiles) * RB * HD;
    const float *pl = pm + static_cast<int64_t>(p.total_tiles) * RB;
    // batches of kOB chunks, every load of a batch issued together (m and l are the same for
    // every thread: broadcast reads)
    constexpr int kOB = 32 / RB;
    float mx[RB], den[RB], acc[RB];
#pragma unroll
    for (int r = 0; r < RB; ++r) {
        mx[r] = -INFINITY;
        den[r] = 0.f;
        acc[r] = 0.f;
    }
    for (int k0 = 0; k0 < cpi; k0 += kOB) {
        float mv[kOB][RB], lv[kOB][RB], ov[kOB][RB];
#pragma unroll
        for (int u = 0; u < kOB; ++u) {
            const int k = k0 + u;
            const int64_t c = k < nfull ? first + k : rem;
#pragma unroll
            for (int r = 0; r < RB; ++r) {
                const bool in = k < cpi && r < n_rows;
                mv[u][r] = in ? __ldcg(pm + c * RB + r) : -INFINITY;
                lv[u][r] = in ? __ldcg(pl + c * RB + r) : 0.f;
                ov[u][r] = in ? __ldcg(p.part + (c * RB + r) * HD + t) : 0.f;
            }
        }
#pragma unroll
        for (int r = 0; r < RB; ++r) {
            float bmx = mx[r];
#pragma unroll
            for (int u = 0; u < kOB; ++u) bmx = fmaxf(bmx, mv[u][r]);
            const float f = (mx[r] == -INFINITY || bmx == -INFINITY) ? 0.f : ex2(mx[r] - bmx);
            den[r] *= f;
            acc[r] *= f;
            mx[r] = bmx;
#pragma unroll
            for (int u = 0; u < kOB; ++u) {
                const float w = (mv[u][r] == -INFINITY || bmx == -INFINITY) ? 0.f : ex2(mv[u][r] - bmx);
                den[r] += w * lv[u][r];
                acc[r] += w * ov[u][r];
            }
        }
    }
#pragma unroll
    for (int r = 0; r < RB; ++r) {
        if (r >= n_rows) continue;
        const float inv = den[r] > 0.f ? 1.0f / den[r] : 0.f;
        static_cast<__nv_bfloat16 *>(p.out)[(static_cast<int64_t>(sq.q_row0 + r / g) * p.hq + kvh * g + r % g) * HD +
                                            t] = __float2bfloat16_rn(acc[r] * inv);
    }
}

template <int HD, int RB>
cudaError_t launch_tc(const CUtensorMap &tm_k, const CUtensorMap &tm_v, const DecodeParams &p, cudaStream_t st)
{
    using C = TcCfg<HD, RB>;
    static std::atomic<uint64_t> configured{0};
    cudaError_t e = set_dyn_smem_once(decode_tc_kernel<HD, RB>, C::kDynSmem, configured);
    if (e != cudaSuccess) return e;
    // programmatic serialization: the CTAs' set-up may overlap the tail of the previous kernel
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(p.total_ctas));
    cfg.blockDim = dim3(kTcThreads);
    cfg.dynamicSmemBytes = C::kDynSmem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, decode_tc_kernel<HD, RB>, tm_k, tm_v, p);
    if (e != cudaSuccess) return e;
    // the merges, also with programmatic serialization (its launch overlaps the decode grid's end)
    cudaLaunchConfig_t ccfg = {};
    ccfg.gridDim = dim3(static_cast<unsigned>(p.n_seqs * p.hkv));
    ccfg.blockDim = dim3(128);
    ccfg.dynamicSmemBytes = 0;
    ccfg.stream = st;
    ccfg.attrs = attr;
    ccfg.numAttrs = 1;
    return cudaLaunchKernelEx(&ccfg, decode_tc_combine_kernel<HD, RB>, p);
}

template <int HD, int RB>
cudaError_t launch_t(const CUtensorMap &tm_k, const CUtensorMap &tm_v, const DecodeParams &p, cudaStream_t st)
{
    using C = DecCfg<HD, RB>;
    static std::atomic<uint64_t> configured{0};
    cudaError_t e = set_dyn_smem_once(decode_attn_kernel<HD, RB>, C::kDynSmem, configured);
    if (e != cudaSuccess) return e;
    decode_attn_kernel<HD, RB><<<p.total_ctas, kDecThreads, C::kDynSmem, st>>>(tm_k, tm_v, p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_decode_attn(int head_dim, int rows_cap, bool tensor_core, const CUtensorMap &tm_k,
                               const CUtensorMap &tm_v, const DecodeParams &p, cudaStream_t st)
{
    if (p.total_ctas <= 0) return cudaSuccess;
    if (tensor_core) {
        if (head_dim == 128) {
            if (rows_cap == 4) return launch_tc<128, 4>(tm_k, tm_v, p, st);
            if (rows_cap == 8) return launch_tc<128, 8>(tm_k, tm_v, p, st);
            if (rows_cap == 16) return launch_tc<128, 16>(tm_k, tm_v, p, st);
        } else if (head_dim == 64) {
            if (rows_cap == 4) return launch_tc<64, 4>(tm_k, tm_v, p, st);
            if (rows_cap == 8) return launch_tc<64, 8>(tm_k, tm_v, p, st);
            if (rows_cap == 16) return launch_tc<64, 16>(tm_k, tm_v, p, st);
        }
        return cudaErrorInvalidValue;
    }
    if (head_dim == 128) {
        if (rows_cap == 4) return launch_t<128, 4>(tm_k, tm_v, p, st);
        if (rows_cap == 8) return launch_t<128, 8>(tm_k, tm_v, p, st);
        if (rows_cap == 16) return launch_t<128, 16>(tm_k, tm_v, p, st);
    } else if (head_dim == 64) {
        if (rows_cap == 4) return launch_t<64, 4>(tm_k, tm_v, p, st);
        if (rows_cap == 8) return launch_t<64, 8>(tm_k, tm_v, p, st);
        if (rows_cap == 16) return launch_t<64, 16>(tm_k, tm_v, p, st);
    }
    return cudaErrorInvalidValue;
}

}  // namespace pe

// Private to the pe library: kernel parameter blocks shared by the host code
// (pe_host.cu) and the kernels (pe_kv.cu, pe_attn.cu).
#pragma once

#include <atomic>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

namespace pe {

constexpr int kBM = 128;               // query rows (GQA-packed) per attention tile
constexpr int kBN = 128;               // keys per attention tile
constexpr int kMaxSegs = 64;           // sequences per append / attention launch
constexpr int kMaxCropSegs = 256;      // sequences per crop launch
constexpr int kAppendMaxPages = 3072;  // new page ids carried by one append launch

// Device status word codes (pe_device_status).
constexpr int kStatusWaitTimeout = 1;
constexpr int kStatusBadPlan = 3;      // the persistent kernel met a partial slot outside its workspace (skipped)

// ---------------------------------------------------------------- append
struct AppendSeg {
    int32_t tok0;          // first token of this segment inside the packed K/V
    int32_t cum0;          // prefix of segment tokens inside this launch
    int32_t n_tokens;
    int32_t len0;          // sequence length before this segment
    int32_t first_new_lp;  // logical index of the first page popped for this segment
    int32_t last_page;     // physical page holding logical page first_new_lp-1 (-1 if none)
    int32_t new0;          // offset of this segment's new page ids in new_pages
    int32_t n_new;
    int32_t table_row;     // seq * max_pages_per_seq
    int32_t seq;
};

struct AppendParams {
    const uint4 *K;        // packed [L][n_total][Hkv][d] bf16, viewed as 16-byte chunks
    const uint4 *V;
    uint4 *k_pool;         // [L][num_pages][Hkv][ps][d]
    uint4 *v_pool;
    int32_t *page_table;   // device mirror [max_seqs][max_pages_per_seq]
    int64_t *seq_len;      // device mirror [max_seqs]
    int32_t L, hkv, dvec, ps, num_pages, n_total, n_segs, seg_tokens;
    AppendSeg segs[kMaxSegs];
    int32_t new_pages[kAppendMaxPages];
};

// ---------------------------------------------------------------- crop
constexpr int kMaxCropFreed = 2048;  // freed page ids carried by one crop launch (debug poison)

struct CropSeg {
    int32_t table_row;
    int32_t keep;          // pages kept
    int32_t old_n;         // pages before the crop
    int32_t seq;
    int64_t new_len;
    int32_t freed0;        // debug poison: this sequence's pages whose last reference went,
    int32_t n_freed;       //   as a range of CropParams::freed
    int32_t tail_page;     // debug poison: last kept page when this sequence is its only holder, else -1
    int32_t pad_;
};

struct CropParams {
    int32_t *page_table;
    int64_t *seq_len;
    uint4 *k_pool;
    uint4 *v_pool;
    int32_t n, poison, L, hkv, ps, dvec, num_pages;
    CropSeg segs[kMaxCropSegs];
    int32_t freed[kMaxCropFreed];
};

// ---------------------------------------------------------------- attention
struct AttnSeq {
    int32_t table_row;     // seq * max_pages_per_seq
    int32_t n_pages;       // ceil(len / ps)
    int32_t q_row0;        // first row of this sequence in packed Q / out
    int32_t n_q;
    int32_t n_keys;        // len
    int32_t item0;         // first CTA work item of this sequence
    int32_t n_qtiles;      // ceil(n_q * group / kBM)
    int32_t n_splits;      // key splits per q-tile (1 without split-KV)
    int64_t part_row0;     // first partial row in the workspace (split-KV)
    int32_t comb0;         // first combine row item (split-KV)
    int32_t pair_top;      // the launch covers q-tile pairs [pair_top - items / (Hkv x splits), pair_top),
                           // heaviest first (pair_top = all pairs, unless a tail launch takes the lightest)
};

struct AttnParams {
    const int32_t *page_table;
    void *out;             // bf16 [rows][Hq][d]
    float *part_o;         // split-KV partial outputs, rows of d fp32 in blocks of 32 rows (part_chunk)
    float *part_lse;       // split-KV partial log2-sum-exp [rows]
    int32_t *status;
    int32_t n_seqs, hq, hkv, group, layer, num_pages, ps, oob_row;
    int32_t split_tiles;   // key tiles per split
    int32_t total_items;
    int32_t total_comb;
    int32_t pairs_fastest;  // one-item kernel: number a sequence's items pairs fastest (else kv-heads fastest)
    int32_t next_stride;   // one-item kernel: CTA b prefetches item b + next_stride's Q tiles into L2 (0: off)
    float scale_log2;      // softmax_scale * log2(e)
    AttnSeq seqs[kMaxSegs];
};

// ---------------------------------------------------------------- persistent (stream-K) attention
// A launch group's work units are (sequence, kv-head, q-tile pair), numbered
// sequence by sequence from AttnSeq::item0 (kv-head fastest, pairs heaviest
// first); a unit loads the key tiles [0, n) of its pair.  The persistent
// kernel runs one CTA per SM: whole units in lockstep rounds, then CTA c's
// contiguous stretch of the remaining (unit, key tile) work; the pieces of
// units cut by a stretch boundary write fp32 partials (O / l and log2-sum-exp)
// into slot `slot`, part `part`, and the warp that writes a slot's last part
// (counted on its ticket) merges the slot's parts.
constexpr int kMaxSkCtas = 160;        // >= SMs of the GPU
constexpr int kSkTicketsPerSlot = 8;   // one per (q-tile, warp of 32 rows)

struct SkCta {
    int32_t u0, t0;        // first unit and its first key tile
    int32_t u1, t1;        // last unit and the key tile it stops before (t1 = 0: u1 is not taken)
    int32_t slot0, part0;  // partial slot and part of u0's piece (slot -1: the whole unit, written directly)
    int32_t slot1, part1;  // the same for u1's piece when u1 > u0
};

struct SkSlot {
    int32_t unit;          // the unit cut into parts
    int32_t n_parts;
};

struct SkParams {
    AttnParams a;          // sequences, shapes, output; part_o / part_lse hold the partials
    int32_t n_ctas, n_slots, max_parts;
    int32_t rounds;        // whole units first: in round r < rounds CTA k takes unit r n_ctas + k (odd r:
                           // r n_ctas + n_ctas - 1 - k); then its tail stretch (cta[k], u0 > u1: none)
    int32_t *tickets;      // [n_slots][2][4] parts written per (slot, q-tile, warp); zero between launches
    SkCta cta[kMaxSkCtas];
    SkSlot slots[kMaxSkCtas];
};

// ---------------------------------------------------------------- decode attention
// Sequences whose queries pack into at most kDecMaxRows rows per kv-head
// (n_q x group) take the decode kernel (pe_decode.cu): CUDA cores, 64-key
// tiles streamed by bulk copies, split-KV merged in-kernel by the last split.
constexpr int kDecMaxRows = 16;
constexpr int kDecKeys = 64;           // keys per decode tile

struct DecodeSeq {
    int32_t table_row;     // seq * max_pages_per_seq
    int32_t n_pages;
    int32_t q_row0;        // first row of this sequence in Q / out
    int32_t n_q;
    int32_t n_keys;        // len
    int32_t cta0;          // CUDA-core kernel: first CTA of this sequence (hkv x n_splits CTAs, kv-head major);
                           // tensor-core kernel: tiles per chunk of this sequence's items
    int32_t n_splits;
    int32_t tile0;         // tensor-core kernel: the first full chunk id of this sequence's items (full
                           // chunks numbered sequence-major, kv-head next)
    int32_t rem0;          // tensor-core kernel: the id of kv-head 0's remainder chunk (kv-head h: rem0 + h),
                           // -1 when the tile count is a multiple of the chunk size
};

struct DecodeParams {
    const int32_t *page_table;
    const void *q;         // bf16 [rows][Hq][d]
    void *out;             // bf16 [rows][Hq][d]
    const void *k_pool;    // bf16 [L][num_pages][Hkv][ps][d]
    const void *v_pool;
    float *part;           // split partials: O [ctas][RB][d], then m [ctas][RB], then l [ctas][RB]
    int32_t *tickets;      // one counter per (sequence, kv-head) of the launch; zero between launches
    int32_t *sched;        // tensor-core kernel: [0] next chunk, [1] CTAs that stopped taking; zero between launches
    int32_t *status;
    int32_t n_seqs, hq, hkv, group, layer, num_pages, ps;
    int32_t oob_row;       // a pool row past the end: boxes there read zeros
    int32_t split_tiles;   // decode tiles per split (CUDA-core kernel) / per chunk (tensor-core kernel, <= 8)
    int32_t total_ctas;
    int32_t total_tiles;   // tensor-core kernel: chunks of all (sequence, kv-head) items
    int32_t full_chunks;   // tensor-core kernel: ids below this are full chunks, the rest remainder chunks
    float scale_log2;      // softmax_scale * log2(e)
    DecodeSeq seqs[kMaxSegs];
    int32_t rem_seq[kMaxSegs];  // tensor-core kernel: the sequence of remainder block j (ids
                                // full_chunks + j hkv .., one per kv-head), blocks longest first
};

// Records `msg` as this thread's last error (pe_last_error) and returns code.
int32_t report_error(int32_t code, const char *msg);

// Launchers (defined in the .cu files).
cudaError_t launch_append(const AppendParams &p, int64_t chunks, cudaStream_t st);
cudaError_t launch_crop(const CropParams &p, cudaStream_t st);
// Fork: copies n device page-table entries from row src_row to dst_row and sets
// the new sequence's device length.
cudaError_t launch_table_copy(int32_t *page_table, int32_t src_row, int32_t dst_row, int32_t n, int64_t *seq_len,
                              int32_t dst_seq, int64_t len, cudaStream_t st);
// Copy-on-write: copies slots [0, slots) of page src to page dst (every layer
// and kv-head, K and V) and points the device table entry at dst.
cudaError_t launch_cow_copy(uint4 *k_pool, uint4 *v_pool, int32_t src, int32_t dst, int32_t slots, int32_t L,
                            int32_t hkv, int32_t ps, int32_t dvec, int32_t num_pages, int32_t *table_entry,
                            cudaStream_t st);
// tm_o: the output as a map of the same shape as tm_q (full q-tiles are stored by TMA); unused when split
cudaError_t launch_replay_attn(int head_dim, bool split, const CUtensorMap &tm_q, const CUtensorMap &tm_k,
                               const CUtensorMap &tm_v, const CUtensorMap &tm_o, const AttnParams &p, cudaStream_t st);
cudaError_t launch_splitkv_combine(int head_dim, const AttnParams &p, cudaStream_t st);
// Persistent stream-K attention (p.n_ctas CTAs), cut units merged in the kernel.
cudaError_t launch_replay_attn_sk(int head_dim, const CUtensorMap &tm_q, const CUtensorMap &tm_k,
                                  const CUtensorMap &tm_v, const SkParams &p, cudaStream_t st);
// rows_cap: 4, 8 or 16 (every sequence's n_q x group fits).
// tm_k / tm_v: the pools as 2-D maps {d, L*num_pages*Hkv*ps} with 64 x min(ps, 64) boxes, 128-byte swizzle.
// tensor_core (d = 128 only): keys on the MMA's M side, 128-key tiles (split_tiles
// counts 128-key tiles); otherwise CUDA cores, 64-key tiles.
cudaError_t launch_decode_attn(int head_dim, int rows_cap, bool tensor_core, const CUtensorMap &tm_k,
                               const CUtensorMap &tm_v, const DecodeParams &p, cudaStream_t st);
cudaError_t launch_bounded_wait_selftest(int32_t *status, uint64_t limit_ns, cudaStream_t st);

// Raises `kernel`'s dynamic shared-memory limit to `bytes` on the current
// device, once per device: the attribute is set on the device that is current
// at the call, so a process that runs caches on several GPUs sets it on each.
// `done` holds one bit per device (devices past 63 set it on every call).
template <typename Kernel>
inline cudaError_t set_dyn_smem_once(Kernel kernel, int bytes, std::atomic<uint64_t> &done)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const uint64_t bit = (dev >= 0 && dev < 64) ? (1ull << dev) : 0;
    if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_acq_rel);
    return e;
}

// Fixed split-KV scratch compiled into the library (pe_attn.cu), used only by
// pe_replay_attn_static_scratch.  static_scratch() returns its device address
// on the current device; the address is looked up once per device.
constexpr int64_t kStaticScratchBytes = 16ll << 20;
cudaError_t static_scratch(float **ptr);

}  // namespace pe

/*
 * pe.h -- paged KV cache with crop and suffix replay, for one GB300 (sm_103a).
 *
 * The operations follow the problem statement of "Forgetting Without
 * Restarting" (Provenance-Guided Selective Replay):
 *   - a metadata-only checkpoint is a token offset, and restoring it is a crop
 *     of the KV cache (Sec. 3.4(b); Sec. 4.1, KVEngine.crop);
 *   - Alg. 1 Restore crops the cache to the last clean boundary; with every
 *     token position a crop point that boundary is tau-1, the last position
 *     before the target's injection step tau (Lemma 1: those states are shared
 *     with the counterfactual run);
 *   - Alg. 1's replay loop advances the state over the T - tau + 1 suffix
 *     positions (Theorem 1, Corollary 1); counterfactually fixed content is
 *     re-materialised by prefill on the cropped cache (Sec. 3.2, Sec. 4.5).
 *     Here that prefill is: append the suffix K/V to the cache, then causal
 *     attention of the suffix queries over prefix + suffix keys.
 *
 * Conventions shared by every call
 *   - tau is 1-based (Sec. 3.1: the target enters at step tau >= 1); a crop to
 *     tau keeps tau-1 tokens.
 *   - Bookkeeping (free list, page tables, lengths) lives on the host, is
 *     updated synchronously and deterministically inside the call, and is
 *     mirrored to the device by work enqueued on `stream`.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Device work of a call runs in stream order; caller buffers
 *     (K, V, Q, out) must stay valid until that work completes.  The library
 *     keeps no reference to them after the call returns.
 *   - All tensors are bf16, row-major, contiguous, 16-byte aligned device
 *     memory unless stated otherwise.
 *   - On any error the cache state is unchanged and pe_last_error() describes
 *     the failure.  This includes a failure of a device step after the
 *     bookkeeping was applied (e.g. an append's kernel launch failing after its
 *     pages were taken): the call undoes its host changes and rewrites the
 *     device page-table rows and lengths of the sequences it touched from the
 *     host, on `stream`, before returning PE_ERR_CUDA.  Pool slots the failed
 *     call already wrote belong to pages or positions outside every
 *     sequence's valid range afterwards, so no later result reads them
 *     (exception: with "debug_poison" on, a batched crop that fails after its
 *     first launch may leave poisoned slots in pages it had already freed).
 *     A cache is not thread-safe: calls on one cache must not run
 *     concurrently.
 *   - Allocation policy: the free list is a LIFO stack whose initial pop order
 *     is `init_free_order`; an append pops one page per new logical page; crop
 *     and release drop one reference per removed page in descending logical
 *     order and push the pages whose last reference goes, so (without forks) a
 *     crop followed by an append of the same length restores the same table.
 */
#ifndef PE_H
#define PE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct pe_cache pe_cache; /* opaque, owned by the library */
typedef int32_t pe_status;

enum {
    PE_OK = 0,
    PE_ERR_INVALID = -1,        /* bad argument: null/misaligned pointer, tau < 1, unknown seq ... */
    PE_ERR_RANGE = -2,          /* index or size out of range: tau-1 > len, n_q > len, layer ... */
    PE_ERR_OOM = -3,            /* free list (or sequence slots) exhausted */
    PE_ERR_CUDA = -4,           /* a CUDA runtime call failed */
    PE_ERR_UNSUPPORTED = -5,    /* shape the kernels do not handle, or device call on a host-only cache */
    PE_ERR_DEVICE_TIMEOUT = -6  /* a kernel's bounded wait ran out (see pe_device_status) */
};

typedef struct {
    int32_t num_layers;         /* L >= 1; one page id addresses the same slot in every layer */
    int32_t num_kv_heads;       /* Hkv >= 1 */
    int32_t head_dim;           /* d: 64 or 128 */
    int32_t page_size;          /* ps tokens per page: 8, 16, 32, 64 or 128 */
    int32_t num_pages;          /* pages in the pool */
    int32_t max_seqs;           /* sequence slots */
    int32_t max_pages_per_seq;  /* page-table row length */
    int32_t host_only;          /* 1: bookkeeping only (no device memory, no kernels); for tests */
    const int32_t *init_free_order; /* host, nullable: pool pop order [num_pages]; NULL = 0,1,2,... */
    void *k_pool;               /* device, nullable: caller-owned K pool, bf16 [L][num_pages][Hkv][ps][d] */
    void *v_pool;               /* device, nullable: caller-owned V pool, same layout.  NULL = the
                                   library allocates (cudaMalloc) and zero-fills both pools */
    int64_t workspace_bytes;    /* split-KV scratch allocated at create; 0 = 256 MiB */
} pe_cache_config;

/* Creates a cache.  Sizes are checked (d, ps, positive counts, int32-addressable
 * pool rows).  Device buffers are allocated on the current CUDA device, which
 * must be of compute capability 10.3 (the kernels are sm_103a code).  Every
 * later call that does device work must be made with that device current
 * (INVALID otherwise, before any state changes); pe_cache_destroy waits for
 * and frees the cache on its own device, whichever device is current.
 * Errors: INVALID, UNSUPPORTED, OOM (host), CUDA. */
pe_status pe_cache_create(const pe_cache_config *cfg, pe_cache **out);
pe_status pe_cache_destroy(pe_cache *cache);

/* New empty sequence (len 0); the lowest free slot id is returned.  OOM if none. */
pe_status pe_seq_create(pe_cache *cache, int32_t *seq_out);
/* Frees every page of `seq` (pushed like a crop to tau = 1) and the slot. */
pe_status pe_seq_release(pe_cache *cache, int32_t seq, void *stream);

/* Crop = restore (Sec. 3.4(b); Alg. 1 Restore).  Keeps the first tau-1 tokens:
 * pages at logical index >= ceil((tau-1)/ps) are removed from the table and
 * lose one reference each (visited in descending logical order); a page whose
 * last reference goes is pushed on the free list.  The device table entries
 * are set to -1 by a kernel on `stream`.  Resets the recomputation counter to
 * 0 and drops checkpoints past the new length.  tau = len+1 keeps every token.
 * freed_out (host, nullable) receives the pages returned to the free list in
 * ascending logical order; n_freed (nullable) their number.
 * Errors: INVALID (tau < 1, unknown seq), RANGE (tau-1 > len, freed_cap too small). */
pe_status pe_crop(pe_cache *cache, int32_t seq, int64_t tau, int32_t *freed_out, int32_t freed_cap,
                  int32_t *n_freed, void *stream);

/* Branching from one base state (Sec. 4.1: every method starts from the same
 * contaminated base, the cache cloned).  The new sequence (lowest free slot)
 * shares every page of `seq` (reference counts), its length, counter and
 * checkpoints; no K/V is copied.  An append into a shared, partially filled
 * last page first copies that page's valid slots into a fresh page on
 * `stream` (copy-on-write); full shared pages are never written.
 * Errors: INVALID (unknown seq), OOM (no sequence slot). */
pe_status pe_seq_fork(pe_cache *cache, int32_t seq, int32_t *new_seq, void *stream);

/* Metadata-only checkpoints (Sec. 3.4(b), Sec. 4.6): a checkpoint is a token
 * offset b, the state after the first b tokens.  pe_checkpoint_add records one
 * (0 <= b <= len; duplicates ignored; RANGE otherwise).  pe_checkpoint_select
 * returns c* = the largest recorded offset b < tau (Alg. 1: the last boundary
 * before the target's entry; RANGE when none, INVALID when tau < 1).
 * pe_restore = select + crop to keep c* tokens (Alg. 1 Restore); the caller
 * then replays positions c*+1 .. T.  pe_seq_checkpoints lists the offsets
 * (ascending). */
pe_status pe_checkpoint_add(pe_cache *cache, int32_t seq, int64_t offset);
pe_status pe_checkpoint_select(const pe_cache *cache, int32_t seq, int64_t tau, int64_t *offset);
pe_status pe_restore(pe_cache *cache, int32_t seq, int64_t tau, int64_t *offset, int32_t *freed_out,
                     int32_t freed_cap, int32_t *n_freed, void *stream);
pe_status pe_seq_checkpoints(const pe_cache *cache, int32_t seq, int64_t *out, int32_t cap, int32_t *n);

/* Crops n sequences (host arrays seqs[n], taus[n]) with one device launch.
 * All-or-nothing: every (seq, tau) is validated before any state changes;
 * a sequence may appear once. */
pe_status pe_crop_batch(pe_cache *cache, int32_t n, const int32_t *seqs, const int64_t *taus, void *stream);

/* Prefill write of the replayed suffix (Sec. 3.2): appends n_tokens positions.
 * K, V: device bf16 [L][n_tokens][Hkv][d].  New pages are popped from the
 * free list before any device work; the copy into the pool runs on `stream`.
 * The recomputation counter grows by n_tokens (Corollary 1 counts it).
 * Errors: RANGE (exceeds max_pages_per_seq), OOM (not enough free pages),
 * INVALID (null/misaligned pointers). */
pe_status pe_append_kv(pe_cache *cache, int32_t seq, const void *K, const void *V, int32_t n_tokens,
                       void *stream);

/* Batched append: sequence i receives tokens [cu_tokens[i], cu_tokens[i+1]) of
 * K_packed / V_packed, device bf16 [L][cu_tokens[n]][Hkv][d]; cu_tokens is a
 * host array [n+1] starting at 0.  One device launch; all-or-nothing. */
pe_status pe_append_kv_batch(pe_cache *cache, int32_t n, const int32_t *seqs, const void *K_packed,
                             const void *V_packed, const int32_t *cu_tokens, void *stream);

/* Replay attention (Alg. 1 replay loop; Sec. 3.2 prefill on the cropped cache).
 * The n_q queries are the LAST n_q positions of `seq`: query i sits at
 * position len-n_q+i and attends keys 0..len-n_q+i of `layer` (causal,
 * bottom-right aligned).  q-head h reads kv-head h / (Hq/Hkv).
 *   O = softmax(softmax_scale * q K^T) V, fp32 accumulation, bf16 output.
 * Q: device bf16 [n_q][Hq][d]; out: device bf16 [n_q][Hq][d].
 * Hq must be a multiple of Hkv with Hq/Hkv a power of two <= 128.
 * Errors: RANGE (n_q > len, layer), INVALID, UNSUPPORTED. */
pe_status pe_replay_attn(pe_cache *cache, int32_t seq, int32_t layer, const void *Q, void *out, int32_t n_q,
                         int32_t num_q_heads, float softmax_scale, void *stream);

/* Batched varlen replay attention: sequence i's queries are rows
 * [cu_q[i], cu_q[i+1]) of Q_packed / out (device bf16 [cu_q[n]][Hq][d]), and
 * are its last cu_q[i+1]-cu_q[i] positions.  cu_q: host [n+1], from 0. */
pe_status pe_replay_attn_batch(pe_cache *cache, int32_t n, const int32_t *seqs, int32_t layer,
                               const void *Q_packed, const int32_t *cu_q, void *out, int32_t num_q_heads,
                               float softmax_scale, void *stream);

/* ---- Replay with the indep split (Sec. 4.5, the T - tau + 1 paragraph;
 * Sec. 4.1 methods B7 and B5').  Post-target turns whose content is the same
 * in the counterfactual world are re-prefilled, many positions per pass;
 * turns that depend on the target are re-decoded, one position per pass.
 * Selective replay (B7) counts model turns independent of the target as
 * known; full reset with a prefix cache (B5') re-decodes every model turn of
 * the suffix.  Both recompute the same T - tau + 1 positions (Corollary 1) and
 * coincide when no model turn is independent. */
enum { PE_TURN_INPUT = 0, PE_TURN_MODEL_INDEP = 1, PE_TURN_MODEL_DEP = 2 };
enum { PE_POLICY_SELECTIVE = 0, PE_POLICY_PREFIX_CACHE = 1 };

/* Plans the passes of n agents' suffix replays (host only, no cache).
 * Agent i's suffix is turns [cu_turns[i], cu_turns[i+1]) of turn_len /
 * turn_kind (host arrays; cu_turns host [n+1], from 0, non-decreasing).
 * A unit is a maximal run of consecutive known positions (one prefill pass)
 * or one position to decode; empty turns contribute nothing.  Agents advance
 * in lockstep rounds: round r runs every agent's r-th unit.
 * take (host int32 [n_rounds][n], row-major, nullable when take_cap == 0)
 * receives the positions agent i appends and attends in round r (0 = idle);
 * *n_rounds (required) the number of rounds; *decode_tokens (nullable) the
 * positions decoded over all agents.  Call with take = NULL, take_cap = 0 to
 * learn the size.
 * Errors: INVALID (bad arrays, kind or policy, negative length, an agent's
 * suffix above INT32_MAX), RANGE (n_rounds * n > take_cap; *n_rounds is set). */
pe_status pe_replay_schedule(int32_t n, const int32_t *cu_turns, const int32_t *turn_len, const int32_t *turn_kind,
                             int32_t policy, int32_t *take, int64_t take_cap, int32_t *n_rounds,
                             int64_t *decode_tokens);

/* Runs the rounds of a replay on the cache: in round r, every agent i with
 * take[r*n + i] > 0 appends its next take[r*n + i] positions (K/V of all
 * layers, as pe_append_kv_batch), then for each layer attends those positions'
 * queries (as pe_replay_attn_batch).  Agent i's positions are rows
 * [cu_tok[i], cu_tok[i+1]) of K, V (device bf16 [L][N][Hkv][d]) and of Q, out
 * (device bf16 [L][N][Hq][d]), N = cu_tok[n]; cu_tok host [n+1], from 0.
 * The rounds must cover each agent's rows exactly (sum over r of take = its
 * row count).  Every argument, the pages all rounds need (checked up front,
 * including copy-on-write) and the page-table capacity are checked before any
 * state changes; a CUDA error (CUDA) in any round undoes the bookkeeping of
 * every round of the call (the outputs of earlier rounds may have been written).
 * On a host-only cache only the bookkeeping runs (Q, out unused).
 * Errors: INVALID, RANGE, OOM, UNSUPPORTED, CUDA. */
pe_status pe_replay_rounds(pe_cache *cache, int32_t n, const int32_t *seqs, int32_t n_rounds, const int32_t *take,
                           const int32_t *cu_tok, const void *K, const void *V, const void *Q, void *out,
                           int32_t num_q_heads, float softmax_scale, void *stream);

/* Variant of pe_replay_attn for callers that cannot allocate device memory at
 * the time they run attention: code inside a stream host callback or a
 * latency-critical serving loop where cudaMalloc (which may synchronise the
 * device) is not allowed, or a process whose device memory is entirely
 * reserved by its own allocator.  The paper has no counterpart; it is a
 * property of this library, not of the method.
 * It always takes the split-KV path and keeps the split partials in one fixed
 * 16 MiB array compiled into the library (every GPU that loads the library
 * holds it until the process exits) instead of the cache's workspace; it
 * calls no cudaMalloc/cudaFree and no allocating routine.  Arguments, result
 * and errors are those of pe_replay_attn; in addition RANGE when one key
 * split of n_q x num_q_heads rows does not fit the array
 * (ceil(n_q*(Hq/Hkv)/128) * Hkv * 128 * (4*d + 4) bytes must be <= 16 MiB).
 * The first call on a device looks up the array's device address (once per
 * device, with that device current); make that first call before any stream
 * capture.  Every call shares the array and overwrites what the previous call
 * left there (no part of it needs to start at zero): calls that overlap on
 * the GPU (different streams, concurrent threads) race and must be ordered by
 * the caller. */
pe_status pe_replay_attn_static_scratch(pe_cache *cache, int32_t seq, int32_t layer, const void *Q, void *out,
                                        int32_t n_q, int32_t num_q_heads, float softmax_scale, void *stream);

/* Host-side state queries (no device work). */
pe_status pe_seq_info(const pe_cache *cache, int32_t seq, int64_t *len, int64_t *appended_since_crop);
pe_status pe_seq_page_table(const pe_cache *cache, int32_t seq, int32_t *out, int32_t cap, int32_t *n);
pe_status pe_free_list(const pe_cache *cache, int32_t *out, int32_t cap, int32_t *n); /* top of stack first */
/* Reference count of every page (out[num_pages]; 0 = on the free list). */
pe_status pe_page_refs(const pe_cache *cache, int32_t *out, int32_t cap);

/* Synchronous copy of a sequence's DEVICE page-table row (first `cap` entries)
 * into host `out`, after all work on `stream`; for checking the mirror. */
pe_status pe_seq_device_page_table(pe_cache *cache, int32_t seq, int32_t *out, int32_t cap, void *stream);

/* Device pool pointers (for reading pool contents back). */
pe_status pe_cache_pools(const pe_cache *cache, void **k_pool, void **v_pool);

/* Options: "splitkv" = -1 (auto, default) / 0 (never) / 1 (always);
 * "num_splits" = 0 (auto) or the split count; "debug_poison" = 0/1: crop
 * fills freed pages and the stale tail of the last kept page with a finite
 * sentinel (bf16 2^100), so that a kernel reading them unmasked gives a
 * visibly wrong result; "decode_kernel" = 1 (default) / 2 / 0: sequences
 * whose n_q x (Hq/Hkv) query rows fit in 16 take a decode kernel -- 1:
 * tcgen05 with keys on the MMA's M side (d = 64 and 128), split items merged
 * by a combine launch; 2: CUDA cores, split-KV merged in-kernel; 0: no
 * decode kernel (the prefill kernel serves every call); "attn_kernel" = 1
 * (default) / 2 / 0: the prefill kernel -- 1: the persistent stream-K kernel
 * for launch groups whose one-work-item-per-CTA plan would need key splits or
 * a tail launch and whose q-tile pairs x Hkv number between a quarter of the
 * SMs and two waves, the one-item kernel otherwise; 2: always persistent; 0:
 * always one-item; "attn_ctas" = 0 (auto) or the persistent kernel's CTA
 * count; "attn_order" = -1 (auto) / 0 / 1: how the one-item kernel numbers a
 * sequence's CTAs -- 0: kv-heads fastest, every head's heaviest q-tile pairs
 * first; 1: pairs fastest, so the CTAs resident at once share one or two
 * kv-heads' keys in L2; auto takes 1 for launches of at least 32 CTAs per SM;
 * "fail_launch_after" = k >= 0
 * (test hook): the device step after the next k fails with PE_ERR_CUDA
 * without being launched, once (-1 = off); on a host-only cache the steps a
 * device cache would launch are counted the same way.  Split
 * partials and the merge counters (decode kernel, persistent kernel) live in
 * the cache's workspace, so attention calls on one cache must not overlap on
 * the GPU (issue them on one stream, or order the streams). */
pe_status pe_set_option(pe_cache *cache, const char *key, int64_t value);

/* Synchronises `stream` and reads the device status word.  *code = 0 when no
 * kernel reported a problem, else the first recorded code (1 = a bounded
 * wait ran out; 2 = the decode kernel met a page id outside the pool and
 * skipped it; 3 = the persistent kernel met a partial slot outside its
 * workspace and skipped it).  clear != 0 resets it, and after a nonzero code
 * also the split-merge counters of the decode and persistent kernels and the
 * decode scheduler's.  Returns DEVICE_TIMEOUT if
 * *code != 0. */
pe_status pe_device_status(pe_cache *cache, int32_t *code, int32_t clear, void *stream);

/* Failure-detection self-test: launches one kernel whose single wait (the same
 * bounded mbarrier wait the attention kernel uses) is on a barrier nothing
 * arrives at.  After limit_ns (1 us .. 2 s) the wait gives up, records status
 * code 1 in the cache's device status word and the kernel returns, leaving the
 * context usable; pe_device_status then reports DEVICE_TIMEOUT.  The paper has
 * no counterpart (its failure handling is at the tool level). */
pe_status pe_selftest_bounded_wait(pe_cache *cache, int64_t limit_ns, void *stream);

/* Plan of the most recent replay-attention launch group on this cache: split
 * = 1 when the split-KV path ran (a combine launch followed the attention, the
 * persistent kernel cut units and merged their parts in-kernel, or the
 * CUDA-core decode kernel merged in-kernel), n_splits = key splits of its
 * first sequence (of the tail launch, when one ran: a group of one sequence
 * whose last wave of CTAs would be mostly empty runs its lightest q-tile pairs
 * in a second, split-KV launch), ctas = attention CTAs launched in all. */
pe_status pe_last_attn_plan(const pe_cache *cache, int32_t *split, int32_t *n_splits, int32_t *ctas);

/* The persistent prefill kernel's work plan for one launch group, made by the
 * same host planner an attention call runs when it takes that kernel
 * ("attn_kernel" = 2), without any device work; host-only caches too.  It
 * lets a caller (or a test) check on the host that the plan covers every key
 * tile once.  The group is sequences seqs[0..n) (1 <= n <= 64, live, distinct)
 * whose queries are their last cu_q[i+1] - cu_q[i] positions (cu_q host [n+1],
 * from 0; each count in [1, len]), with num_q_heads as in pe_replay_attn; the
 * planner orders them longest first (ties in the given order).  num_sms: the
 * SM count to plan for, 1..160 (0 = the cache's device; required for a
 * host-only cache).  The split partials are sized against the cache's
 * workspace_bytes.  A unit is (sequence, kv-head, pair of 128-row q-tiles):
 * sequences in planning order, then pairs heaviest (latest queries) first,
 * kv-heads fastest; its key tiles are the 128-key tiles its later q-tile sees.
 * The kernel's CTA k first takes whole units in `rounds` lockstep rounds (in
 * round r the unit r*n_ctas + k, or r*n_ctas + n_ctas-1-k when r is odd), then
 * its tail stretch: from key tile t0 of unit u0 up to key tile t1 of unit u1
 * (t1 = 0: up to the start of u1), or nothing when u0 > u1.  A cut unit's
 * pieces are its parts, written as fp32 partials and merged in the kernel.
 * Outputs (host):
 *   info[5] (required): n_ctas, rounds, n_slots (cut units), max_parts, n_units;
 *   order_out[n] (nullable): the sequences in planning order;
 *   unit_tiles[units_cap] (nullable): each unit's key tiles;
 *   ctas[ctas_cap][8] (nullable): per CTA u0, t0, u1, t1, slot0, part0, slot1,
 *     part1 -- the partial slot and part of the stretch's first and last
 *     piece (slot -1: that piece is a whole unit, written directly);
 *   slots[slots_cap][2] (nullable): per cut unit its unit and part count.
 * Errors: INVALID, UNSUPPORTED (group size), RANGE (a cap below the plan's
 * size; info is written first).  The paper has no counterpart: this plans the
 * build's own kernel. */
pe_status pe_attn_plan_persistent(pe_cache *cache, int32_t n, const int32_t *seqs, const int32_t *cu_q,
                                  int32_t num_q_heads, int32_t num_sms, int32_t *info, int32_t *order_out,
                                  int32_t *unit_tiles, int32_t units_cap, int32_t *ctas, int32_t ctas_cap,
                                  int32_t *slots, int32_t slots_cap);

/* Every launch an attention call would make for this batch (the arguments of
 * pe_replay_attn_batch without tensors), planned by the same host code with
 * no device work and no change to the cache; host-only caches too.  It lets a
 * caller (or a test) check the plans on the host.  A sequence with no queries
 * takes no launch.  num_sms as in pe_attn_plan_persistent.  The launches are written to words[cap] (host,
 * nullable: call with NULL to learn *n_words, required) one after another,
 * each as 7 + 10 * n_seqs int64 words:
 *   kind (0: the one-item prefill kernel; 1: its split-KV tail launch, over
 *     pairs [0, pair_top) of its one sequence; 2: the persistent kernel, see
 *     pe_attn_plan_persistent; 3: sequences the decode kernel takes, not
 *     planned further), split (partials merged by a combine launch, or cut
 *     units for kind 2), CTAs, combine rows, split_tiles (128-key tiles per
 *     split), pairs_fastest (the one-item kernel's CTA order), n_seqs;
 *   then per sequence: seq, item0 (its first CTA), n_q, n_keys, n_qtiles,
 *     n_splits, pair_top, part_row0 (its first partial row), comb0 (its first
 *     combine row), q_row0 (its first row of Q and out).
 * A one-item launch's CTA b works on sequence i with item0_i <= b < item0_{i+1}
 * (the last: CTAs), local = b - item0_i; with pairs_fastest, pair = pair_top -
 * 1 - local % P (P = that sequence's CTAs / (Hkv x n_splits)), split = (local
 * / P) % n_splits, kv-head = local / P / n_splits; else kv-head = local % Hkv,
 * split = (local / Hkv) % n_splits, pair = pair_top - 1 - local / Hkv /
 * n_splits.  It computes q-tiles 2 pair and 2 pair + 1 (those below n_qtiles)
 * over key tiles [split x split_tiles, +split_tiles); a split launch writes
 * partial row part_row0 + ((q-tile x Hkv + kv-head) x n_splits + split) x 128
 * + r for row r, and its combine merges, for each of its combine rows
 * comb0 + (q-tile x Hkv + kv-head) x 128 + r, the n_splits rows from there.
 * Errors: INVALID, RANGE (cap below *n_words, n_q > len), UNSUPPORTED.  The
 * paper has no counterpart: this plans the build's own kernels. */
pe_status pe_attn_plan_launches(pe_cache *cache, int32_t n, const int32_t *seqs, const int32_t *cu_q,
                                int32_t num_q_heads, int32_t num_sms, int64_t *words, int64_t cap,
                                int64_t *n_words);

/* Number of kernel launches this cache has made so far (crop, append,
 * attention, combine); lets a caller count its device work. */
pe_status pe_kernel_launches(const pe_cache *cache, int64_t *count);

/* ---- Provenance graph (Sec. 3.4(a); Alg. 1 lines 1-3), host only ----------
 * The runtime records artifacts in execution order: id (unique), type,
 * parents (ids already added; edges run parent -> child), the source ids the
 * artifact carries (e.g. a forget target z and the artifacts derived while z
 * was resident), its token span [token_begin, token_end) in the session, its
 * turn, and whether it committed an external side effect.
 *   pe_prov_locate_source: LocateSource(z), the artifact through which z
 *     entered: a carrier of z none of whose parents carries z (earliest
 *     token_begin, then smallest id); RANGE when nothing carries z.
 *   pe_prov_taint_closure: TaintClosure(s) = I(z), the artifacts reachable
 *     from s (s included), ids ascending into out[cap]; *n their number and
 *     *n_committed how many committed side effects (Theorem 1's assumption A3
 *     needs 0 for an exact replay).  RANGE when s is unknown or cap < *n.
 *   pe_prov_first_entry: FirstEntry(s) = tau, the 1-based position of the
 *     closure's first token; pe_crop(seq, tau) then keeps the clean prefix.
 * Errors of pe_prov_add: INVALID (duplicate id, unknown parent, bad span). */
typedef struct pe_prov pe_prov;
pe_status pe_prov_create(pe_prov **out);
pe_status pe_prov_destroy(pe_prov *graph);
pe_status pe_prov_add(pe_prov *graph, int64_t id, int32_t type, const int64_t *parents, int32_t n_parents,
                      const int64_t *source_ids, int32_t n_sources, int64_t token_begin, int64_t token_end,
                      int32_t turn, int32_t committed);
pe_status pe_prov_locate_source(const pe_prov *graph, int64_t z, int64_t *source);
pe_status pe_prov_taint_closure(const pe_prov *graph, int64_t source, int64_t *out, int32_t cap, int32_t *n,
                                int32_t *n_committed);
pe_status pe_prov_first_entry(const pe_prov *graph, int64_t source, int64_t *tau);

/* Thread-local description of the last error on this thread ("" if none). */
const char *pe_last_error(void);
/* Library version string. */
const char *pe_version(void);

#ifdef __cplusplus
}
#endif
#endif /* PE_H */

// Host side of the pe library: the paged KV store's bookkeeping (free list,
// page tables, lengths, recomputation counters), argument checks, tensor maps
// and kernel launches behind the C ABI declared in include/pe.h.
//
// Crop = restore of a metadata-only checkpoint (Sec. 3.4(b), Sec. 4.1 crop);
// Alg. 1 Restore crops to tau-1; the replay loop re-prefills the T-tau+1
// suffix positions (Theorem 1, Corollary 1, Sec. 3.2).
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "pe.h"
#include "pe_internal.h"

using namespace pe;

namespace {

thread_local std::string g_err;

pe_status fail(pe_status code, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_err = buf;
    return code;
}

pe_status cuda_fail(cudaError_t e, const char *what)
{
    return fail(PE_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

// Merge counters in one zeroed device array: decode's per (sequence, kv-head)
// of a launch, its scheduler's two, then the persistent attention's per slot.
int64_t ticket_count(int32_t hkv) { return static_cast<int64_t>(kMaxSegs) * hkv + 2 + kMaxSkCtas * kSkTicketsPerSlot; }

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    }
    return fn;
}

}  // namespace

int32_t pe::report_error(int32_t code, const char *msg)
{
    g_err = msg;
    return code;
}

// Undo log of one C-ABI call's changes to the host bookkeeping.  Every change
// a call makes goes through the journal helpers below; a call that fails after
// changing the state (a kernel launch failed after pages were taken or given
// back) undoes them and re-mirrors the touched sequences' device rows, so an
// error leaves the cache as it was before the call.  Kept small: a touched
// sequence saves its table from the first changed entry; the free list saves
// only the entries popped below its start height; reference counts are not
// logged at all, since every change to one goes with a change of a table entry
// of a touched sequence and is undone from the two tables' difference.
struct SeqSave {
    int32_t seq;
    int32_t from;                // table entries [from, size0) are saved in `tail`
    int32_t size0;               // table size before the call
    std::vector<int32_t> tail;
    int64_t len, appended;
    std::vector<int64_t> ckpt;
    uint8_t alive;
};

struct Journal {
    size_t low = 0;                    // lowest free-list height the call reached (its start height first)
    std::vector<int32_t> popped;       // entries of the start free list popped below `low`, in pop order
    std::vector<SeqSave> seqs;         // one per touched sequence
    std::vector<int32_t> seq_index;    // sequence -> index in seqs, -1 when untouched
};

struct pe_cache {
    pe_cache_config cfg{};
    bool host_only = false;
    // host bookkeeping (authoritative)
    std::vector<int32_t> free_stack;               // top = back()
    std::vector<std::vector<int32_t>> table;       // per sequence slot
    std::vector<int64_t> len, appended;
    std::vector<uint8_t> alive;
    std::vector<int32_t> refs;                     // sequences holding each page (0 = free)
    std::vector<std::vector<int64_t>> ckpt;        // per sequence: checkpoint token offsets, ascending
    // device state
    int device = 0;
    int num_sms = 148;
    void *k_pool = nullptr, *v_pool = nullptr;
    bool own_pools = false;
    int32_t *d_table = nullptr;
    int64_t *d_len = nullptr;
    int32_t *d_status = nullptr;
    float *d_ws = nullptr;
    int64_t ws_bytes = 0;
    int32_t *d_tickets = nullptr;  // merge counters: decode (per sequence and kv-head, then the scheduler's
                                   // two), then the persistent attention's (per slot, q-tile and warp)
    int64_t pool_rows = 0;  // L * num_pages * Hkv * ps
    CUtensorMap tm_k{}, tm_v{};    // tensor-core kernel: 64 x ps boxes
    CUtensorMap tm_kd{}, tm_vd{};  // decode kernel: 64 x min(ps, 64) boxes
    // options
    int splitkv = -1, num_splits = 0, debug_poison = 0, decode_kernel = 1, dec_chunks_per_sm = 3;
    int attn_kernel = 1;          // prefill kernel: 1 auto, 2 persistent stream-K, 0 one work item per CTA
    int attn_ctas = 0;            // persistent kernel's CTA count (0 = chosen by the planner)
    int attn_order = -1;          // one-item kernel's item order: -1 auto, 0 kv-heads fastest, 1 pairs fastest
    int64_t launches = 0;
    int32_t last_split = 0, last_splits = 0, last_ctas = 0;  // plan of the last attention launch
    Journal jr;                   // changes of the call in progress
    std::vector<int64_t> *plan_rec = nullptr;  // set only inside pe_attn_plan_launches: record, do not launch
    int64_t fail_after = -1;      // test hook "fail_launch_after": device steps left before an injected failure
};

namespace {

pe_status check_seq(const pe_cache *c, int32_t seq)
{
    if (!c) return fail(PE_ERR_INVALID, "null cache");
    if (seq < 0 || seq >= c->cfg.max_seqs || !c->alive[seq]) return fail(PE_ERR_INVALID, "unknown sequence %d", seq);
    return PE_OK;
}

// A device cache's memory and tensor maps belong to the device that was current
// when it was created; a call made with another device current would launch
// there with pointers that device cannot use, so it is refused before any
// state changes.
pe_status check_device(const pe_cache *c)
{
    if (!c) return fail(PE_ERR_INVALID, "null cache");
    if (c->host_only) return PE_OK;
    int dev = -1;
    const cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev != c->device)
        return fail(PE_ERR_INVALID, "the cache lives on device %d, but device %d is current", c->device, dev);
    return PE_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// ---- journal: every bookkeeping change of a call, undone if the call fails
// Saves sequence `seq`'s state before the call changes its table entries at
// index >= from (or its length, counter, checkpoints, liveness).
void j_seq(pe_cache *c, int32_t seq, int32_t from)
{
    Journal &j = c->jr;
    if (j.seq_index.empty()) j.seq_index.assign(c->cfg.max_seqs, -1);
    const std::vector<int32_t> &t = c->table[seq];
    int32_t &ix = j.seq_index[seq];
    if (ix < 0) {
        ix = static_cast<int32_t>(j.seqs.size());
        SeqSave sv;
        sv.seq = seq;
        sv.size0 = static_cast<int32_t>(t.size());
        sv.from = std::min(from, sv.size0);
        sv.tail.assign(t.begin() + sv.from, t.end());
        sv.len = c->len[seq];
        sv.appended = c->appended[seq];
        sv.ckpt = c->ckpt[seq];
        sv.alive = c->alive[seq];
        j.seqs.push_back(std::move(sv));
        return;
    }
    SeqSave &sv = j.seqs[ix];
    if (from < sv.from) {  // entries [from, sv.from) are still unchanged: save them too
        sv.tail.insert(sv.tail.begin(), t.begin() + from, t.begin() + sv.from);
        sv.from = from;
    }
}

void free_push(pe_cache *c, int32_t pg) { c->free_stack.push_back(pg); }

int32_t free_pop(pe_cache *c)
{
    const int32_t pg = c->free_stack.back();
    c->free_stack.pop_back();
    Journal &j = c->jr;
    if (c->free_stack.size() < j.low) {  // an entry of the start free list
        j.low = c->free_stack.size();
        j.popped.push_back(pg);
    }
    return pg;
}

void set_ref(pe_cache *c, int32_t pg, int32_t v) { c->refs[pg] = v; }

void journal_clear(pe_cache *c)
{
    Journal &j = c->jr;
    for (const SeqSave &sv : j.seqs) j.seq_index[sv.seq] = -1;
    j.seqs.clear();
    j.popped.clear();
    j.low = c->free_stack.size();
}

// Undoes the call's changes and rewrites the device mirror
// (table row and length) of every touched live sequence on `st`, after any
// device work the call already enqueued.
void rollback(pe_cache *c, cudaStream_t st)
{
    Journal &j = c->jr;
    // the free list: back to its start entries below `low`, then the popped ones in reverse pop order
    c->free_stack.resize(j.low);
    for (auto it = j.popped.rbegin(); it != j.popped.rend(); ++it) c->free_stack.push_back(*it);
    for (const SeqSave &sv : j.seqs) {
        std::vector<int32_t> &t = c->table[sv.seq];
        // reference counts: one more for an entry the call removed or replaced, one fewer for one it added
        const size_t now = t.size(), end = std::max<size_t>(now, static_cast<size_t>(sv.size0));
        for (size_t i = sv.from; i < end; ++i) {
            const int32_t was = i < static_cast<size_t>(sv.size0) ? sv.tail[i - sv.from] : -1;
            const int32_t is = i < now ? t[i] : -1;
            if (was == is) continue;
            if (was >= 0) c->refs[was] += 1;
            if (is >= 0) c->refs[is] -= 1;
        }
        t.resize(sv.size0);
        std::copy(sv.tail.begin(), sv.tail.end(), t.begin() + sv.from);
        c->len[sv.seq] = sv.len;
        c->appended[sv.seq] = sv.appended;
        c->ckpt[sv.seq] = sv.ckpt;
        c->alive[sv.seq] = sv.alive;
        if (!c->host_only && sv.alive) {
            const int64_t row = static_cast<int64_t>(sv.seq) * c->cfg.max_pages_per_seq;
            if (!t.empty())
                cudaMemcpyAsync(c->d_table + row, t.data(), sizeof(int32_t) * t.size(), cudaMemcpyHostToDevice, st);
            cudaMemcpyAsync(c->d_len + sv.seq, &c->len[sv.seq], sizeof(int64_t), cudaMemcpyHostToDevice, st);
        }
    }
    if (!c->host_only) cudaStreamSynchronize(st);  // the copies read host memory the next call may change
    journal_clear(c);
}

// One C-ABI call that changes bookkeeping: end() keeps the changes on success
// and rolls them back on any error.
struct CallTxn {
    pe_cache *c;
    cudaStream_t st;
    CallTxn(pe_cache *c_, cudaStream_t st_) : c(c_), st(st_) { journal_clear(c); }
    pe_status end(pe_status s)
    {
        if (s != PE_OK) rollback(c, st);
        else journal_clear(c);
        return s;
    }
    ~CallTxn() { journal_clear(c); }
};

// Test hook: with "fail_launch_after" = k, the device step after the next k
// fails with PE_ERR_CUDA without running (on a host-only cache the steps a
// device cache would launch are counted the same way).
bool injected_failure(pe_cache *c)
{
    if (c->fail_after < 0) return false;
    if (c->fail_after-- > 0) return false;
    c->fail_after = -1;
    return true;
}

pe_status launch_fault(const char *what)
{
    return fail(PE_ERR_CUDA, "%s: launch failure injected by the fail_launch_after test hook", what);
}

pe_status encode_2d(CUtensorMap *m, void *base, uint64_t cols, uint64_t rows, uint32_t box_cols, uint32_t box_rows)
{
    EncodeTiledFn fn = encode_fn();
    if (!fn) return fail(PE_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols * 2};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t es[2] = {1, 1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, es,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(PE_ERR_CUDA, "cuTensorMapEncodeTiled (2d) failed: %d", static_cast<int>(r));
    return PE_OK;
}

// Q viewed as [rows][Hq][d]: box (64, g, 128/g) gathers 128/g queries x g heads.
pe_status encode_q(CUtensorMap *m, const void *q, int64_t rows, int hq, int d, int g)
{
    EncodeTiledFn fn = encode_fn();
    if (!fn) return fail(PE_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(hq), static_cast<cuuint64_t>(rows)};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(d) * 2, static_cast<cuuint64_t>(hq) * d * 2};
    cuuint32_t box[3] = {64, static_cast<cuuint32_t>(g), static_cast<cuuint32_t>(kBM / g)};
    cuuint32_t es[3] = {1, 1, 1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(q), dims, strides, box, es,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(PE_ERR_CUDA, "cuTensorMapEncodeTiled (q) failed: %d", static_cast<int>(r));
    return PE_OK;
}

void free_device(pe_cache *c)
{
    if (c->own_pools) {
        if (c->k_pool) cudaFree(c->k_pool);
        if (c->v_pool) cudaFree(c->v_pool);
    }
    if (c->d_table) cudaFree(c->d_table);
    if (c->d_len) cudaFree(c->d_len);
    if (c->d_status) cudaFree(c->d_status);
    if (c->d_ws) cudaFree(c->d_ws);
    if (c->d_tickets) cudaFree(c->d_tickets);
    c->k_pool = c->v_pool = nullptr;
    c->d_tickets = nullptr;
    c->d_table = nullptr;
    c->d_len = nullptr;
    c->d_status = nullptr;
    c->d_ws = nullptr;
}

// ---- crop bookkeeping shared by pe_crop, pe_crop_batch, pe_restore and pe_seq_release
struct CropPlan {
    int32_t seq;
    int32_t keep, old_n;
    int64_t new_len;
    int32_t n_freed;                 // pages whose last reference this crop drops
    std::vector<int32_t> freed;      // filled by apply_crop, ascending logical order
    int32_t tail_page = -1;          // last kept page when this sequence is its only holder
};

// Drops one reference per removed page (descending logical order); a page whose
// last reference goes is pushed onto the free list.
void apply_crop(pe_cache *c, CropPlan &pl, int32_t *freed_out)
{
    j_seq(c, pl.seq, pl.keep);
    std::vector<int32_t> &t = c->table[pl.seq];
    // the freed pages' ids are kept only for the caller and the debug poison
    const bool keep_ids = freed_out != nullptr || c->debug_poison;
    pl.freed.clear();
    for (int32_t e = pl.old_n - 1; e >= pl.keep; --e) {
        const int32_t pg = t[e];
        set_ref(c, pg, c->refs[pg] - 1);
        if (c->refs[pg] == 0) {
            free_push(c, pg);
            if (keep_ids) pl.freed.push_back(pg);
        }
    }
    std::reverse(pl.freed.begin(), pl.freed.end());  // ascending logical order
    if (freed_out) std::copy(pl.freed.begin(), pl.freed.end(), freed_out);
    t.resize(pl.keep);
    c->len[pl.seq] = pl.new_len;
    c->appended[pl.seq] = 0;
    std::vector<int64_t> &ck = c->ckpt[pl.seq];
    while (!ck.empty() && ck.back() > pl.new_len) ck.pop_back();
    pl.tail_page = (pl.keep > 0 && pl.new_len % c->cfg.page_size != 0 && c->refs[t[pl.keep - 1]] == 1)
                       ? t[pl.keep - 1]
                       : -1;
}

pe_status launch_crops(pe_cache *c, const std::vector<CropPlan> &plans, cudaStream_t st)
{
    std::vector<char> buf(sizeof(CropParams));
    CropParams &p = *reinterpret_cast<CropParams *>(buf.data());
    std::memset(&p, 0, sizeof p);
    p.page_table = c->d_table;
    p.seq_len = c->d_len;
    p.k_pool = static_cast<uint4 *>(c->k_pool);
    p.v_pool = static_cast<uint4 *>(c->v_pool);
    p.poison = c->debug_poison;
    p.L = c->cfg.num_layers;
    p.hkv = c->cfg.num_kv_heads;
    p.ps = c->cfg.page_size;
    p.dvec = c->cfg.head_dim / 8;
    p.num_pages = c->cfg.num_pages;
    size_t i = 0;
    while (i < plans.size()) {
        p.n = 0;
        int32_t nf = 0;
        while (i < plans.size() && p.n < kMaxCropSegs) {
            const CropPlan &pl = plans[i];
            const int32_t want = c->debug_poison ? static_cast<int32_t>(pl.freed.size()) : 0;
            if (p.n > 0 && nf + want > kMaxCropFreed) break;  // next launch
            ++i;
            CropSeg &sg = p.segs[p.n++];
            sg.table_row = pl.seq * c->cfg.max_pages_per_seq;
            sg.keep = pl.keep;
            sg.old_n = pl.old_n;
            sg.seq = pl.seq;
            sg.new_len = pl.new_len;
            sg.freed0 = nf;
            sg.n_freed = std::min(want, kMaxCropFreed - nf);
            for (int32_t k = 0; k < sg.n_freed; ++k) p.freed[nf + k] = pl.freed[k];
            nf += sg.n_freed;
            sg.tail_page = pl.tail_page;
        }
        if (injected_failure(c)) return launch_fault("crop kernel");
        if (c->host_only) continue;
        cudaError_t e = launch_crop(p, st);
        if (e != cudaSuccess) return cuda_fail(e, "crop kernel launch");
        c->launches++;
    }
    return PE_OK;
}

pe_status plan_crop(const pe_cache *c, int32_t seq, int64_t tau, CropPlan *pl)
{
    pe_status s = check_seq(c, seq);
    if (s != PE_OK) return s;
    if (tau < 1) return fail(PE_ERR_INVALID, "tau = %lld < 1", static_cast<long long>(tau));
    if (tau - 1 > c->len[seq])
        return fail(PE_ERR_RANGE, "tau - 1 = %lld exceeds the sequence length %lld", static_cast<long long>(tau - 1),
                    static_cast<long long>(c->len[seq]));
    pl->seq = seq;
    pl->new_len = tau - 1;
    pl->keep = static_cast<int32_t>(ceil_div(tau - 1, c->cfg.page_size));
    pl->old_n = static_cast<int32_t>(c->table[seq].size());
    pl->n_freed = 0;
    for (int32_t e = pl->keep; e < pl->old_n; ++e) pl->n_freed += c->refs[c->table[seq][e]] == 1 ? 1 : 0;
    return PE_OK;
}

// ---- append bookkeeping
struct AppendPlan {
    int32_t seq;
    int32_t tok0;  // offset in the packed K/V
    int32_t n;
    int32_t need;  // pages to pop (including the copy-on-write page)
    bool cow;      // the partial last page is shared: copy it before writing
};

pe_status plan_append(const pe_cache *c, int32_t seq, int64_t n, AppendPlan *pl)
{
    pe_status s = check_seq(c, seq);
    if (s != PE_OK) return s;
    if (n < 0) return fail(PE_ERR_INVALID, "negative token count");
    const int64_t new_len = c->len[seq] + n;
    const int64_t pages = ceil_div(new_len, c->cfg.page_size);
    if (pages > c->cfg.max_pages_per_seq)
        return fail(PE_ERR_RANGE, "sequence %d would need %lld pages > max_pages_per_seq %d", seq,
                    static_cast<long long>(pages), c->cfg.max_pages_per_seq);
    if (new_len > INT32_MAX) return fail(PE_ERR_RANGE, "sequence length exceeds int32");
    pl->seq = seq;
    pl->n = static_cast<int32_t>(n);
    const std::vector<int32_t> &t = c->table[seq];
    pl->cow = n > 0 && c->len[seq] % c->cfg.page_size != 0 && c->refs[t.back()] > 1;
    pl->need = static_cast<int32_t>(pages - static_cast<int64_t>(t.size())) + (pl->cow ? 1 : 0);
    return PE_OK;
}

// A batch is planned as if its sequences were appended one after another: a
// copy-on-write planned for an earlier sequence drops one reference of the
// shared page, so a later sequence sharing that page may hold it alone by its
// turn and need no copy (and no extra page).
void settle_batch_cow(const pe_cache *c, std::vector<AppendPlan> &plans)
{
    std::vector<std::pair<int32_t, int32_t>> dropped;  // (page, references dropped by earlier plans)
    for (AppendPlan &pl : plans) {
        if (!pl.cow) continue;
        const int32_t pg = c->table[pl.seq].back();
        auto it = std::find_if(dropped.begin(), dropped.end(), [&](const auto &x) { return x.first == pg; });
        const int32_t d = it == dropped.end() ? 0 : it->second;
        if (c->refs[pg] - d <= 1) {
            pl.cow = false;
            pl.need -= 1;
            continue;
        }
        if (it == dropped.end()) dropped.emplace_back(pg, 1);
        else it->second += 1;
    }
}

// Copy-on-write of a sequence's shared, partially filled last page: pop a
// fresh page, copy the valid slots on the device, drop one reference.
pe_status apply_cow(pe_cache *c, int32_t seq, cudaStream_t st)
{
    j_seq(c, seq, static_cast<int32_t>(c->table[seq].size()) - 1);
    std::vector<int32_t> &t = c->table[seq];
    const int32_t src = t.back();
    const int32_t dst = free_pop(c);
    set_ref(c, dst, 1);
    set_ref(c, src, c->refs[src] - 1);
    t.back() = dst;
    if (injected_failure(c)) return launch_fault("copy-on-write");
    if (!c->host_only) {
        const int32_t slots = static_cast<int32_t>(c->len[seq] % c->cfg.page_size);
        int32_t *entry = c->d_table + static_cast<int64_t>(seq) * c->cfg.max_pages_per_seq + (t.size() - 1);
        cudaError_t e = launch_cow_copy(static_cast<uint4 *>(c->k_pool), static_cast<uint4 *>(c->v_pool), src, dst,
                                        slots, c->cfg.num_layers, c->cfg.num_kv_heads, c->cfg.page_size,
                                        c->cfg.head_dim / 8, c->cfg.num_pages, entry, st);
        if (e != cudaSuccess) return cuda_fail(e, "copy-on-write launch");
        c->launches++;
    }
    return PE_OK;
}

// Pops pages for every plan (the caller checked there are enough), then
// launches the copies.  Launches are cut so that each carries at most
// kMaxSegs segments and kAppendMaxPages new page ids.
pe_status apply_appends(pe_cache *c, const std::vector<AppendPlan> &plans, const void *K, const void *V,
                        int64_t n_total, cudaStream_t st)
{
    const int ps = c->cfg.page_size;
    std::vector<char> pbuf(sizeof(AppendParams));
    AppendParams *p = reinterpret_cast<AppendParams *>(pbuf.data());
    std::memset(p, 0, sizeof(AppendParams));
    {
        p->K = static_cast<const uint4 *>(K);
        p->V = static_cast<const uint4 *>(V);
        p->k_pool = static_cast<uint4 *>(c->k_pool);
        p->v_pool = static_cast<uint4 *>(c->v_pool);
        p->page_table = c->d_table;
        p->seq_len = c->d_len;
        p->L = c->cfg.num_layers;
        p->hkv = c->cfg.num_kv_heads;
        p->dvec = c->cfg.head_dim / 8;
        p->ps = ps;
        p->num_pages = c->cfg.num_pages;
        p->n_total = static_cast<int32_t>(n_total);
    }
    auto flush = [&]() -> pe_status {
        if (p->n_segs == 0) return PE_OK;
        p->seg_tokens = p->segs[p->n_segs - 1].cum0 + p->segs[p->n_segs - 1].n_tokens;
        const int64_t chunks = static_cast<int64_t>(p->L) * p->seg_tokens * p->hkv * p->dvec;
        if (injected_failure(c)) return launch_fault("append kernel");
        if (!c->host_only) {
            cudaError_t e = launch_append(*p, chunks, st);
            if (e != cudaSuccess) return cuda_fail(e, "append kernel launch");
            c->launches++;
        }
        p->n_segs = 0;
        return PE_OK;
    };
    int32_t pages_in_launch = 0;
    for (const AppendPlan &pl : plans) {
        // decided now, on the current references (the planners' page counts agree: settle_batch_cow)
        const std::vector<int32_t> &tt = c->table[pl.seq];
        if (pl.n > 0 && c->len[pl.seq] % ps != 0 && c->refs[tt.back()] > 1) {
            pe_status s = apply_cow(c, pl.seq, st);
            if (s != PE_OK) return s;
        }
        int32_t done = 0;
        if (pl.n > 0) j_seq(c, pl.seq, static_cast<int32_t>(c->table[pl.seq].size()));
        while (done < pl.n) {
            const int64_t len0 = c->len[pl.seq];
            std::vector<int32_t> &t = c->table[pl.seq];
            // tokens that fit without exceeding the page budget of this launch
            const int64_t room_pages = kAppendMaxPages - pages_in_launch;
            const int64_t have_slots = static_cast<int64_t>(t.size()) * ps - len0;  // free slots in last page
            int64_t take = pl.n - done;
            const int64_t max_take = have_slots + room_pages * ps;
            if (take > max_take) take = max_take;
            if (take <= 0 || p->n_segs == kMaxSegs) {
                pe_status s = flush();
                if (s != PE_OK) return s;
                pages_in_launch = 0;
                continue;
            }
            const int32_t first_new_lp = static_cast<int32_t>(t.size());
            const int32_t need = static_cast<int32_t>(ceil_div(len0 + take, ps) - static_cast<int64_t>(t.size()));
            {
                AppendSeg &sg = p->segs[p->n_segs];
                sg.tok0 = pl.tok0 + done;
                sg.cum0 = p->n_segs == 0 ? 0 : p->segs[p->n_segs - 1].cum0 + p->segs[p->n_segs - 1].n_tokens;
                sg.n_tokens = static_cast<int32_t>(take);
                sg.len0 = static_cast<int32_t>(len0);
                sg.first_new_lp = first_new_lp;
                sg.last_page = first_new_lp > 0 ? t[first_new_lp - 1] : -1;
                sg.new0 = pages_in_launch;
                sg.n_new = need;
                sg.table_row = pl.seq * c->cfg.max_pages_per_seq;
                sg.seq = pl.seq;
            }
            for (int32_t i = 0; i < need; ++i) {
                const int32_t pg = free_pop(c);
                set_ref(c, pg, 1);
                t.push_back(pg);
                p->new_pages[pages_in_launch + i] = pg;
            }
            pages_in_launch += need;
            p->n_segs++;
            c->len[pl.seq] = len0 + take;
            c->appended[pl.seq] += take;
            done += static_cast<int32_t>(take);
        }
    }
    return flush();
}

// ---- attention planning
struct AttnItem {
    int32_t seq;
    int32_t q_row0;
    int32_t n_q;
};

// Decode kernel launches (groups of kMaxSegs sequences).  Key splits: about two
// waves of the CTAs that fit on the GPU at once, at least 2 tiles per split;
// "splitkv" = 0 keeps one split, "num_splits" fixes the count.
pe_status run_decode(pe_cache *c, const std::vector<AttnItem> &items, int32_t layer, const void *Q, void *out,
                     int32_t hq, float scale, cudaStream_t st)
{
    const pe_cache_config &cf = c->cfg;
    const int hkv = cf.num_kv_heads;
    const int d = cf.head_dim;
    const int g = hq / hkv;
    // tensor-core form (128-key tiles, one CTA per SM) unless "decode_kernel" = 2: CUDA cores (64-key tiles)
    const bool tc = (d == 128 || d == 64) && c->decode_kernel == 1;
    const int64_t tile_keys = tc ? 128 : kDecKeys;
    std::vector<char> pbuf(sizeof(DecodeParams));
    DecodeParams &p = *reinterpret_cast<DecodeParams *>(pbuf.data());
    for (size_t lo = 0; lo < items.size(); lo += kMaxSegs) {
        const size_t hi = std::min(items.size(), lo + kMaxSegs);
        if (tc) {
            // chunks of at most 8 tiles; CTAs (one per SM) take them from a counter
            std::memset(&p, 0, sizeof p);
            int64_t tiles = 0, max_rows = 1, max_tiles = 1;
            for (size_t i = lo; i < hi; ++i) {
                const int64_t nt = ceil_div(c->len[items[i].seq], 128);
                tiles += nt * hkv;
                max_tiles = std::max(max_tiles, nt);
                max_rows = std::max<int64_t>(max_rows, static_cast<int64_t>(items[i].n_q) * g);
            }
            const int rb = max_rows <= 4 ? 4 : (max_rows <= 8 ? 8 : 16);
            // chunks of ceil(tiles / (k x SMs)) tiles, 1..8 (k = "decode_chunks_per_sm", 3 by default)
            const int64_t k_per_sm = c->dec_chunks_per_sm;
            int64_t force = std::min<int64_t>(8, std::max<int64_t>(1, ceil_div(tiles, k_per_sm * c->num_sms)));
            if (c->splitkv == 1 && c->num_splits > 0) force = std::min<int64_t>(8, ceil_div(max_tiles, c->num_splits));
            // Chunk ids, longest first: every item's full chunks (sequence-major, kv-head next), then the
            // items' shorter remainder chunks, sequences by decreasing remainder length (ties: batch
            // order), so that the chunks the CTAs take last are the shortest.
            int64_t chunks = 0;
            bool any_split = false;
            for (int pass = 0;; ++pass) {
                chunks = 0;
                p.n_seqs = 0;
                any_split = false;
                int32_t rems[kMaxSegs];  // sequences with a remainder chunk
                int32_t rem_tiles[kMaxSegs];
                int n_rem = 0;
                for (size_t i = lo; i < hi; ++i) {
                    const AttnItem &it = items[i];
                    const int64_t nt = ceil_div(c->len[it.seq], 128);
                    int64_t ct = pass > 0 ? 8 : force;  // on a second pass the partials must fit: longest chunks
                    DecodeSeq &q = p.seqs[p.n_seqs];
                    q.table_row = it.seq * cf.max_pages_per_seq;
                    q.n_pages = static_cast<int32_t>(c->table[it.seq].size());
                    q.q_row0 = it.q_row0;
                    q.n_q = it.n_q;
                    q.n_keys = static_cast<int32_t>(c->len[it.seq]);
                    q.tile0 = static_cast<int32_t>(chunks);
                    q.cta0 = static_cast<int32_t>(ct);
                    q.rem0 = -1;
                    const int64_t cpi = ceil_div(nt, ct);
                    q.n_splits = static_cast<int32_t>(cpi);
                    any_split = any_split || cpi > 1;
                    chunks += (nt / ct) * hkv;
                    if (nt % ct) {  // insertion by decreasing remainder length, stable
                        int j = n_rem++;
                        for (; j > 0 && rem_tiles[j - 1] < nt % ct; --j) {
                            rems[j] = rems[j - 1];
                            rem_tiles[j] = rem_tiles[j - 1];
                        }
                        rems[j] = p.n_seqs;
                        rem_tiles[j] = static_cast<int32_t>(nt % ct);
                    }
                    p.n_seqs++;
                }
                p.full_chunks = static_cast<int32_t>(std::min<int64_t>(chunks, INT32_MAX));
                for (int j = 0; j < n_rem; ++j) {
                    p.seqs[rems[j]].rem0 = static_cast<int32_t>(std::min<int64_t>(chunks, INT32_MAX));
                    p.rem_seq[j] = rems[j];
                    chunks += hkv;
                }
                if (chunks * rb * (d + 2) * 4 <= c->ws_bytes || pass > 0) break;
            }
            if (chunks * rb * (d + 2) * 4 > c->ws_bytes || chunks > INT32_MAX)
                return fail(PE_ERR_RANGE, "decode partials exceed the workspace (%lld chunks)", static_cast<long long>(chunks));
            p.split_tiles = 0;
            p.total_tiles = static_cast<int32_t>(chunks);
            p.total_ctas = static_cast<int32_t>(std::min<int64_t>(chunks, c->num_sms));
            p.page_table = c->d_table;
            p.q = Q;
            p.out = out;
            p.k_pool = c->k_pool;
            p.v_pool = c->v_pool;
            p.part = c->d_ws;
            p.tickets = c->d_tickets;
            p.sched = c->d_tickets + kMaxSegs * hkv;
            p.status = c->d_status;
            p.hq = hq;
            p.hkv = hkv;
            p.group = g;
            p.layer = layer;
            p.num_pages = cf.num_pages;
            p.ps = cf.page_size;
            p.oob_row = static_cast<int32_t>(c->pool_rows);
            p.scale_log2 = scale * 1.4426950408889634f;
            c->last_split = any_split ? 1 : 0;
            c->last_splits = p.seqs[0].n_splits;
            c->last_ctas = p.total_ctas;
            if (injected_failure(c)) return launch_fault("decode attention");
            cudaError_t e = launch_decode_attn(d, rb, true, c->tm_kd, c->tm_vd, p, st);
            if (e != cudaSuccess) return cuda_fail(e, "decode attention launch");
            c->launches++;
            continue;
        }
        int64_t max_rows = 1, work = 0, max_tiles = 1;
        for (size_t i = lo; i < hi; ++i) {
            const int64_t tiles = ceil_div(c->len[items[i].seq], tile_keys);
            max_rows = std::max<int64_t>(max_rows, static_cast<int64_t>(items[i].n_q) * g);
            max_tiles = std::max(max_tiles, tiles);
            work += tiles * hkv;
        }
        const int rb = max_rows <= 4 ? 4 : (max_rows <= 8 ? 8 : 16);
        const int64_t resident = static_cast<int64_t>(c->num_sms) * (!tc && rb <= 8 ? 2 : 1);
        auto ctas_for = [&](int64_t stile) {
            int64_t n = 0;
            for (size_t i = lo; i < hi; ++i) n += ceil_div(ceil_div(c->len[items[i].seq], tile_keys), stile) * hkv;
            return n;
        };
        // about two waves of resident CTAs, never a third one started by a few stragglers
        int64_t split_tiles = std::max<int64_t>(2, ceil_div(work, 2 * resident));
        while (split_tiles < max_tiles && ctas_for(split_tiles) > 2 * resident) ++split_tiles;
        if (c->splitkv == 0) split_tiles = max_tiles;
        if (c->splitkv != 0 && c->num_splits > 0) split_tiles = std::max<int64_t>(1, ceil_div(max_tiles, c->num_splits));
        if (c->splitkv == 1 && c->num_splits == 0 && split_tiles >= max_tiles && max_tiles > 1)
            split_tiles = ceil_div(max_tiles, 2);
        split_tiles = std::min(split_tiles, max_tiles);
        for (;;) {
            std::memset(&p, 0, sizeof p);
            int32_t cta = 0;
            bool any_split = false;
            for (size_t i = lo; i < hi; ++i) {
                const AttnItem &it = items[i];
                DecodeSeq &q = p.seqs[p.n_seqs++];
                q.table_row = it.seq * cf.max_pages_per_seq;
                q.n_pages = static_cast<int32_t>(c->table[it.seq].size());
                q.q_row0 = it.q_row0;
                q.n_q = it.n_q;
                q.n_keys = static_cast<int32_t>(c->len[it.seq]);
                q.n_splits = static_cast<int32_t>(ceil_div(ceil_div(c->len[it.seq], tile_keys), split_tiles));
                q.cta0 = cta;
                cta += q.n_splits * hkv;
                any_split = any_split || q.n_splits > 1;
            }
            p.total_ctas = cta;
            const int64_t need = static_cast<int64_t>(cta) * rb * (d + 2) * 4;
            if (!any_split || need <= c->ws_bytes) break;
            split_tiles *= 2;  // partials do not fit the workspace: fewer splits
        }
        p.page_table = c->d_table;
        p.q = Q;
        p.out = out;
        p.k_pool = c->k_pool;
        p.v_pool = c->v_pool;
        p.part = c->d_ws;
        p.tickets = c->d_tickets;
        p.status = c->d_status;
        p.hq = hq;
        p.hkv = hkv;
        p.group = g;
        p.layer = layer;
        p.num_pages = cf.num_pages;
        p.ps = cf.page_size;
        p.oob_row = static_cast<int32_t>(c->pool_rows);
        p.split_tiles = static_cast<int32_t>(split_tiles);
        p.scale_log2 = scale * 1.4426950408889634f;
        c->last_split = p.seqs[0].n_splits > 1 ? 1 : 0;
        c->last_splits = p.seqs[0].n_splits;
        c->last_ctas = p.total_ctas;
        if (injected_failure(c)) return launch_fault("decode attention");
        cudaError_t e = launch_decode_attn(d, rb, tc, c->tm_kd, c->tm_vd, p, st);
        if (e != cudaSuccess) return cuda_fail(e, "decode attention launch");
        c->launches++;
    }
    return PE_OK;
}

// ---- persistent stream-K plan of one launch group (replay_attn_sk_kernel)
// Units are (sequence, kv-head, q-tile pair) in the kernel's order: sequences
// as given (longest first), kv-head fastest, pairs heaviest first.  A unit
// costs its key tiles plus kSkUnitCost for loading Q and writing the output;
// CTA c takes the work between boundaries c and c + 1 at c / P of the total.
// With cuts allowed a boundary falls inside a unit (at a key tile, each piece
// at least kSkMinPiece tiles), else at the unit boundary nearest to it; cuts
// are kept when the cost model (the busiest CTA, plus the merge of the last
// parts at the end of the kernel) prefers them by 5 %, or always with
// "splitkv" = 1.
constexpr double kSkUnitCost = 2.0;
constexpr int kSkMinPiece = 2;

struct SkBound {
    int32_t u, t;  // unit and key tile (t = 0: the start of unit u)
    bool operator==(const SkBound &o) const { return u == o.u && t == o.t; }
};

pe_status plan_sk(pe_cache *c, const std::vector<AttnItem> &order, size_t lo, size_t hi, int32_t layer, void *out,
                  int32_t hq, float scale, SkParams &P, std::vector<int32_t> *unit_tiles = nullptr)
{
    const pe_cache_config &cf = c->cfg;
    const int hkv = cf.num_kv_heads, d = cf.head_dim, g = hq / hkv, bmq = kBM / g;
    std::memset(&P, 0, sizeof P);
    AttnParams &p = P.a;
    p.page_table = c->d_table;
    p.out = out;
    p.status = c->d_status;
    p.hq = hq;
    p.hkv = hkv;
    p.group = g;
    p.layer = layer;
    p.num_pages = cf.num_pages;
    p.ps = cf.page_size;
    p.oob_row = static_cast<int32_t>(c->pool_rows);
    p.scale_log2 = scale * 1.4426950408889634f;
    std::vector<int32_t> n_all;   // key tiles per unit
    std::vector<double> cum{0.0};  // cost before each unit
    for (size_t i = lo; i < hi; ++i) {
        const AttnItem &it = order[i];
        AttnSeq &q = p.seqs[p.n_seqs++];
        q.table_row = it.seq * cf.max_pages_per_seq;
        q.n_pages = static_cast<int32_t>(c->table[it.seq].size());
        q.q_row0 = it.q_row0;
        q.n_q = it.n_q;
        q.n_keys = static_cast<int32_t>(c->len[it.seq]);
        q.n_qtiles = static_cast<int32_t>(ceil_div(static_cast<int64_t>(it.n_q) * g, kBM));
        q.pair_top = (q.n_qtiles + 1) / 2;
        q.n_splits = 1;
        q.item0 = static_cast<int32_t>(n_all.size());
        for (int32_t local = 0; local < q.pair_top * hkv; ++local) {
            const int32_t pair = q.pair_top - 1 - local / hkv;
            const int32_t qt_last = std::min(2 * pair + 1, q.n_qtiles - 1);
            const int64_t q_last = std::min<int64_t>((qt_last + 1) * static_cast<int64_t>(bmq), it.n_q) - 1;
            const int32_t n = static_cast<int32_t>(ceil_div(c->len[it.seq] - it.n_q + q_last + 1, kBN));
            n_all.push_back(n);
            cum.push_back(cum.back() + n + kSkUnitCost);
        }
    }
    const int32_t U = static_cast<int32_t>(n_all.size());
    auto unit_at = [&](double x) {  // the unit whose cost range holds x
        return static_cast<int32_t>(std::upper_bound(cum.begin(), cum.end(), x) - cum.begin()) - 1;
    };

    // A plan for nc CTAs.  Whole units first, in lockstep rounds: in round r CTA k takes unit
    // r nc + k (k reversed in odd rounds), so the CTAs running at once work on neighbouring units
    // and share their K/V in L2.  The last one to two rounds of units (the tail) are spread so that
    // every CTA ends with about the same total: CTA k's contiguous tail stretch is what its rounds
    // lack of the mean.  b[k] = (unit, key tile) where CTA k's tail stretch starts, b[nc] = (U, 0).
    struct Plan {
        int32_t nc = 1, R = 0;
        std::vector<double> own;
        std::vector<SkBound> b;
    };
    auto make = [&](int32_t nc, bool cuts, Plan &pl) {
        pl.nc = nc;
        pl.R = U >= 2 * nc ? U / nc - 1 : 0;
        const int32_t T0 = pl.R * nc;  // first tail unit
        pl.own.assign(nc, 0.0);
        for (int32_t r = 0; r < pl.R; ++r)
            for (int32_t k = 0; k < nc; ++k)
                pl.own[k] += n_all[r * nc + ((r & 1) ? nc - 1 - k : k)] + kSkUnitCost;
        const double W = cum.back() - cum[T0];
        const double mean = cum.back() / nc;
        std::vector<double> want(nc), pos(nc + 1, 0.0);
        double sum_want = 0.0;
        for (int32_t k = 0; k < nc; ++k) sum_want += (want[k] = std::max(0.0, mean - pl.own[k]));
        for (int32_t k = 0; k < nc; ++k) pos[k + 1] = pos[k] + (sum_want > 0 ? want[k] * W / sum_want : W / nc);
        pl.b.assign(nc + 1, SkBound{T0, 0});
        pl.b[nc] = SkBound{U, 0};
        for (int32_t k = 1; k < nc; ++k) {
            const double x = cum[T0] + pos[k];
            SkBound bd{U, 0};
            if (x < cum.back()) {
                const int32_t u = std::min(unit_at(x), U - 1);
                const double off = x - cum[u];
                const int32_t t = static_cast<int32_t>(std::lround(off - kSkUnitCost));
                bd = SkBound{u, 0};
                if (cuts && t >= kSkMinPiece && n_all[u] - t >= kSkMinPiece) bd.t = t;
                else if (off > 0.5 * (n_all[u] + kSkUnitCost)) bd = SkBound{u + 1, 0};
            }
            const SkBound &prev = pl.b[k - 1];
            if (bd.u < prev.u || (bd.u == prev.u && bd.t < prev.t)) bd = prev;  // an empty stretch
            pl.b[k] = bd;
        }
    };
    // the busiest CTA: its rounds plus its tail stretch (a cut piece pays its own set-up)
    auto busiest = [&](const Plan &pl) {
        auto at = [&](const SkBound &x) {
            return (x.u < U ? cum[x.u] : cum.back()) + (x.t > 0 ? kSkUnitCost + x.t : 0.0);
        };
        double worst = 0.0;
        for (int32_t k = 0; k < pl.nc; ++k) {
            double tail = at(pl.b[k + 1]) - at(pl.b[k]);
            if (tail > 0 && pl.b[k].t > 0) tail += kSkUnitCost;
            worst = std::max(worst, pl.own[k] + tail);
        }
        return worst;
    };
    // cut units of a plan: slots and part counts; false when the partials do not fit
    std::vector<int32_t> slot_of;
    std::vector<int32_t> cuts_in;  // interior boundaries per cut unit
    int32_t n_slots = 0, max_parts = 1;
    auto slots_for = [&](const std::vector<SkBound> &bb) {
        slot_of.assign(U, -1);
        cuts_in.clear();
        n_slots = 0;
        max_parts = 1;
        for (size_t i = 0; i < bb.size(); ++i) {
            const SkBound &x = bb[i];
            // an empty stretch repeats its boundary: count each cut once
            if (x.t <= 0 || x.u >= U || (i > 0 && bb[i - 1] == x)) continue;
            if (slot_of[x.u] < 0) {
                slot_of[x.u] = n_slots++;
                cuts_in.push_back(0);
            }
            cuts_in[slot_of[x.u]] += 1;
        }
        for (int32_t k = 0; k < n_slots; ++k) max_parts = std::max(max_parts, cuts_in[k] + 1);
        const int64_t rows = static_cast<int64_t>(n_slots) * max_parts * 2 * kBM;
        return n_slots <= kMaxSkCtas && max_parts <= 32 && rows * (static_cast<int64_t>(d) * 4 + 4) <= c->ws_bytes;
    };

    // CTAs: one per SM, fewer when the work is small (about 3 cost units each at least)
    int32_t n_cta = static_cast<int32_t>(std::min<int64_t>(
        std::min<int64_t>(c->num_sms, kMaxSkCtas), std::max<int64_t>(1, static_cast<int64_t>(cum.back() / 3.0))));
    if (c->attn_ctas > 0) n_cta = std::min(c->attn_ctas, kMaxSkCtas);
    Plan whole, cut;
    make(n_cta, false, whole);
    bool cuts = false;
    if (c->splitkv != 0) {
        // fewer CTAs when a unit would be cut into more than 32 parts or the partials overflow the workspace
        for (int32_t nc = n_cta; nc >= 2; nc = std::min(nc - 1, nc * 31 / std::max<int32_t>(max_parts, 32))) {
            make(nc, true, cut);
            if (!slots_for(cut.b)) continue;
            if (n_slots > 0 && (c->splitkv == 1 || busiest(cut) + 2.0 < 0.95 * busiest(whole))) cuts = true;
            break;
        }
    }
    const Plan &pl = cuts ? cut : whole;
    if (!cuts) {
        n_slots = 0;
        max_parts = 1;
    }
    P.n_ctas = pl.nc;
    P.rounds = pl.R;
    P.n_slots = n_slots;
    P.max_parts = max_parts;
    if (cuts) {
        for (int32_t u = 0; u < U; ++u)
            if (slot_of[u] >= 0) P.slots[slot_of[u]] = SkSlot{u, cuts_in[slot_of[u]] + 1};
        p.part_o = c->d_ws;  // (null on a host-only cache, which only plans)
        p.part_lse = c->d_ws ? c->d_ws + static_cast<int64_t>(n_slots) * max_parts * 2 * kBM * d : nullptr;
    }
    P.tickets = c->d_tickets ? c->d_tickets + kMaxSegs * hkv + 2 : nullptr;
    for (int32_t k = 0; k < pl.nc; ++k) {
        const SkBound &a = pl.b[k], &z = pl.b[k + 1];
        SkCta &w = P.cta[k];
        w.slot0 = w.slot1 = -1;
        w.part0 = w.part1 = 0;
        if (a == z) {  // no tail stretch
            w.u0 = 1;
            w.u1 = 0;
            w.t0 = w.t1 = 0;
            continue;
        }
        w.u0 = a.u;
        w.t0 = a.t;
        w.u1 = z.u;
        w.t1 = z.t;
        if (cuts && slot_of[a.u] >= 0) {
            w.slot0 = slot_of[a.u];
            int32_t part = 0;  // interior boundaries of unit a.u at or before tile a.t, each counted once
            for (size_t i = 0; i < pl.b.size(); ++i) {
                const SkBound &x = pl.b[i];
                if (x.u == a.u && x.t > 0 && x.t <= a.t && !(i > 0 && pl.b[i - 1] == x)) ++part;
            }
            w.part0 = part;
        }
        if (cuts && z.u != a.u && z.t > 0) {
            w.slot1 = slot_of[z.u];
            w.part1 = 0;
        }
    }
    if (unit_tiles) *unit_tiles = n_all;
    return PE_OK;
}

// Plan query (pe_attn_plan_launches): one launch as words -- kind, split,
// CTAs, combine rows, split_tiles, pairs_fastest, n_seqs, then per sequence
// seq, item0, n_q, n_keys, n_qtiles, n_splits, pair_top, part_row0, comb0,
// q_row0.
void record_launch(const pe_cache *c, int32_t kind, bool split, const AttnParams &p, int32_t ctas)
{
    std::vector<int64_t> &r = *c->plan_rec;
    const int64_t head[7] = {kind, split ? 1 : 0, ctas, p.total_comb, p.split_tiles, p.pairs_fastest, p.n_seqs};
    r.insert(r.end(), head, head + 7);
    for (int32_t i = 0; i < p.n_seqs; ++i) {
        const AttnSeq &q = p.seqs[i];
        const int64_t w[10] = {q.table_row / c->cfg.max_pages_per_seq, q.item0, q.n_q, q.n_keys, q.n_qtiles,
                               q.n_splits, q.pair_top, q.part_row0, q.comb0, q.q_row0};
        r.insert(r.end(), w, w + 10);
    }
}

pe_status run_attention(pe_cache *c, const std::vector<AttnItem> &items, int32_t layer, const void *Q,
                        int64_t q_rows, void *out, int32_t hq, float scale, cudaStream_t st)
{
    const pe_cache_config &cf = c->cfg;
    const int hkv = cf.num_kv_heads;
    const int d = cf.head_dim;
    const int g = hq / hkv;
    const int bmq = kBM / g;
    // Items whose queries pack into at most kDecMaxRows rows per kv-head take
    // the decode kernel; the rest the tensor-core kernel.
    std::vector<AttnItem> order, dec;
    for (const AttnItem &it : items) {
        if (it.n_q <= 0) continue;
        // (the tcgen05 decode kernel always splits keys across CTAs: "splitkv" = 0 keeps the prefill kernel)
        const bool tc_nosplit = c->decode_kernel == 1 && c->splitkv == 0;
        if (c->decode_kernel && static_cast<int64_t>(it.n_q) * g <= kDecMaxRows && (d == 64 || d == 128) && !tc_nosplit)
            dec.push_back(it);
        else
            order.push_back(it);
    }
    if (!dec.empty() && c->plan_rec) {  // plan query: the decode kernel's sequences, not planned here
        std::vector<char> dbuf(sizeof(AttnParams));
        AttnParams &dp = *reinterpret_cast<AttnParams *>(dbuf.data());
        for (size_t lo = 0; lo < dec.size(); lo += kMaxSegs) {
            std::memset(&dp, 0, sizeof dp);
            for (size_t i = lo; i < std::min(dec.size(), lo + kMaxSegs); ++i) {
                AttnSeq &q = dp.seqs[dp.n_seqs++];
                q.table_row = dec[i].seq * cf.max_pages_per_seq;
                q.n_q = dec[i].n_q;
                q.n_keys = static_cast<int32_t>(c->len[dec[i].seq]);
                q.q_row0 = dec[i].q_row0;
            }
            record_launch(c, 3, false, dp, 0);
        }
    } else if (!dec.empty()) {
        pe_status s = run_decode(c, dec, layer, Q, out, hq, scale, st);
        if (s != PE_OK) return s;
    }
    std::stable_sort(order.begin(), order.end(), [&](const AttnItem &a, const AttnItem &b) {
        return c->len[a.seq] > c->len[b.seq];
    });
    if (order.empty()) return PE_OK;

    CUtensorMap tm_q, tm_o;  // Q, and the output as a map of the same shape (TMA stores of full q-tiles)
    const bool rec = c->plan_rec != nullptr;  // a plan query: no tensors, no launches
    pe_status s = PE_OK;
    if (!rec && (s = encode_q(&tm_q, Q, q_rows, hq, d, g)) != PE_OK) return s;
    if (!rec && (s = encode_q(&tm_o, out, q_rows, hq, d, g)) != PE_OK) return s;

    // split-KV decision over the whole launch group; plan_est: the cost model's time of the plan
    double plan_est = 0.0;
    // time of one key tile per CTA in the cost models: about 1.5 us, compute- or HBM-bound alike; 1 us at
    // d = 64, whose next S GEMM overlaps the softmax
    const double tile_s = d == 64 ? 1.0e-6 : 1.5e-6;
    // splitkv: the "splitkv" option's value for this plan (-1 auto, 0 never, 1 always)
    auto plan_group = [&](size_t lo, size_t hi, AttnParams &p, bool &split, int splitkv) -> pe_status {
        // C CTAs (pairs of q-tiles x kv-heads), W key tiles per CTA on average.
        int64_t C = 0, tiles = 0, rows = 0, valid_rows = 0, max_tiles = 0;
        for (size_t i = lo; i < hi; ++i) {
            const AttnItem &it = order[i];
            const int64_t len = c->len[it.seq];
            const int64_t nqt = ceil_div(static_cast<int64_t>(it.n_q) * g, kBM);
            for (int64_t pp = 0; pp < ceil_div(nqt, 2); ++pp) {
                const int64_t q_last = std::min<int64_t>((std::min(2 * pp + 1, nqt - 1) + 1) * bmq, it.n_q) - 1;
                tiles += ceil_div(len - it.n_q + q_last + 1, kBN) * hkv;
            }
            C += ceil_div(nqt, 2) * hkv;
            rows += nqt * hkv * kBM;                               // workspace slots (whole tiles)
            valid_rows += static_cast<int64_t>(it.n_q) * g * hkv;  // partial rows written and read
            max_tiles = std::max(max_tiles, ceil_div(len, kBN));
        }
        // Estimated time with s key splits: the CTAs run in ceil(C s / N) waves of
        // (W/s + 2) tile times, and never faster than the longest CTA
        // (max_tiles/s + 2); splits add their fp32 partials' HBM round trip and
        // a combine launch.
        const double W = C > 0 ? static_cast<double>(tiles) / C : 0.0;
        const int64_t row_bytes = static_cast<int64_t>(d) * 4 + 4;
        // (the combine kernel is a programmatic dependent of the attention grid: about 5 us more, measured
        // on the 1-agent d = 64 launch: 5 splits + combine 14.0 us, one pass 13.0 us)
        auto cost = [&](int64_t sp) {
            const double waves = std::ceil(static_cast<double>(C * sp) / c->num_sms);
            double t = std::max(waves * (W / sp + 2.0), static_cast<double>(max_tiles) / sp + 2.0) * tile_s;
            if (sp > 1) t += static_cast<double>(valid_rows * sp * row_bytes * 2) / 6.0e12 + 5e-6;
            return t;
        };
        int64_t best = 1;
        if (splitkv != 0) {
            // at least 4 key tiles per split, unless the CTAs are too few to fill the SMs
            int64_t s_max = std::min<int64_t>(128, std::max<int64_t>(1, max_tiles / 4));
            if (C > 0 && C * 2 <= c->num_sms) s_max = std::max(s_max, std::min<int64_t>(max_tiles, c->num_sms / C));
            double best_t = splitkv == 1 ? 1e30 : cost(1);
            for (int64_t sp = 2; sp <= s_max; ++sp) {
                if (rows * sp * row_bytes > c->ws_bytes) break;
                const double t = cost(sp);
                if (t < best_t) { best_t = t; best = sp; }
            }
            if (splitkv == -1 && best > 1 && best_t > 0.95 * cost(1)) best = 1;  // keep the single pass unless clearly faster
        }
        if (splitkv != 0 && c->num_splits > 0) best = c->num_splits;
        plan_est = cost(best);
        int split_tiles = static_cast<int>(max_tiles);
        split = best > 1 || splitkv == 1;
        if (split) split_tiles = static_cast<int>(std::max<int64_t>(1, ceil_div(max_tiles, std::max<int64_t>(best, 1))));
        std::memset(&p, 0, sizeof p);
        p.page_table = c->d_table;
        p.out = out;
        p.status = c->d_status;
        p.hq = hq;
        p.hkv = hkv;
        p.group = g;
        p.layer = layer;
        p.num_pages = cf.num_pages;
        p.ps = cf.page_size;
        p.oob_row = static_cast<int32_t>(c->pool_rows);
        p.scale_log2 = scale * 1.4426950408889634f;
        p.next_stride = c->num_sms;  // one CTA per SM: CTA b's successor on its SM is about b + SMs
        for (;;) {
            int32_t item = 0, comb = 0;
            int64_t prow = 0;
            p.n_seqs = 0;
            for (size_t i = lo; i < hi; ++i) {
                const AttnItem &it = order[i];
                AttnSeq &q = p.seqs[p.n_seqs++];
                q.table_row = it.seq * cf.max_pages_per_seq;
                q.n_pages = static_cast<int32_t>(c->table[it.seq].size());
                q.q_row0 = it.q_row0;
                q.n_q = it.n_q;
                q.n_keys = static_cast<int32_t>(c->len[it.seq]);
                q.n_qtiles = static_cast<int32_t>(ceil_div(static_cast<int64_t>(it.n_q) * g, kBM));
                q.pair_top = (q.n_qtiles + 1) / 2;
                const int64_t ktiles = ceil_div(c->len[it.seq], kBN);
                q.n_splits = split ? static_cast<int32_t>(ceil_div(ktiles, split_tiles)) : 1;
                q.item0 = item;
                q.part_row0 = prow;
                q.comb0 = comb;
                item += ((q.n_qtiles + 1) / 2) * hkv * q.n_splits;
                if (split) {
                    prow += static_cast<int64_t>(q.n_qtiles) * hkv * q.n_splits * kBM;
                    comb += q.n_qtiles * hkv * kBM;
                }
            }
            p.total_items = item;
            p.total_comb = comb;
            // launches of many waves number each sequence's items pairs fastest, so that the CTAs resident
            // at once share one or two kv-heads' keys in L2 (long suffix: DRAM reads 4.6 -> 1.4 GB per
            // launch); with fewer waves, every kv-head's heaviest pairs first keeps the last wave short
            p.pairs_fastest = c->attn_order >= 0 ? c->attn_order : (item >= 32 * static_cast<int64_t>(c->num_sms) ? 1 : 0);
            p.split_tiles = split_tiles;
            if (!split) break;
            const int64_t need = prow * (static_cast<int64_t>(d) * 4 + 4);
            if (need <= c->ws_bytes) {
                p.part_o = c->d_ws;
                p.part_lse = c->d_ws ? c->d_ws + prow * d : nullptr;  // (null on a host-only cache)
                break;
            }
            if (split_tiles >= max_tiles) {
                split = false;  // cannot fit any split into the workspace: run unsplit
                continue;
            }
            split_tiles *= 2;
        }
        (void)bmq;
        return PE_OK;
    };

    // Tail launch for a launch group of one sequence (one long agent): when its CTAs leave the last
    // wave mostly empty, the lightest q-tile pairs (the last CTAs in the heaviest-first order) move
    // to a second launch that splits their keys over every SM; the first launch then fills whole
    // waves.  Chosen by the same cost model, when it beats the group's plan by 5 %.
    struct TailPlan {
        int64_t pairs = 0, splits = 0, split_tiles = 0, qtiles = 0;
    };
    auto plan_tail = [&](const AttnItem &it, TailPlan &tp) -> bool {
        const int64_t len = c->len[it.seq];
        const int64_t nqt = ceil_div(static_cast<int64_t>(it.n_q) * g, kBM);
        const int64_t n_pairs = ceil_div(nqt, 2);
        const int64_t C = n_pairs * hkv, N = c->num_sms;
        if (C <= N || C % N == 0) return false;
        const int64_t cut = ceil_div(C % N, hkv);  // lightest pairs moved to the tail launch
        if (cut >= n_pairs) return false;
        const int64_t ktiles = ceil_div(len, kBN);
        double wa = 0.0, wb = 0.0;  // mean key tiles of a pair in the first / tail launch
        for (int64_t pp = 0; pp < n_pairs; ++pp) {
            const int64_t q_last = std::min<int64_t>((std::min(2 * pp + 1, nqt - 1) + 1) * bmq, it.n_q) - 1;
            const double t = static_cast<double>(ceil_div(len - it.n_q + q_last + 1, kBN));
            (pp < cut ? wb : wa) += t;
        }
        wa /= static_cast<double>(n_pairs - cut);
        wb /= static_cast<double>(cut);
        const int64_t qt_b = std::min<int64_t>(nqt, 2 * cut);
        const int64_t row_bytes = static_cast<int64_t>(d) * 4 + 4;
        const double t_a = std::ceil(static_cast<double>(C - cut * hkv) / N) * (wa + 2.0) * tile_s;
        double best_t = 1e30;
        for (int64_t sp = 2; sp <= std::min<int64_t>(128, std::max<int64_t>(2, ktiles / 4)); ++sp) {
            if (qt_b * hkv * sp * kBM * row_bytes > c->ws_bytes) break;
            const double waves = std::ceil(static_cast<double>(cut * hkv * sp) / N);
            const double t = t_a + waves * (wb / sp + 2.0) * tile_s +
                             static_cast<double>(qt_b * hkv * kBM * sp * row_bytes * 2) / 6.0e12 + 10e-6;
            if (t < best_t) {
                best_t = t;
                tp.splits = sp;
            }
        }
        if (tp.splits == 0 || best_t > 0.95 * plan_est) return false;
        tp.pairs = cut;
        tp.qtiles = qt_b;
        tp.split_tiles = ceil_div(ktiles, tp.splits);
        return true;
    };

    std::vector<char> pbuf(sizeof(AttnParams));
    AttnParams &p = *reinterpret_cast<AttnParams *>(pbuf.data());
    std::vector<char> sbuf;
    for (size_t lo = 0; lo < order.size(); lo += kMaxSegs) {
        const size_t hi = std::min(order.size(), lo + kMaxSegs);
        bool split = false;
        s = plan_group(lo, hi, p, split, c->splitkv);
        if (s != PE_OK) return s;
        TailPlan tp;
        const bool tail = hi - lo == 1 && c->splitkv == -1 && c->num_splits == 0 && plan_tail(order[lo], tp);
        // The persistent stream-K kernel where the one-item plan leaves SMs idle (it needs key splits
        // or a tail launch) and its units fill between a quarter of the SMs and two waves: one CTA
        // per SM, whole units in rounds, the rest cut into equal stretches.  Elsewhere the one-item
        // kernel, whose tile loop runs a little faster (measured: short suffix 195 -> 184 us and
        // tau/T 0.9 311 -> 303 us with the persistent kernel; tau/T 0.7 716 -> 749 us and the
        // 8-unit tiny launch 14 -> 16 us without it).
        int64_t units = 0;
        for (size_t i = lo; i < hi; ++i)
            units += ceil_div(ceil_div(static_cast<int64_t>(order[i].n_q) * g, kBM), 2) * hkv;
        const bool sk_fits = 4 * units >= c->num_sms && units < 2 * static_cast<int64_t>(c->num_sms);
        const bool sk = c->num_splits == 0 &&
                        (c->attn_kernel == 2 || (c->attn_kernel == 1 && (split || tail) && sk_fits));
        if (sk) {
            if (sbuf.empty()) sbuf.resize(sizeof(SkParams));
            SkParams &P = *reinterpret_cast<SkParams *>(sbuf.data());
            if ((s = plan_sk(c, order, lo, hi, layer, out, hq, scale, P)) != PE_OK) return s;
            c->last_split = P.n_slots > 0 ? 1 : 0;
            c->last_splits = P.max_parts;
            c->last_ctas = P.n_ctas;
            if (rec) {
                record_launch(c, 2, P.n_slots > 0, P.a, P.n_ctas);
                continue;
            }
            if (injected_failure(c)) return launch_fault("replay attention");
            cudaError_t e = launch_replay_attn_sk(d, tm_q, c->tm_k, c->tm_v, P, st);
            if (e != cudaSuccess) return cuda_fail(e, "replay attention launch");
            c->launches++;
            continue;
        }
        if (tail && split) {  // the first launch runs unsplit: re-plan the group without splits
            s = plan_group(lo, hi, p, split, 0);
            if (s != PE_OK) return s;
        }
        if (tail) {
            p.total_items -= static_cast<int32_t>(tp.pairs * hkv);  // pairs [cut, n_pairs), heaviest first
            p.pairs_fastest =
                c->attn_order >= 0 ? c->attn_order : (p.total_items >= 32 * static_cast<int64_t>(c->num_sms) ? 1 : 0);
        }
        c->last_split = split || tail ? 1 : 0;
        c->last_splits = tail ? static_cast<int32_t>(tp.splits) : (split ? p.seqs[0].n_splits : 1);
        c->last_ctas = p.total_items + (tail ? static_cast<int32_t>(tp.pairs * hkv * tp.splits) : 0);
        if (rec) record_launch(c, 0, split, p, p.total_items);
        if (injected_failure(c)) return launch_fault("replay attention");
        cudaError_t e = rec ? cudaSuccess : launch_replay_attn(d, split, tm_q, c->tm_k, c->tm_v, tm_o, p, st);
        if (e != cudaSuccess) return cuda_fail(e, "replay attention launch");
        if (!rec) c->launches++;
        if (split && !rec) {
            if (injected_failure(c)) return launch_fault("split-KV combine");
            e = launch_splitkv_combine(d, p, st);
            if (e != cudaSuccess) return cuda_fail(e, "split-KV combine launch");
            c->launches++;
        }
        if (tail) {
            // the lightest pairs [0, cut), keys split over the SMs, merged by the combine kernel
            AttnSeq &q = p.seqs[0];
            q.pair_top = static_cast<int32_t>(tp.pairs);
            q.n_splits = static_cast<int32_t>(tp.splits);
            q.item0 = 0;
            q.part_row0 = 0;
            q.comb0 = 0;
            p.split_tiles = static_cast<int32_t>(tp.split_tiles);
            p.total_items = static_cast<int32_t>(tp.pairs * hkv * tp.splits);
            p.total_comb = static_cast<int32_t>(tp.qtiles * hkv * kBM);  // q-tiles [0, 2 cut)
            p.pairs_fastest = c->attn_order > 0 ? 1 : 0;
            p.part_o = c->d_ws;
            p.part_lse = c->d_ws ? c->d_ws + tp.qtiles * hkv * tp.splits * kBM * d : nullptr;
            if (rec) {
                record_launch(c, 1, true, p, p.total_items);
                continue;
            }
            if (injected_failure(c)) return launch_fault("replay attention tail");
            e = launch_replay_attn(d, true, tm_q, c->tm_k, c->tm_v, tm_q, p, st);
            if (e != cudaSuccess) return cuda_fail(e, "replay attention tail launch");
            c->launches++;
            if (injected_failure(c)) return launch_fault("split-KV combine");
            e = launch_splitkv_combine(d, p, st);
            if (e != cudaSuccess) return cuda_fail(e, "split-KV combine launch");
            c->launches++;
        }
    }
    return PE_OK;
}

// Pointers are only checked when the call has queries (an empty tensor may be null).
pe_status check_attn_args(const pe_cache *c, int32_t layer, const void *Q, const void *out, int32_t hq, float scale,
                          bool has_rows = true)
{
    if (c->host_only) return fail(PE_ERR_UNSUPPORTED, "attention on a host-only cache");
    if (pe_status s = check_device(c)) return s;
    if (layer < 0 || layer >= c->cfg.num_layers) return fail(PE_ERR_RANGE, "layer %d out of range", layer);
    if (has_rows && (!Q || !out)) return fail(PE_ERR_INVALID, "null Q or out");
    if (has_rows && (!aligned16(Q) || !aligned16(out))) return fail(PE_ERR_INVALID, "Q and out must be 16-byte aligned");
    if (hq <= 0 || hq % c->cfg.num_kv_heads != 0)
        return fail(PE_ERR_INVALID, "num_q_heads %d is not a multiple of num_kv_heads %d", hq, c->cfg.num_kv_heads);
    const int g = hq / c->cfg.num_kv_heads;
    if (g > kBM || (g & (g - 1)) != 0)
        return fail(PE_ERR_UNSUPPORTED, "group size %d must be a power of two <= %d", g, kBM);
    if (!(scale > 0.f) || !std::isfinite(scale)) return fail(PE_ERR_INVALID, "softmax_scale must be positive");
    return PE_OK;
}

}  // namespace

extern "C" {

const char *pe_last_error(void) { return g_err.c_str(); }
const char *pe_version(void) { return "pe 0.1 (sm_103a)"; }

pe_status pe_cache_create(const pe_cache_config *cfg, pe_cache **out)
{
    g_err.clear();
    if (!cfg || !out) return fail(PE_ERR_INVALID, "null argument");
    *out = nullptr;
    const pe_cache_config &c = *cfg;
    if (c.num_layers < 1 || c.num_kv_heads < 1 || c.num_pages < 1 || c.max_seqs < 1 || c.max_pages_per_seq < 1)
        return fail(PE_ERR_INVALID, "all counts must be positive");
    if (c.head_dim != 64 && c.head_dim != 128) return fail(PE_ERR_UNSUPPORTED, "head_dim must be 64 or 128");
    const int ps = c.page_size;
    if (ps != 8 && ps != 16 && ps != 32 && ps != 64 && ps != 128)
        return fail(PE_ERR_UNSUPPORTED, "page_size must be 8, 16, 32, 64 or 128");
    const int64_t pool_rows = static_cast<int64_t>(c.num_layers) * c.num_pages * c.num_kv_heads * ps;
    if (pool_rows + ps >= INT32_MAX) return fail(PE_ERR_UNSUPPORTED, "pool too large for int32 row coordinates");
    if (static_cast<int64_t>(c.max_seqs) * c.max_pages_per_seq >= INT32_MAX)
        return fail(PE_ERR_UNSUPPORTED, "page table too large");
    if ((c.k_pool == nullptr) != (c.v_pool == nullptr)) return fail(PE_ERR_INVALID, "give both pools or neither");
    if (c.k_pool && (!aligned16(c.k_pool) || !aligned16(c.v_pool)))
        return fail(PE_ERR_INVALID, "pools must be 16-byte aligned");
    std::vector<int32_t> order(c.num_pages);
    if (c.init_free_order) {
        std::vector<uint8_t> seen(c.num_pages, 0);
        for (int i = 0; i < c.num_pages; ++i) {
            const int32_t pg = c.init_free_order[i];
            if (pg < 0 || pg >= c.num_pages || seen[pg]) return fail(PE_ERR_INVALID, "init_free_order is not a permutation");
            seen[pg] = 1;
            order[i] = pg;
        }
    } else {
        for (int i = 0; i < c.num_pages; ++i) order[i] = i;
    }

    pe_cache *cc = new (std::nothrow) pe_cache();
    if (!cc) return fail(PE_ERR_OOM, "host allocation failed");
    cc->cfg = c;
    cc->cfg.init_free_order = nullptr;
    cc->host_only = c.host_only != 0;
    cc->free_stack.assign(order.rbegin(), order.rend());  // first popped = order[0]
    cc->table.resize(c.max_seqs);
    cc->len.assign(c.max_seqs, 0);
    cc->appended.assign(c.max_seqs, 0);
    cc->alive.assign(c.max_seqs, 0);
    cc->refs.assign(c.num_pages, 0);
    cc->ckpt.resize(c.max_seqs);
    cc->pool_rows = pool_rows;
    cc->ws_bytes = c.workspace_bytes > 0 ? c.workspace_bytes : (256ll << 20);  // (also sizes host-only plans)
    if (cc->host_only) {
        *out = cc;
        return PE_OK;
    }

    cudaError_t e = cudaGetDevice(&cc->device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&cc->num_sms, cudaDevAttrMultiProcessorCount, cc->device);
    if (e != cudaSuccess) {
        delete cc;
        return cuda_fail(e, "no CUDA device");
    }
    int major = 0, minor = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, cc->device);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, cc->device);
    if (major != 10 || minor != 3) {  // sm_103a code runs on compute capability 10.3 only
        delete cc;
        return fail(PE_ERR_UNSUPPORTED, "kernels are built for sm_103a; device is sm_%d%d", major, minor);
    }
    const size_t pool_bytes = static_cast<size_t>(pool_rows) * c.head_dim * 2;
    const size_t table_bytes = static_cast<size_t>(c.max_seqs) * c.max_pages_per_seq * sizeof(int32_t);
    pe_status st = PE_OK;
    do {
        if (c.k_pool) {
            cc->k_pool = c.k_pool;
            cc->v_pool = c.v_pool;
        } else {
            cc->own_pools = true;
            if ((e = cudaMalloc(&cc->k_pool, pool_bytes)) != cudaSuccess) { st = cuda_fail(e, "cudaMalloc K pool"); break; }
            if ((e = cudaMalloc(&cc->v_pool, pool_bytes)) != cudaSuccess) { st = cuda_fail(e, "cudaMalloc V pool"); break; }
            // finite zeros: stale slots read under the causal mask must not hold NaN/Inf
            if ((e = cudaMemset(cc->k_pool, 0, pool_bytes)) != cudaSuccess) { st = cuda_fail(e, "memset"); break; }
            if ((e = cudaMemset(cc->v_pool, 0, pool_bytes)) != cudaSuccess) { st = cuda_fail(e, "memset"); break; }
        }
        if ((e = cudaMalloc(&cc->d_table, table_bytes)) != cudaSuccess) { st = cuda_fail(e, "cudaMalloc page table"); break; }
        if ((e = cudaMemset(cc->d_table, 0xFF, table_bytes)) != cudaSuccess) { st = cuda_fail(e, "memset"); break; }
        if ((e = cudaMalloc(&cc->d_len, sizeof(int64_t) * c.max_seqs)) != cudaSuccess) { st = cuda_fail(e, "cudaMalloc"); break; }
        if ((e = cudaMemset(cc->d_len, 0, sizeof(int64_t) * c.max_seqs)) != cudaSuccess) { st = cuda_fail(e, "memset"); break; }
        if ((e = cudaMalloc(&cc->d_status, sizeof(int32_t))) != cudaSuccess) { st = cuda_fail(e, "cudaMalloc"); break; }
        if ((e = cudaMemset(cc->d_status, 0, sizeof(int32_t))) != cudaSuccess) { st = cuda_fail(e, "memset"); break; }
        if ((e = cudaMalloc(&cc->d_ws, cc->ws_bytes)) != cudaSuccess) { st = cuda_fail(e, "cudaMalloc workspace"); break; }
        // per-(sequence, kv-head) merge tickets, the decode scheduler's chunk and done counters, then
        // the persistent attention's merge tickets
        const size_t tickets = sizeof(int32_t) * ticket_count(c.num_kv_heads);
        if ((e = cudaMalloc(&cc->d_tickets, tickets)) != cudaSuccess) { st = cuda_fail(e, "cudaMalloc"); break; }
        if ((e = cudaMemset(cc->d_tickets, 0, tickets)) != cudaSuccess) { st = cuda_fail(e, "memset"); break; }
        if ((st = encode_2d(&cc->tm_k, cc->k_pool, c.head_dim, pool_rows, 64, ps)) != PE_OK) break;
        if ((st = encode_2d(&cc->tm_v, cc->v_pool, c.head_dim, pool_rows, 64, ps)) != PE_OK) break;
        const uint32_t dec_rows = ps < kDecKeys ? ps : kDecKeys;
        if ((st = encode_2d(&cc->tm_kd, cc->k_pool, c.head_dim, pool_rows, 64, dec_rows)) != PE_OK) break;
        if ((st = encode_2d(&cc->tm_vd, cc->v_pool, c.head_dim, pool_rows, 64, dec_rows)) != PE_OK) break;
        if ((e = cudaDeviceSynchronize()) != cudaSuccess) { st = cuda_fail(e, "create sync"); break; }
    } while (false);
    if (st != PE_OK) {
        free_device(cc);
        delete cc;
        return st;
    }
    *out = cc;
    return PE_OK;
}

pe_status pe_cache_destroy(pe_cache *cache)
{
    if (!cache) return fail(PE_ERR_INVALID, "null cache");
    if (!cache->host_only) {
        // wait for and free on the cache's own device, whichever device is current
        int prev = -1;
        const bool switched = cudaGetDevice(&prev) == cudaSuccess && prev != cache->device &&
                              cudaSetDevice(cache->device) == cudaSuccess;
        cudaDeviceSynchronize();
        free_device(cache);
        if (switched) cudaSetDevice(prev);
    }
    delete cache;
    return PE_OK;
}

pe_status pe_seq_create(pe_cache *c, int32_t *seq_out)
{
    if (!c || !seq_out) return fail(PE_ERR_INVALID, "null argument");
    for (int32_t s = 0; s < c->cfg.max_seqs; ++s) {
        if (!c->alive[s]) {
            c->alive[s] = 1;
            c->table[s].clear();
            c->len[s] = 0;
            c->appended[s] = 0;
            c->ckpt[s].clear();
            *seq_out = s;
            return PE_OK;
        }
    }
    return fail(PE_ERR_OOM, "no free sequence slot (max_seqs = %d)", c->cfg.max_seqs);
}

pe_status pe_seq_release(pe_cache *c, int32_t seq, void *stream)
{
    std::vector<CropPlan> pl(1);
    pe_status s = check_device(c);
    if (s != PE_OK) return s;
    s = plan_crop(c, seq, 1, &pl[0]);
    if (s != PE_OK) return s;
    CallTxn tx(c, static_cast<cudaStream_t>(stream));
    apply_crop(c, pl[0], nullptr);
    c->alive[seq] = 0;
    c->ckpt[seq].clear();
    return tx.end(launch_crops(c, pl, static_cast<cudaStream_t>(stream)));
}

pe_status pe_seq_fork(pe_cache *c, int32_t seq, int32_t *new_seq, void *stream)
{
    pe_status s = check_seq(c, seq);
    if (s != PE_OK) return s;
    if ((s = check_device(c)) != PE_OK) return s;
    if (!new_seq) return fail(PE_ERR_INVALID, "null new_seq");
    int32_t ns = -1;
    for (int32_t q = 0; q < c->cfg.max_seqs; ++q)
        if (!c->alive[q]) { ns = q; break; }
    if (ns < 0) return fail(PE_ERR_OOM, "no free sequence slot (max_seqs = %d)", c->cfg.max_seqs);
    CallTxn tx(c, static_cast<cudaStream_t>(stream));
    j_seq(c, ns, 0);
    c->alive[ns] = 1;
    c->table[ns] = c->table[seq];
    for (int32_t pg : c->table[ns]) set_ref(c, pg, c->refs[pg] + 1);
    c->len[ns] = c->len[seq];
    c->appended[ns] = c->appended[seq];
    c->ckpt[ns] = c->ckpt[seq];
    if (injected_failure(c)) return tx.end(launch_fault("fork table copy"));
    if (!c->host_only) {
        cudaError_t e = launch_table_copy(c->d_table, seq * c->cfg.max_pages_per_seq, ns * c->cfg.max_pages_per_seq,
                                          static_cast<int32_t>(c->table[ns].size()), c->d_len, ns, c->len[ns],
                                          static_cast<cudaStream_t>(stream));
        if (e != cudaSuccess) return tx.end(cuda_fail(e, "fork table copy launch"));
        c->launches++;
    }
    *new_seq = ns;
    return tx.end(PE_OK);
}

pe_status pe_checkpoint_add(pe_cache *c, int32_t seq, int64_t offset)
{
    pe_status s = check_seq(c, seq);
    if (s != PE_OK) return s;
    if (offset < 0 || offset > c->len[seq])
        return fail(PE_ERR_RANGE, "checkpoint offset %lld outside [0, %lld]", static_cast<long long>(offset),
                    static_cast<long long>(c->len[seq]));
    std::vector<int64_t> &ck = c->ckpt[seq];
    auto it = std::lower_bound(ck.begin(), ck.end(), offset);
    if (it == ck.end() || *it != offset) ck.insert(it, offset);
    return PE_OK;
}

pe_status pe_checkpoint_select(const pe_cache *c, int32_t seq, int64_t tau, int64_t *offset)
{
    pe_status s = check_seq(c, seq);
    if (s != PE_OK) return s;
    if (tau < 1) return fail(PE_ERR_INVALID, "tau = %lld < 1", static_cast<long long>(tau));
    const std::vector<int64_t> &ck = c->ckpt[seq];
    auto it = std::lower_bound(ck.begin(), ck.end(), tau);  // first offset >= tau
    if (it == ck.begin()) return fail(PE_ERR_RANGE, "no checkpoint before tau = %lld", static_cast<long long>(tau));
    if (offset) *offset = *(it - 1);
    return PE_OK;
}

pe_status pe_seq_checkpoints(const pe_cache *c, int32_t seq, int64_t *out, int32_t cap, int32_t *n)
{
    pe_status s = check_seq(c, seq);
    if (s != PE_OK) return s;
    const std::vector<int64_t> &ck = c->ckpt[seq];
    if (n) *n = static_cast<int32_t>(ck.size());
    if (out) {
        if (cap < static_cast<int32_t>(ck.size())) return fail(PE_ERR_RANGE, "cap %d < %zu checkpoints", cap, ck.size());
        std::copy(ck.begin(), ck.end(), out);
    }
    return PE_OK;
}

pe_status pe_restore(pe_cache *c, int32_t seq, int64_t tau, int64_t *offset, int32_t *freed_out, int32_t freed_cap,
                     int32_t *n_freed, void *stream)
{
    int64_t b = 0;
    pe_status s = pe_checkpoint_select(c, seq, tau, &b);
    if (s != PE_OK) return s;
    if (tau - 1 > c->len[seq])
        return fail(PE_ERR_RANGE, "tau - 1 = %lld exceeds the sequence length %lld", static_cast<long long>(tau - 1),
                    static_cast<long long>(c->len[seq]));
    s = pe_crop(c, seq, b + 1, freed_out, freed_cap, n_freed, stream);
    if (s == PE_OK && offset) *offset = b;
    return s;
}

pe_status pe_page_refs(const pe_cache *c, int32_t *out, int32_t cap)
{
    if (!c || !out) return fail(PE_ERR_INVALID, "null argument");
    if (cap < c->cfg.num_pages) return fail(PE_ERR_RANGE, "cap %d < %d pages", cap, c->cfg.num_pages);
    std::copy(c->refs.begin(), c->refs.end(), out);
    return PE_OK;
}

pe_status pe_crop(pe_cache *c, int32_t seq, int64_t tau, int32_t *freed_out, int32_t freed_cap, int32_t *n_freed,
                  void *stream)
{
    std::vector<CropPlan> pl(1);
    pe_status s = check_device(c);
    if (s != PE_OK) return s;
    s = plan_crop(c, seq, tau, &pl[0]);
    if (s != PE_OK) return s;
    const int32_t nf = pl[0].n_freed;
    if (freed_out && freed_cap < nf) return fail(PE_ERR_RANGE, "freed_cap %d < %d freed pages", freed_cap, nf);
    CallTxn tx(c, static_cast<cudaStream_t>(stream));
    apply_crop(c, pl[0], freed_out);
    s = tx.end(launch_crops(c, pl, static_cast<cudaStream_t>(stream)));
    if (s == PE_OK && n_freed) *n_freed = nf;
    return s;
}

pe_status pe_crop_batch(pe_cache *c, int32_t n, const int32_t *seqs, const int64_t *taus, void *stream)
{
    if (pe_status s = check_device(c)) return s;
    if (n < 0 || (n > 0 && (!seqs || !taus))) return fail(PE_ERR_INVALID, "bad batch arguments");
    std::vector<CropPlan> plans(n);
    std::vector<uint8_t> seen(c->cfg.max_seqs, 0);
    for (int32_t i = 0; i < n; ++i) {
        pe_status s = plan_crop(c, seqs[i], taus[i], &plans[i]);
        if (s != PE_OK) return s;
        if (seen[seqs[i]]) return fail(PE_ERR_INVALID, "sequence %d appears twice in the batch", seqs[i]);
        seen[seqs[i]] = 1;
    }
    CallTxn tx(c, static_cast<cudaStream_t>(stream));
    for (CropPlan &pl : plans) apply_crop(c, pl, nullptr);
    return tx.end(launch_crops(c, plans, static_cast<cudaStream_t>(stream)));
}

pe_status pe_append_kv(pe_cache *c, int32_t seq, const void *K, const void *V, int32_t n_tokens, void *stream)
{
    AppendPlan pl{};
    pe_status s = check_device(c);
    if (s != PE_OK) return s;
    if ((s = plan_append(c, seq, n_tokens, &pl)) != PE_OK) return s;
    if (!c->host_only && n_tokens > 0) {
        if (!K || !V) return fail(PE_ERR_INVALID, "null K or V");
        if (!aligned16(K) || !aligned16(V)) return fail(PE_ERR_INVALID, "K and V must be 16-byte aligned");
    }
    if (pl.need > static_cast<int32_t>(c->free_stack.size()))
        return fail(PE_ERR_OOM, "append needs %d pages, %zu free", pl.need, c->free_stack.size());
    pl.tok0 = 0;
    CallTxn tx(c, static_cast<cudaStream_t>(stream));
    return tx.end(apply_appends(c, {pl}, K, V, n_tokens, static_cast<cudaStream_t>(stream)));
}

pe_status pe_append_kv_batch(pe_cache *c, int32_t n, const int32_t *seqs, const void *K, const void *V,
                             const int32_t *cu_tokens, void *stream)
{
    if (pe_status s = check_device(c)) return s;
    if (n < 0 || (n > 0 && (!seqs || !cu_tokens))) return fail(PE_ERR_INVALID, "bad batch arguments");
    if (n > 0 && cu_tokens[0] != 0) return fail(PE_ERR_INVALID, "cu_tokens[0] must be 0");
    std::vector<AppendPlan> plans(n);
    std::vector<uint8_t> seen(c->cfg.max_seqs, 0);
    for (int32_t i = 0; i < n; ++i) {
        if (cu_tokens[i + 1] < cu_tokens[i]) return fail(PE_ERR_INVALID, "cu_tokens must be non-decreasing");
        pe_status s = plan_append(c, seqs[i], cu_tokens[i + 1] - cu_tokens[i], &plans[i]);
        if (s != PE_OK) return s;
        if (seen[seqs[i]]) return fail(PE_ERR_INVALID, "sequence %d appears twice in the batch", seqs[i]);
        seen[seqs[i]] = 1;
        plans[i].tok0 = cu_tokens[i];
    }
    settle_batch_cow(c, plans);
    int64_t need = 0;
    for (const AppendPlan &pl : plans) need += pl.need;
    const int64_t total = n > 0 ? cu_tokens[n] : 0;
    if (!c->host_only && total > 0) {
        if (!K || !V) return fail(PE_ERR_INVALID, "null K or V");
        if (!aligned16(K) || !aligned16(V)) return fail(PE_ERR_INVALID, "K and V must be 16-byte aligned");
    }
    if (need > static_cast<int64_t>(c->free_stack.size()))
        return fail(PE_ERR_OOM, "batch append needs %lld pages, %zu free", static_cast<long long>(need),
                    c->free_stack.size());
    CallTxn tx(c, static_cast<cudaStream_t>(stream));
    return tx.end(apply_appends(c, plans, K, V, total, static_cast<cudaStream_t>(stream)));
}

pe_status pe_replay_attn(pe_cache *c, int32_t seq, int32_t layer, const void *Q, void *out, int32_t n_q,
                         int32_t num_q_heads, float softmax_scale, void *stream)
{
    pe_status s = check_seq(c, seq);
    if (s != PE_OK) return s;
    if ((s = check_attn_args(c, layer, Q, out, num_q_heads, softmax_scale, n_q > 0)) != PE_OK) return s;
    if (n_q < 0) return fail(PE_ERR_INVALID, "negative n_q");
    if (n_q > c->len[seq])
        return fail(PE_ERR_RANGE, "n_q = %d exceeds the sequence length %lld", n_q, static_cast<long long>(c->len[seq]));
    if (n_q == 0) return PE_OK;
    return run_attention(c, {AttnItem{seq, 0, n_q}}, layer, Q, n_q, out, num_q_heads, softmax_scale,
                         static_cast<cudaStream_t>(stream));
}

pe_status pe_replay_attn_batch(pe_cache *c, int32_t n, const int32_t *seqs, int32_t layer, const void *Q_packed,
                               const int32_t *cu_q, void *out, int32_t num_q_heads, float softmax_scale, void *stream)
{
    if (!c) return fail(PE_ERR_INVALID, "null cache");
    if (n < 0 || (n > 0 && (!seqs || !cu_q))) return fail(PE_ERR_INVALID, "bad batch arguments");
    if (n == 0) return PE_OK;
    pe_status s = check_attn_args(c, layer, Q_packed, out, num_q_heads, softmax_scale, cu_q[n] > 0);
    if (s != PE_OK) return s;
    if (cu_q[0] != 0) return fail(PE_ERR_INVALID, "cu_q[0] must be 0");
    std::vector<AttnItem> items(n);
    for (int32_t i = 0; i < n; ++i) {
        if ((s = check_seq(c, seqs[i])) != PE_OK) return s;
        const int32_t nq = cu_q[i + 1] - cu_q[i];
        if (nq < 0) return fail(PE_ERR_INVALID, "cu_q must be non-decreasing");
        if (nq > c->len[seqs[i]])
            return fail(PE_ERR_RANGE, "sequence %d: n_q = %d exceeds its length %lld", seqs[i], nq,
                        static_cast<long long>(c->len[seqs[i]]));
        items[i] = AttnItem{seqs[i], cu_q[i], nq};
    }
    if (cu_q[n] == 0) return PE_OK;
    return run_attention(c, items, layer, Q_packed, cu_q[n], out, num_q_heads, softmax_scale,
                         static_cast<cudaStream_t>(stream));
}

pe_status pe_replay_rounds(pe_cache *c, int32_t n, const int32_t *seqs, int32_t n_rounds, const int32_t *take,
                           const int32_t *cu_tok, const void *K, const void *V, const void *Q, void *out,
                           int32_t num_q_heads, float softmax_scale, void *stream)
{
    if (pe_status s = check_device(c)) return s;
    if (n < 0 || n_rounds < 0 || (n > 0 && (!seqs || !cu_tok)) || (n > 0 && n_rounds > 0 && !take))
        return fail(PE_ERR_INVALID, "bad rounds arguments");
    if (n == 0) return PE_OK;
    if (cu_tok[0] != 0) return fail(PE_ERR_INVALID, "cu_tok[0] must be 0");
    const int64_t N = cu_tok[n];
    pe_status s;
    if (c->host_only) {
        if (num_q_heads <= 0 || num_q_heads % c->cfg.num_kv_heads != 0)
            return fail(PE_ERR_INVALID, "num_q_heads %d is not a multiple of num_kv_heads", num_q_heads);
    } else if ((s = check_attn_args(c, 0, Q, out, num_q_heads, softmax_scale, N > 0)) != PE_OK) {
        return s;
    }
    if (!c->host_only && N > 0) {
        if (!K || !V) return fail(PE_ERR_INVALID, "null K or V");
        if (!aligned16(K) || !aligned16(V)) return fail(PE_ERR_INVALID, "K and V must be 16-byte aligned");
    }
    // every agent: a live, distinct sequence whose rounds cover its rows exactly,
    // and room for all of its positions (pages counted once, up front)
    std::vector<uint8_t> seen(c->cfg.max_seqs, 0);
    std::vector<AppendPlan> whole(n);
    for (int32_t i = 0; i < n; ++i) {
        if (cu_tok[i + 1] < cu_tok[i]) return fail(PE_ERR_INVALID, "cu_tok must be non-decreasing");
        AppendPlan &pl = whole[i];
        if ((s = plan_append(c, seqs[i], cu_tok[i + 1] - cu_tok[i], &pl)) != PE_OK) return s;
        if (seen[seqs[i]]) return fail(PE_ERR_INVALID, "sequence %d appears twice", seqs[i]);
        seen[seqs[i]] = 1;
        int64_t sum = 0;
        for (int32_t r = 0; r < n_rounds; ++r) {
            const int32_t t = take[static_cast<int64_t>(r) * n + i];
            if (t < 0) return fail(PE_ERR_INVALID, "negative take in round %d", r);
            sum += t;
        }
        if (sum != cu_tok[i + 1] - cu_tok[i])
            return fail(PE_ERR_INVALID, "agent %d: rounds cover %lld of its %d rows", i, static_cast<long long>(sum),
                        cu_tok[i + 1] - cu_tok[i]);
    }
    // a sequence copies its shared last page in its first round with work, in agent order
    settle_batch_cow(c, whole);
    int64_t need = 0;
    for (const AppendPlan &pl : whole) need += pl.need;
    if (need > static_cast<int64_t>(c->free_stack.size()))
        return fail(PE_ERR_OOM, "the rounds need %lld pages, %zu free", static_cast<long long>(need),
                    c->free_stack.size());

    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    CallTxn tx(c, st);
    const int64_t row_bytes = static_cast<int64_t>(num_q_heads) * c->cfg.head_dim * 2;  // one bf16 [Hq][d] row
    std::vector<int32_t> done(n, 0);
    std::vector<AppendPlan> plans;
    std::vector<AttnItem> items;
    for (int32_t r = 0; r < n_rounds; ++r) {
        plans.clear();
        items.clear();
        for (int32_t i = 0; i < n; ++i) {
            const int32_t t = take[static_cast<int64_t>(r) * n + i];
            if (t == 0) continue;
            AppendPlan pl{};
            plan_append(c, seqs[i], t, &pl);  // checked above for the whole suffix
            pl.tok0 = cu_tok[i] + done[i];
            plans.push_back(pl);
            items.push_back(AttnItem{seqs[i], cu_tok[i] + done[i], t});
            done[i] += t;
        }
        if (plans.empty()) continue;
        if ((s = apply_appends(c, plans, K, V, N, st)) != PE_OK) return tx.end(s);
        if (c->host_only) continue;
        for (int32_t layer = 0; layer < c->cfg.num_layers; ++layer) {
            const int64_t off = static_cast<int64_t>(layer) * N * row_bytes;
            s = run_attention(c, items, layer, static_cast<const char *>(Q) + off, N, static_cast<char *>(out) + off,
                              num_q_heads, softmax_scale, st);
            if (s != PE_OK) return tx.end(s);
        }
    }
    return tx.end(PE_OK);
}

pe_status pe_replay_attn_static_scratch(pe_cache *c, int32_t seq, int32_t layer, const void *Q, void *out,
                                        int32_t n_q, int32_t num_q_heads, float softmax_scale, void *stream)
{
    // Same computation as pe_replay_attn through the split-KV kernel and its
    // combine, but the partials go to the library's fixed device array, and
    // nothing here allocates (parameters live on the stack).
    pe_status s = check_seq(c, seq);
    if (s != PE_OK) return s;
    if ((s = check_attn_args(c, layer, Q, out, num_q_heads, softmax_scale)) != PE_OK) return s;
    if (n_q < 0) return fail(PE_ERR_INVALID, "negative n_q");
    if (n_q > c->len[seq])
        return fail(PE_ERR_RANGE, "n_q = %d exceeds the sequence length %lld", n_q, static_cast<long long>(c->len[seq]));
    if (n_q == 0) return PE_OK;
    const pe_cache_config &cf = c->cfg;
    const int hkv = cf.num_kv_heads, d = cf.head_dim, g = num_q_heads / hkv;
    const int64_t n_qtiles = ceil_div(static_cast<int64_t>(n_q) * g, kBM);
    const int64_t ktiles = ceil_div(c->len[seq], kBN);
    const int64_t row_bytes = static_cast<int64_t>(d) * 4 + 4;   // fp32 partial row + its LSE
    const int64_t split_bytes = n_qtiles * hkv * kBM * row_bytes;  // one split of every q-tile
    const int64_t max_splits = kStaticScratchBytes / split_bytes;
    if (max_splits < 1)
        return fail(PE_ERR_RANGE,
                    "static scratch too small: one key split of %d queries x %d heads needs %lld bytes, the fixed "
                    "array holds %lld",
                    n_q, num_q_heads, static_cast<long long>(split_bytes),
                    static_cast<long long>(kStaticScratchBytes));
    float *scratch = nullptr;
    cudaError_t e = static_scratch(&scratch);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress of the static scratch");
    // split count: about four CTAs per SM, at least 4 key tiles per split, within the array
    const int64_t pairs = ceil_div(n_qtiles, 2) * hkv;
    int64_t n_splits = std::max<int64_t>(1, std::min<int64_t>(ceil_div(4LL * c->num_sms, pairs), ceil_div(ktiles, 4)));
    n_splits = std::min(n_splits, max_splits);
    const int split_tiles = static_cast<int>(ceil_div(ktiles, n_splits));
    n_splits = ceil_div(ktiles, split_tiles);

    CUtensorMap tm_q;
    if ((s = encode_q(&tm_q, Q, n_q, num_q_heads, d, g)) != PE_OK) return s;
    AttnParams p;
    std::memset(&p, 0, sizeof p);
    p.page_table = c->d_table;
    p.out = out;
    p.status = c->d_status;
    p.n_seqs = 1;
    p.hq = num_q_heads;
    p.hkv = hkv;
    p.group = g;
    p.layer = layer;
    p.num_pages = cf.num_pages;
    p.ps = cf.page_size;
    p.oob_row = static_cast<int32_t>(c->pool_rows);
    p.split_tiles = split_tiles;
    p.scale_log2 = softmax_scale * 1.4426950408889634f;
    AttnSeq &q = p.seqs[0];
    q.table_row = seq * cf.max_pages_per_seq;
    q.n_pages = static_cast<int32_t>(c->table[seq].size());
    q.q_row0 = 0;
    q.n_q = n_q;
    q.n_keys = static_cast<int32_t>(c->len[seq]);
    q.n_qtiles = static_cast<int32_t>(n_qtiles);
    q.n_splits = static_cast<int32_t>(n_splits);
    q.pair_top = static_cast<int32_t>(ceil_div(n_qtiles, 2));
    const int64_t prow = n_qtiles * hkv * n_splits * kBM;
    p.total_items = static_cast<int32_t>(ceil_div(n_qtiles, 2) * hkv * n_splits);
    p.total_comb = static_cast<int32_t>(n_qtiles * hkv * kBM);
    p.part_o = scratch;
    p.part_lse = scratch + prow * d;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (injected_failure(c)) return launch_fault("replay attention");
    e = launch_replay_attn(d, true, tm_q, c->tm_k, c->tm_v, tm_q, p, st);
    if (e != cudaSuccess) return cuda_fail(e, "replay attention launch");
    c->launches++;
    if (injected_failure(c)) return launch_fault("split-KV combine");
    e = launch_splitkv_combine(d, p, st);
    if (e != cudaSuccess) return cuda_fail(e, "split-KV combine launch");
    c->launches++;
    return PE_OK;
}

pe_status pe_seq_info(const pe_cache *c, int32_t seq, int64_t *len, int64_t *appended_since_crop)
{
    pe_status s = check_seq(c, seq);
    if (s != PE_OK) return s;
    if (len) *len = c->len[seq];
    if (appended_since_crop) *appended_since_crop = c->appended[seq];
    return PE_OK;
}

pe_status pe_seq_page_table(const pe_cache *c, int32_t seq, int32_t *out, int32_t cap, int32_t *n)
{
    pe_status s = check_seq(c, seq);
    if (s != PE_OK) return s;
    const std::vector<int32_t> &t = c->table[seq];
    if (n) *n = static_cast<int32_t>(t.size());
    if (out) {
        if (cap < static_cast<int32_t>(t.size())) return fail(PE_ERR_RANGE, "cap %d < %zu entries", cap, t.size());
        std::copy(t.begin(), t.end(), out);
    }
    return PE_OK;
}

pe_status pe_free_list(const pe_cache *c, int32_t *out, int32_t cap, int32_t *n)
{
    if (!c) return fail(PE_ERR_INVALID, "null cache");
    const size_t nf = c->free_stack.size();
    if (n) *n = static_cast<int32_t>(nf);
    if (out) {
        if (cap < static_cast<int32_t>(nf)) return fail(PE_ERR_RANGE, "cap %d < %zu free pages", cap, nf);
        for (size_t i = 0; i < nf; ++i) out[i] = c->free_stack[nf - 1 - i];
    }
    return PE_OK;
}

pe_status pe_seq_device_page_table(pe_cache *c, int32_t seq, int32_t *out, int32_t cap, void *stream)
{
    pe_status s = check_seq(c, seq);
    if (s != PE_OK) return s;
    if (c->host_only) return fail(PE_ERR_UNSUPPORTED, "host-only cache has no device table");
    if ((s = check_device(c)) != PE_OK) return s;
    if (!out || cap < 0 || cap > c->cfg.max_pages_per_seq) return fail(PE_ERR_INVALID, "bad output buffer");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaStreamSynchronize(st);
    if (e == cudaSuccess)
        e = cudaMemcpy(out, c->d_table + static_cast<int64_t>(seq) * c->cfg.max_pages_per_seq,
                       sizeof(int32_t) * cap, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "device page table read");
    return PE_OK;
}

pe_status pe_cache_pools(const pe_cache *c, void **k_pool, void **v_pool)
{
    if (!c) return fail(PE_ERR_INVALID, "null cache");
    if (k_pool) *k_pool = c->k_pool;
    if (v_pool) *v_pool = c->v_pool;
    return PE_OK;
}

pe_status pe_set_option(pe_cache *c, const char *key, int64_t value)
{
    if (!c || !key) return fail(PE_ERR_INVALID, "null argument");
    if (!std::strcmp(key, "splitkv")) {
        if (value < -1 || value > 1) return fail(PE_ERR_INVALID, "splitkv must be -1, 0 or 1");
        c->splitkv = static_cast<int>(value);
    } else if (!std::strcmp(key, "num_splits")) {
        if (value < 0 || value > 4096) return fail(PE_ERR_INVALID, "num_splits out of range");
        c->num_splits = static_cast<int>(value);
    } else if (!std::strcmp(key, "debug_poison")) {
        c->debug_poison = value ? 1 : 0;
    } else if (!std::strcmp(key, "decode_chunks_per_sm")) {
        if (value < 1 || value > 64) return fail(PE_ERR_INVALID, "decode_chunks_per_sm must be 1..64");
        c->dec_chunks_per_sm = static_cast<int>(value);
    } else if (!std::strcmp(key, "decode_kernel")) {
        if (value < 0 || value > 2) return fail(PE_ERR_INVALID, "decode_kernel must be 0, 1 or 2");
        c->decode_kernel = static_cast<int>(value);
    } else if (!std::strcmp(key, "attn_kernel")) {
        if (value < 0 || value > 2) return fail(PE_ERR_INVALID, "attn_kernel must be 0, 1 or 2");
        c->attn_kernel = static_cast<int>(value);
    } else if (!std::strcmp(key, "attn_order")) {
        if (value < -1 || value > 1) return fail(PE_ERR_INVALID, "attn_order must be -1, 0 or 1");
        c->attn_order = static_cast<int>(value);
    } else if (!std::strcmp(key, "attn_ctas")) {
        if (value < 0 || value > kMaxSkCtas) return fail(PE_ERR_INVALID, "attn_ctas must be 0..%d", kMaxSkCtas);
        c->attn_ctas = static_cast<int>(value);
    } else if (!std::strcmp(key, "fail_launch_after")) {
        if (value < -1) return fail(PE_ERR_INVALID, "fail_launch_after must be -1 (off) or >= 0");
        c->fail_after = value;
    } else {
        return fail(PE_ERR_INVALID, "unknown option '%s'", key);
    }
    return PE_OK;
}

pe_status pe_selftest_bounded_wait(pe_cache *c, int64_t limit_ns, void *stream)
{
    if (!c) return fail(PE_ERR_INVALID, "null cache");
    if (c->host_only) return fail(PE_ERR_UNSUPPORTED, "host-only cache has no device");
    if (pe_status s = check_device(c)) return s;
    if (limit_ns < 1000 || limit_ns > 2000000000ll) return fail(PE_ERR_RANGE, "limit_ns must be in [1 us, 2 s]");
    cudaError_t e = launch_bounded_wait_selftest(c->d_status, static_cast<uint64_t>(limit_ns),
                                                 static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "self-test launch");
    c->launches++;
    return PE_OK;
}

pe_status pe_last_attn_plan(const pe_cache *c, int32_t *split, int32_t *n_splits, int32_t *ctas)
{
    if (!c) return fail(PE_ERR_INVALID, "null cache");
    if (split) *split = c->last_split;
    if (n_splits) *n_splits = c->last_splits;
    if (ctas) *ctas = c->last_ctas;
    return PE_OK;
}

pe_status pe_attn_plan_persistent(pe_cache *c, int32_t n, const int32_t *seqs, const int32_t *cu_q,
                                  int32_t num_q_heads, int32_t num_sms, int32_t *info, int32_t *order_out,
                                  int32_t *unit_tiles, int32_t units_cap, int32_t *ctas, int32_t ctas_cap,
                                  int32_t *slots, int32_t slots_cap)
{
    if (!c) return fail(PE_ERR_INVALID, "null cache");
    if (n < 1 || n > kMaxSegs || !seqs || !cu_q || !info) return fail(PE_ERR_INVALID, "bad plan arguments");
    if (cu_q[0] != 0) return fail(PE_ERR_INVALID, "cu_q[0] must be 0");
    const int32_t hkv = c->cfg.num_kv_heads;
    if (num_q_heads <= 0 || num_q_heads % hkv != 0)
        return fail(PE_ERR_INVALID, "num_q_heads %d is not a multiple of num_kv_heads %d", num_q_heads, hkv);
    const int32_t g = num_q_heads / hkv;
    if (g > kBM || (g & (g - 1)) != 0) return fail(PE_ERR_UNSUPPORTED, "group size %d must be a power of two <= %d", g, kBM);
    if (num_sms < 0 || num_sms > kMaxSkCtas) return fail(PE_ERR_RANGE, "num_sms must be 0..%d", kMaxSkCtas);
    if (num_sms == 0 && c->host_only) return fail(PE_ERR_INVALID, "a host-only cache has no SM count: give num_sms");
    std::vector<AttnItem> order;
    std::vector<uint8_t> seen(c->cfg.max_seqs, 0);
    for (int32_t i = 0; i < n; ++i) {
        pe_status s = check_seq(c, seqs[i]);
        if (s != PE_OK) return s;
        if (seen[seqs[i]]) return fail(PE_ERR_INVALID, "sequence %d appears twice", seqs[i]);
        seen[seqs[i]] = 1;
        const int32_t nq = cu_q[i + 1] - cu_q[i];
        if (nq < 1 || nq > c->len[seqs[i]])
            return fail(PE_ERR_RANGE, "sequence %d: n_q = %d outside [1, %lld]", seqs[i], nq,
                        static_cast<long long>(c->len[seqs[i]]));
        order.push_back(AttnItem{seqs[i], cu_q[i], nq});
    }
    // the attention call's order: longest sequence first, ties in call order
    std::stable_sort(order.begin(), order.end(),
                     [&](const AttnItem &a, const AttnItem &b) { return c->len[a.seq] > c->len[b.seq]; });
    std::vector<char> buf(sizeof(SkParams));
    SkParams &P = *reinterpret_cast<SkParams *>(buf.data());
    std::vector<int32_t> tiles;
    const int saved_sms = c->num_sms;
    if (num_sms > 0) c->num_sms = num_sms;
    const pe_status s = plan_sk(c, order, 0, order.size(), 0, nullptr, num_q_heads, 1.0f, P, &tiles);
    c->num_sms = saved_sms;
    if (s != PE_OK) return s;
    const int32_t n_units = static_cast<int32_t>(tiles.size());
    info[0] = P.n_ctas;
    info[1] = P.rounds;
    info[2] = P.n_slots;
    info[3] = P.max_parts;
    info[4] = n_units;
    if (order_out)
        for (size_t i = 0; i < order.size(); ++i) order_out[i] = order[i].seq;
    if ((unit_tiles && units_cap < n_units) || (ctas && ctas_cap < P.n_ctas) || (slots && slots_cap < P.n_slots))
        return fail(PE_ERR_RANGE, "plan needs %d units, %d CTAs, %d slots", n_units, P.n_ctas, P.n_slots);
    if (unit_tiles) std::copy(tiles.begin(), tiles.end(), unit_tiles);
    if (ctas)
        for (int32_t k = 0; k < P.n_ctas; ++k) {
            const SkCta &w = P.cta[k];
            const int32_t row[8] = {w.u0, w.t0, w.u1, w.t1, w.slot0, w.part0, w.slot1, w.part1};
            std::copy(row, row + 8, ctas + 8 * k);
        }
    if (slots)
        for (int32_t k = 0; k < P.n_slots; ++k) {
            slots[2 * k] = P.slots[k].unit;
            slots[2 * k + 1] = P.slots[k].n_parts;
        }
    return PE_OK;
}

pe_status pe_attn_plan_launches(pe_cache *c, int32_t n, const int32_t *seqs, const int32_t *cu_q, int32_t num_q_heads,
                                int32_t num_sms, int64_t *words, int64_t cap, int64_t *n_words)
{
    if (!c) return fail(PE_ERR_INVALID, "null cache");
    if (n < 1 || !seqs || !cu_q || !n_words) return fail(PE_ERR_INVALID, "bad plan arguments");
    if (cu_q[0] != 0) return fail(PE_ERR_INVALID, "cu_q[0] must be 0");
    const int32_t hkv = c->cfg.num_kv_heads;
    if (num_q_heads <= 0 || num_q_heads % hkv != 0)
        return fail(PE_ERR_INVALID, "num_q_heads %d is not a multiple of num_kv_heads %d", num_q_heads, hkv);
    const int32_t g = num_q_heads / hkv;
    if (g > kBM || (g & (g - 1)) != 0) return fail(PE_ERR_UNSUPPORTED, "group size %d must be a power of two <= %d", g, kBM);
    if (num_sms < 0 || num_sms > kMaxSkCtas) return fail(PE_ERR_RANGE, "num_sms must be 0..%d", kMaxSkCtas);
    if (num_sms == 0 && c->host_only) return fail(PE_ERR_INVALID, "a host-only cache has no SM count: give num_sms");
    std::vector<AttnItem> items(n);
    for (int32_t i = 0; i < n; ++i) {
        pe_status s = check_seq(c, seqs[i]);
        if (s != PE_OK) return s;
        const int32_t nq = cu_q[i + 1] - cu_q[i];
        if (nq < 0) return fail(PE_ERR_INVALID, "cu_q must be non-decreasing");
        if (nq > c->len[seqs[i]])
            return fail(PE_ERR_RANGE, "sequence %d: n_q = %d exceeds its length %lld", seqs[i], nq,
                        static_cast<long long>(c->len[seqs[i]]));
        items[i] = AttnItem{seqs[i], cu_q[i], nq};
    }
    // plan as an attention call would, recording instead of launching; nothing of the cache changes
    std::vector<int64_t> rec;
    const int saved_sms = c->num_sms;
    const int64_t saved_fail = c->fail_after;
    const int32_t saved_plan[3] = {c->last_split, c->last_splits, c->last_ctas};
    if (num_sms > 0) c->num_sms = num_sms;
    c->fail_after = -1;
    c->plan_rec = &rec;
    const pe_status s = run_attention(c, items, 0, nullptr, cu_q[n], nullptr, num_q_heads, 1.0f, nullptr);
    c->plan_rec = nullptr;
    c->num_sms = saved_sms;
    c->fail_after = saved_fail;
    c->last_split = saved_plan[0];
    c->last_splits = saved_plan[1];
    c->last_ctas = saved_plan[2];
    if (s != PE_OK) return s;
    *n_words = static_cast<int64_t>(rec.size());
    if (words) {
        if (cap < *n_words) return fail(PE_ERR_RANGE, "the plan takes %lld words, cap is %lld",
                                        static_cast<long long>(*n_words), static_cast<long long>(cap));
        std::copy(rec.begin(), rec.end(), words);
    }
    return PE_OK;
}

pe_status pe_kernel_launches(const pe_cache *c, int64_t *count)
{
    if (!c || !count) return fail(PE_ERR_INVALID, "null argument");
    *count = c->launches;
    return PE_OK;
}

pe_status pe_device_status(pe_cache *c, int32_t *code, int32_t clear, void *stream)
{
    if (!c || !code) return fail(PE_ERR_INVALID, "null argument");
    *code = 0;
    if (c->host_only) return PE_OK;
    if (pe_status s = check_device(c)) return s;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaStreamSynchronize(st);
    if (e == cudaSuccess) e = cudaMemcpy(code, c->d_status, sizeof(int32_t), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess && clear) e = cudaMemset(c->d_status, 0, sizeof(int32_t));
    // after a kernel gave up, its merge tickets and scheduler counters may be mid-count: reset them
    if (e == cudaSuccess && clear && *code != 0)
        e = cudaMemset(c->d_tickets, 0, sizeof(int32_t) * ticket_count(c->cfg.num_kv_heads));
    if (e != cudaSuccess) return cuda_fail(e, "device status read");
    if (*code != 0) return fail(PE_ERR_DEVICE_TIMEOUT, "a kernel reported status %d", *code);
    return PE_OK;
}

}  // extern "C"

// Append (prefill write of the replayed suffix, Sec. 3.2) and crop
// (restore = crop, Sec. 3.4(b); Alg. 1 Restore) kernels.
//
// Both are HBM/latency-bound copies: every thread moves whole 16-byte chunks
// (8 bf16) with vector loads and stores; consecutive threads touch consecutive
// chunks of one d-row, so a warp reads 512 contiguous bytes of the caller's
// K/V and writes whole 256-byte rows (d = 128) of a page slot.
#include "pe_internal.h"
#include "ptx.cuh"

namespace pe {

// The finite poison written by the debug crop: bf16 2^100 (0x7180) in every lane.
constexpr uint32_t kPoisonPair = 0x71807180u;

__device__ __forceinline__ uint4 ld_stream(const uint4 *p)
{
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__global__ void __launch_bounds__(256) append_kv_kernel(const __grid_constant__ AppendParams p, int64_t chunks)
{
    // the attention launch that follows may start its set-up now; it waits for this grid's writes
    ptx::griddep_launch_dependents();
    // launched with programmatic serialization: only the launch overlaps the previous kernel; every
    // read and write here waits for it (a crop before may still be poisoning freed pages)
    ptx::griddep_wait();
    // 1) mirror the new page ids and lengths into the device tables
    if (blockIdx.x == 0) {
        for (int s = 0; s < p.n_segs; ++s) {
            const AppendSeg &sg = p.segs[s];
            for (int i = threadIdx.x; i < sg.n_new; i += blockDim.x)
                p.page_table[sg.table_row + sg.first_new_lp + i] = p.new_pages[sg.new0 + i];
            if (threadIdx.x == 0)
                p.seq_len[sg.seq] = static_cast<int64_t>(sg.len0) + sg.n_tokens;
        }
    }
    // 2) scatter K/V rows into their page slots
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; c < chunks; c += stride) {
        const int dv = static_cast<int>(c % p.dvec);
        int64_t r = c / p.dvec;
        const int h = static_cast<int>(r % p.hkv);
        r /= p.hkv;
        const int t = static_cast<int>(r % p.seg_tokens);  // token within this launch's segments
        const int l = static_cast<int>(r / p.seg_tokens);
        int lo = 0, hi = p.n_segs - 1;
        while (lo < hi) {  // last segment with cum0 <= t
            const int mid = (lo + hi + 1) >> 1;
            if (p.segs[mid].cum0 <= t) lo = mid; else hi = mid - 1;
        }
        const AppendSeg &sg = p.segs[lo];
        const int local = t - sg.cum0;
        const int pos = sg.len0 + local;
        const int lp = pos / p.ps;
        const int slot = pos - lp * p.ps;
        const int page = lp < sg.first_new_lp ? sg.last_page : p.new_pages[sg.new0 + (lp - sg.first_new_lp)];
        const int64_t src = ((static_cast<int64_t>(l) * p.n_total + sg.tok0 + local) * p.hkv + h) * p.dvec + dv;
        const int64_t dst =
            (((static_cast<int64_t>(l) * p.num_pages + page) * p.hkv + h) * p.ps + slot) * p.dvec + dv;
        const uint4 kv = ld_stream(p.K + src);
        const uint4 vv = ld_stream(p.V + src);
        p.k_pool[dst] = kv;
        p.v_pool[dst] = vv;
    }
}

cudaError_t launch_append(const AppendParams &p, int64_t chunks, cudaStream_t st)
{
    static int sms = 0;
    if (sms == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (sms <= 0) sms = 148;
    }
    int64_t blocks = (chunks + 255) / 256;
    const int64_t cap = static_cast<int64_t>(sms) * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(blocks));
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, append_kv_kernel, p, chunks);
}

// One block per cropped sequence.  Debug poison first overwrites the pages
// whose last reference this crop dropped (every layer, head, slot, K and V) and
// the stale tail of the last kept page when no other sequence holds it; then
// the table entries [keep, old_n) of this sequence become -1.
__global__ void __launch_bounds__(256) crop_kernel(const __grid_constant__ CropParams p)
{
    // launched with programmatic serialization: the launch overlaps the previous kernel (an attention
    // launch that may still read the pages this crop frees); every write here waits for it
    ptx::griddep_launch_dependents();
    ptx::griddep_wait();
    const CropSeg &sg = p.segs[blockIdx.x];
    int32_t *row = p.page_table + sg.table_row;
    if (p.poison) {
        const uint4 poison = make_uint4(kPoisonPair, kPoisonPair, kPoisonPair, kPoisonPair);
        const int slot_chunks = p.dvec;                          // chunks per (page, head, slot)
        const int page_chunks = p.hkv * p.ps * slot_chunks;      // per (layer, page)
        for (int e = 0; e < sg.n_freed; ++e) {
            const int page = p.freed[sg.freed0 + e];
            if (page < 0 || page >= p.num_pages) continue;
            for (int l = 0; l < p.L; ++l) {
                const int64_t base = (static_cast<int64_t>(l) * p.num_pages + page) * page_chunks;
                for (int i = threadIdx.x; i < page_chunks; i += blockDim.x) {
                    p.k_pool[base + i] = poison;
                    p.v_pool[base + i] = poison;
                }
            }
        }
        const int tail = static_cast<int>(sg.new_len % p.ps);
        const int page = sg.tail_page;
        if (tail != 0 && page >= 0 && page < p.num_pages) {
            const int per_head = (p.ps - tail) * slot_chunks;
            for (int l = 0; l < p.L; ++l)
                for (int h = 0; h < p.hkv; ++h) {
                    const int64_t base =
                        (((static_cast<int64_t>(l) * p.num_pages + page) * p.hkv + h) * p.ps + tail) * slot_chunks;
                    for (int i = threadIdx.x; i < per_head; i += blockDim.x) {
                        p.k_pool[base + i] = poison;
                        p.v_pool[base + i] = poison;
                    }
                }
        }
        __syncthreads();
    }
    for (int e = sg.keep + static_cast<int>(threadIdx.x); e < sg.old_n; e += blockDim.x)
        row[e] = -1;
    if (threadIdx.x == 0)
        p.seq_len[sg.seq] = sg.new_len;
}

cudaError_t launch_crop(const CropParams &p, cudaStream_t st)
{
    if (p.n <= 0) return cudaSuccess;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(p.n));
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, crop_kernel, p);
}

__global__ void __launch_bounds__(256) table_copy_kernel(int32_t *page_table, int32_t src_row, int32_t dst_row,
                                                         int32_t n, int64_t *seq_len, int32_t dst_seq, int64_t len)
{
    for (int i = threadIdx.x; i < n; i += blockDim.x) page_table[dst_row + i] = page_table[src_row + i];
    if (threadIdx.x == 0) seq_len[dst_seq] = len;
}

cudaError_t launch_table_copy(int32_t *page_table, int32_t src_row, int32_t dst_row, int32_t n, int64_t *seq_len,
                              int32_t dst_seq, int64_t len, cudaStream_t st)
{
    table_copy_kernel<<<1, 256, 0, st>>>(page_table, src_row, dst_row, n, seq_len, dst_seq, len);
    return cudaGetLastError();
}

// Grid: (layer x kv-head) blocks; each copies `slots` rows of d (16-byte chunks).
__global__ void __launch_bounds__(256) cow_copy_kernel(uint4 *k_pool, uint4 *v_pool, int32_t src, int32_t dst,
                                                       int32_t slots, int32_t hkv, int32_t ps, int32_t dvec,
                                                       int32_t num_pages, int32_t *table_entry)
{
    const int l = blockIdx.x / hkv;
    const int h = blockIdx.x % hkv;
    const int64_t s_base = ((static_cast<int64_t>(l) * num_pages + src) * hkv + h) * ps * dvec;
    const int64_t d_base = ((static_cast<int64_t>(l) * num_pages + dst) * hkv + h) * ps * dvec;
    for (int i = threadIdx.x; i < slots * dvec; i += blockDim.x) {
        k_pool[d_base + i] = k_pool[s_base + i];
        v_pool[d_base + i] = v_pool[s_base + i];
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) *table_entry = dst;
}

cudaError_t launch_cow_copy(uint4 *k_pool, uint4 *v_pool, int32_t src, int32_t dst, int32_t slots, int32_t L,
                            int32_t hkv, int32_t ps, int32_t dvec, int32_t num_pages, int32_t *table_entry,
                            cudaStream_t st)
{
    cow_copy_kernel<<<L * hkv, 256, 0, st>>>(k_pool, v_pool, src, dst, slots, hkv, ps, dvec, num_pages, table_entry);
    return cudaGetLastError();
}

}  // namespace pe

// Device helpers shared by the attention kernels (pe_attn.cu, pe_attn_sk.cu,
// pe_decode.cu): bounded mbarrier waits with an error status, exp2 on the MUFU
// unit, packed fp32x2 arithmetic, 16-column TMEM loads/stores, the TS form of
// tcgen05.mma and bf16 packing.  Private to the library.
#pragma once

#include <cstdint>
#include <cuda_bf16.h>

#include "pe_internal.h"
#include "ptx.cuh"

namespace pe {

constexpr uint64_t kWaitNs = 1000000000ull;  // 1 s: limit of every mbarrier wait

struct WaitCtx {
    volatile int *abort;
    int32_t *status;
};

// Bounded mbarrier wait.  Returns false (and stops the CTA's pipeline) when the
// wait ran out or another role already gave up.
__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, const WaitCtx &w,
                                         uint64_t limit_ns = kWaitNs)
{
    if (ptx::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = ptx::globaltimer();
    for (;;) {
        if (ptx::mbar_try_wait(bar, parity)) return true;
        if (*w.abort) return false;
        if (ptx::globaltimer() - t0 > limit_ns) {
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

__device__ __forceinline__ float max3(float a, float b, float c)
{
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// (a*b + c) on two fp32 lanes at once
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c)
{
    uint64_t ra, rb, rc, rd;
    asm("mov.b64 %0, {%1, %2};" : "=l"(ra) : "f"(a.x), "f"(a.y));
    asm("mov.b64 %0, {%1, %2};" : "=l"(rb) : "f"(b.x), "f"(b.y));
    asm("mov.b64 %0, {%1, %2};" : "=l"(rc) : "f"(c.x), "f"(c.y));
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(rd) : "l"(ra), "l"(rb), "l"(rc));
    float2 d;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(d.x), "=f"(d.y) : "l"(rd));
    return d;
}

__device__ __forceinline__ float2 add2(float2 a, float2 b)
{
    uint64_t ra, rb, rd;
    asm("mov.b64 %0, {%1, %2};" : "=l"(ra) : "f"(a.x), "f"(a.y));
    asm("mov.b64 %0, {%1, %2};" : "=l"(rb) : "f"(b.x), "f"(b.y));
    asm("add.f32x2 %0, %1, %2;" : "=l"(rd) : "l"(ra), "l"(rb));
    float2 d;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(d.x), "=f"(d.y) : "l"(rd));
    return d;
}

// 32 lanes x 16 consecutive 32-bit TMEM columns from registers.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&v)[16])
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]),
        "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
        : "memory");
}

// 32 lanes x 16 consecutive 32-bit TMEM columns into registers.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&v)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
        : "r"(taddr)
        : "memory");
}

// D[tmem] (+)= A[tmem] * B[smem] (A = P, bf16 packed two per column).
__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Split partials (O / l, fp32, HD columns a row) are stored in blocks of 32 rows, 16-byte chunk major:
// chunk k of row r at [r & ~31][k][r & 31].  Row blocks start at multiples of 32 rows, so a warp whose
// lane i holds row 32 w + i writes or reads one chunk of its 32 rows as 512 contiguous bytes.
template <int HD>
__device__ __forceinline__ float4 *part_chunk(float *part_o, int64_t row, int k)
{
    return reinterpret_cast<float4 *>(part_o + (row & ~static_cast<int64_t>(31)) * HD) + k * 32 + (row & 31);
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&h);
}

}  // namespace pe

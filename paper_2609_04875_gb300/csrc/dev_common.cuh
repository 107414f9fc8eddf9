// Device helpers shared by the attention kernels (pe_attn.cu, pe_decode.cu):
// bounded mbarrier waits with an error status, exp2 on the MUFU unit, packed
// fp32x2 arithmetic and bf16 packing.  Private to the library.
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

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&h);
}

}  // namespace pe

// Device helpers shared by the bf16 tree-attention kernels (the per-layer
// split kernel and the multi-layer kernel): proxy fences, named barriers,
// packed fp32 pairs, exp2, the 128B swizzle of TMA/tcgen05 tiles, bf16
// packing and the rotate-half RoPE of 8-element chunks.
#pragma once

#include "gv_internal.cuh"

namespace gv {

// Makes generic-proxy shared-memory writes visible to the async proxy (the
// tensor cores and TMA).  Writes of other threads are covered when they are
// ordered before the fence by a barrier (__syncwarp, bar.sync), so each
// hand-off below fences once, in the thread that signals, after the barrier:
// the fence costs grow with the number of threads that execute it.
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}
// Named barrier of two warps (64 threads) that also returns whether every
// thread passed a nonzero flag.
__device__ __forceinline__ bool pair_bar_and(int id, int flag) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.s32 q, %2, 0;\n\t"
        "bar.red.and.pred p, %1, 64, q;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(r)
        : "r"(id), "r"(flag)
        : "memory");
    return r != 0;
}
// Named barrier of `nthreads` threads (a multiple of 32) that returns whether
// every one of them passed a nonzero flag.
__device__ __forceinline__ bool bar_and(int id, int nthreads, int flag) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.s32 q, %3, 0;\n\t"
        "bar.red.and.pred p, %1, %2, q;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(r)
        : "r"(id), "r"(nthreads), "r"(flag)
        : "memory");
    return r != 0;
}
// Packed fp32 pairs (one instruction for two lanes' worth of work) and the
// three-input max of sm_100+.
__device__ __forceinline__ uint64_t f32x2(float a, float b) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
    return r;
}
__device__ __forceinline__ float2 split_f32x2(uint64_t r) {
    float2 v;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(v.x), "=f"(v.y) : "l"(r));
    return v;
}
__device__ __forceinline__ uint64_t ffma_f32x2(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}
__device__ __forceinline__ uint64_t fadd_f32x2(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ float max3(float a, float b, float c) {
    float m;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(m) : "f"(a), "f"(b), "f"(c));
    return m;
}
__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
// Byte offset of 16-byte chunk c of row r inside a 128B-swizzled tile whose
// rows are 128 bytes apart (the layout TMA writes and tcgen05 reads).
__device__ __forceinline__ uint32_t sw128(int r, int c) {
    return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ float2 unpack_bf16(uint32_t u) {
    __nv_bfloat162 v = *reinterpret_cast<__nv_bfloat162*>(&u);
    return __bfloat1622float2(v);
}

// Rotate 8 consecutive elements of the low half (lo) and the matching 8 of the
// high half (hi) with 8 (cos, sin) pairs held as 4 float4; results as bf16.
__device__ __forceinline__ void rope8(const uint4& lo, const uint4& hi, const float4* cs, uint4& olo,
                                      uint4& ohi) {
    const uint32_t* l = reinterpret_cast<const uint32_t*>(&lo);
    const uint32_t* h = reinterpret_cast<const uint32_t*>(&hi);
    uint32_t* ol = reinterpret_cast<uint32_t*>(&olo);
    uint32_t* oh = reinterpret_cast<uint32_t*>(&ohi);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const float2 a = unpack_bf16(l[e]);
        const float2 b = unpack_bf16(h[e]);
        const float4 c = cs[e];   // (cos, sin) of element 2e, then of 2e+1
        ol[e] = pack_bf16(a.x * c.x - b.x * c.y, a.y * c.z - b.y * c.w);
        oh[e] = pack_bf16(b.x * c.x + a.x * c.y, b.y * c.z + a.y * c.w);
    }
}

}  // namespace gv

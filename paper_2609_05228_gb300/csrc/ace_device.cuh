// ace_device.cuh — device helpers shared by the library's kernels.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "ace_internal.h"

namespace ace {

// Index guards of the debug build (compiled with ACE_DEBUG_CHECKS): a
// computed index that falls outside its array sets kErrBounds in the layer's
// error word and the caller skips (or neutralises) the access; no trap. The
// release build compiles every guard to `true`.
#ifdef ACE_DEBUG_CHECKS
#define ACE_IDX_OK(cond, err) ((cond) ? true : (atomicOr((err), ::ace::kErrBounds), false))
#else
#define ACE_IDX_OK(cond, err) true
#endif

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ int warp_sum_int(int v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ unsigned lanemask_lt() {
    unsigned m;
    asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
    return m;
}

// 16-byte vectors of the storage type, widened to float.
template <typename T> struct Vec16;

template <> struct Vec16<float> {
    static constexpr int N = 4;
    __device__ __forceinline__ static void to_float(const uint4& v, float* f) {
        f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
        f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
    }
};

template <> struct Vec16<__nv_bfloat16> {
    static constexpr int N = 8;
    __device__ __forceinline__ static void to_float(const uint4& v, float* f) {
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            f[2 * i] = __uint_as_float(w[i] << 16);
            f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
        }
    }
};

__device__ __forceinline__ float to_f32(float v) { return v; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 v) { return __bfloat162float(v); }
template <typename T> __device__ __forceinline__ T from_f32(float v);
template <> __device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) {
    return __float2bfloat16_rn(v);
}

// Programmatic dependent launch: wait for the predecessor grid's results /
// allow the successor grid to be scheduled. No-ops without PDL.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Streaming 16-byte load that does not allocate in L1 (weights are read once).
__device__ __forceinline__ uint4 ld_stream(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
    return v;
}

// L2 cache policy that marks the lines a load touches as evict-last.
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}

// 16-byte load with an L2 cache policy.
__device__ __forceinline__ uint4 ld_l2_keep(const void* p, uint64_t policy) {
    uint4 v;
    asm volatile("ld.global.L2::cache_hint.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p), "l"(policy));
    return v;
}

// 16-byte streaming store (data read once later: evict first).
__device__ __forceinline__ void st_stream(void* p, const uint4& v) {
    asm volatile("st.global.cs.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}

// exp(x) for float32 x <= 0 in a fixed operation sequence (each multiply and
// add rounded to nearest even, none fused), so that the gates are
// reproducible bit for bit by any implementation following the same steps:
//   n = rint(x * log2(e));  r = (x - n*ln2_hi) - n*ln2_lo   (Cody & Waite 1980,
//   ln2_hi = 355/512 has 9 significant bits so n*ln2_hi is exact);
//   p = sum_{j=0..7} r^j / j!  in Horner form;  result = p * 2^n.
// Inputs below -87 return 0 (there 2^n would leave the normal range).
__device__ __forceinline__ float ace_exp32(float x) {
    const float kLog2e = 0x1.715476p+0f;     // float32(1 / ln 2)
    const float kLn2Hi = 0x1.63p-1f;          // 355 / 512
    const float kLn2Lo = -0x1.bd0106p-13f;    // float32(ln 2 - 355/512)
    const float c7 = 0x1.a01a02p-13f;         // float32(1/5040)
    const float c6 = 0x1.6c16c2p-10f;         // float32(1/720)
    const float c5 = 0x1.111112p-7f;          // float32(1/120)
    const float c4 = 0x1.555556p-5f;          // float32(1/24)
    const float c3 = 0x1.555556p-3f;          // float32(1/6)
    const float n = rintf(__fmul_rn(x, kLog2e));
    float r = __fsub_rn(x, __fmul_rn(n, kLn2Hi));
    r = __fsub_rn(r, __fmul_rn(n, kLn2Lo));
    float p = c7;
    p = __fadd_rn(__fmul_rn(p, r), c6);
    p = __fadd_rn(__fmul_rn(p, r), c5);
    p = __fadd_rn(__fmul_rn(p, r), c4);
    p = __fadd_rn(__fmul_rn(p, r), c3);
    p = __fadd_rn(__fmul_rn(p, r), 0.5f);
    p = __fadd_rn(__fmul_rn(p, r), 1.0f);
    p = __fadd_rn(__fmul_rn(p, r), 1.0f);
    int ni = (int)n;
    ni = ni < -126 ? -126 : (ni > 127 ? 127 : ni);
    const float scale = __int_as_float((ni + 127) << 23);
    const float out = __fmul_rn(p, scale);
    return x < -87.0f ? 0.0f : out;
}

// ---------------------------------------------------------------- mbarrier / bulk copy

constexpr long long kSpinCycles = 4000000000LL;   // bound on every mbarrier wait (~2 s at 2 GHz)

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait: false (and kErrTimeout set) if the phase did not complete.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, int* err) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (clock64() - t0 > kSpinCycles) {
            atomicOr(err, kErrTimeout);
            return false;
        }
    }
    return true;
}

// Bounded wait of a pipeline role that also gives up once another role of
// the CTA has set `abort_flag`. The flag is read only while the phase is
// still incomplete, so a wait that succeeds at once costs one try_wait.
__device__ __forceinline__ bool mbar_wait_or_abort(uint64_t* bar, uint32_t parity, int* err,
                                                   volatile int* abort_flag) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (*abort_flag) return false;
        if (clock64() - t0 > kSpinCycles) {
            atomicOr(err, kErrTimeout);
            return false;
        }
    }
    return true;
}

// 1-D bulk copy global -> shared (16-byte aligned addresses, size a multiple
// of 16), completing `bytes` of transaction count on `bar`.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}

__device__ __forceinline__ void mbar_inval(uint64_t* bar) {
    asm volatile("mbarrier.inval.shared::cta.b64 [%0];" ::"r"(smem_u32(bar)) : "memory");
}

}  // namespace ace

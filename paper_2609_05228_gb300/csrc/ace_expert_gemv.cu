// ace_expert_gemv.cu — the SwiGLU experts (Eq. swiglu_expert) over the
// retained slots only, as weight-streaming GEMVs, and the gate-weighted
// combine (Eq. ace_sparse_output).
//
// Work items are (distinct retained expert, slice of weight rows); the
// compaction's last block sizes the slices so that there are about four
// items per SM. Each item streams its weight rows once per chunk of up to
// kGemvTokenChunk tokens routed to that expert, with 16-byte non-caching
// loads; the tokens' activations sit in shared memory.
//   gate/up: act[r, j] = SiLU(h_t . W_gate[e, j]) * (h_t . W_up[e, j])
//   down:    y[r, c]   = g_hat(r) * (act[r] . W_down[e, c])
//   combine: out[t, c] = sum over t's kept slots, in rank order, of y[r, c]
#include <math.h>

#include "ace_device.cuh"
#include "ace_internal.h"

namespace ace {
namespace {

constexpr int kTC = kGemvTokenChunk;

__device__ __forceinline__ float silu(float u) { return u / (1.0f + expf(-u)); }

template <typename T>
__global__ void __launch_bounds__(256) k_gemv_gateup(const T* __restrict__ h, const T* __restrict__ w_gate,
                                                     const T* __restrict__ w_up,
                                                     const int32_t* __restrict__ offsets,
                                                     const int32_t* __restrict__ dlist,
                                                     const int32_t* __restrict__ perm,
                                                     const int32_t* __restrict__ meta,
                                                     float* __restrict__ act, int d, int m, int k) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    uint4* hs = reinterpret_cast<uint4*>(smem_raw);     // [kTC][d / V] vectors
    constexpr int V = Vec16<T>::N;
    const int nvec = d / V;
    const int D = meta[kMetaDistinct];
    const int S = meta[kMetaSlice1];
    const int nsl = m / S;
    const int items = D * nsl;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
    for (int item = blockIdx.x; item < items; item += gridDim.x) {
        const int e = dlist[item / nsl];
        const int sl = item % nsl;
        const int r0 = offsets[e], ne = offsets[e + 1] - r0;
        for (int tc0 = 0; tc0 < ne; tc0 += kTC) {
            const int ntc = min(kTC, ne - tc0);
            __syncthreads();
            for (int i = threadIdx.x; i < kTC * nvec; i += blockDim.x) {
                const int q = i / nvec, c = i % nvec;
                uint4 v = make_uint4(0, 0, 0, 0);
                if (q < ntc) {
                    const int tok = perm[r0 + tc0 + q] / k;
                    v = reinterpret_cast<const uint4*>(h + (size_t)tok * d)[c];
                }
                hs[i] = v;
            }
            __syncthreads();
            for (int row = warp; row < S; row += nwarps) {
                const int j = sl * S + row;
                const uint4* wg = reinterpret_cast<const uint4*>(w_gate + ((size_t)e * m + j) * d);
                const uint4* wu = reinterpret_cast<const uint4*>(w_up + ((size_t)e * m + j) * d);
                float ag[kTC], au[kTC];
#pragma unroll
                for (int q = 0; q < kTC; ++q) { ag[q] = 0.f; au[q] = 0.f; }
                for (int c = lane; c < nvec; c += 32) {
                    float fg[V], fu[V];
                    Vec16<T>::to_float(ld_stream(wg + c), fg);
                    Vec16<T>::to_float(ld_stream(wu + c), fu);
#pragma unroll
                    for (int q = 0; q < kTC; ++q) {
                        if (q < ntc) {
                            float fh[V];
                            Vec16<T>::to_float(hs[q * nvec + c], fh);
#pragma unroll
                            for (int i = 0; i < V; ++i) {
                                ag[q] = fmaf(fh[i], fg[i], ag[q]);
                                au[q] = fmaf(fh[i], fu[i], au[q]);
                            }
                        }
                    }
                }
#pragma unroll
                for (int q = 0; q < kTC; ++q) {
                    if (q < ntc) {
                        const float g = warp_sum(ag[q]);
                        const float u = warp_sum(au[q]);
                        if (lane == 0) act[(size_t)(r0 + tc0 + q) * m + j] = silu(g) * u;
                    }
                }
            }
        }
    }
}

template <typename T>
__global__ void __launch_bounds__(256) k_gemv_down(const float* __restrict__ act, const T* __restrict__ w_down,
                                                   const float* __restrict__ ghat,
                                                   const int32_t* __restrict__ offsets,
                                                   const int32_t* __restrict__ dlist,
                                                   const int32_t* __restrict__ perm,
                                                   const int32_t* __restrict__ meta,
                                                   float* __restrict__ yslot, int d, int m) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    float* as = reinterpret_cast<float*>(smem_raw);      // [kTC][m]
    __shared__ float gs[kTC];
    constexpr int V = Vec16<T>::N;
    const int nvec = m / V;
    const int D = meta[kMetaDistinct];
    const int S = meta[kMetaSlice2];
    const int nsl = d / S;
    const int items = D * nsl;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
    for (int item = blockIdx.x; item < items; item += gridDim.x) {
        const int e = dlist[item / nsl];
        const int sl = item % nsl;
        const int r0 = offsets[e], ne = offsets[e + 1] - r0;
        for (int tc0 = 0; tc0 < ne; tc0 += kTC) {
            const int ntc = min(kTC, ne - tc0);
            __syncthreads();
            for (int i = threadIdx.x; i < kTC * (m / 4); i += blockDim.x) {
                const int q = i / (m / 4), c = i % (m / 4);
                float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
                if (q < ntc) v = reinterpret_cast<const float4*>(act + (size_t)(r0 + tc0 + q) * m)[c];
                reinterpret_cast<float4*>(as)[i] = v;
            }
            if (threadIdx.x < kTC) gs[threadIdx.x] = threadIdx.x < ntc ? ghat[perm[r0 + tc0 + threadIdx.x]] : 0.f;
            __syncthreads();
            for (int row = warp; row < S; row += nwarps) {
                const int c = sl * S + row;
                const uint4* wd = reinterpret_cast<const uint4*>(w_down + ((size_t)e * d + c) * m);
                float acc[kTC];
#pragma unroll
                for (int q = 0; q < kTC; ++q) acc[q] = 0.f;
                for (int v = lane; v < nvec; v += 32) {
                    float fw[V];
                    Vec16<T>::to_float(ld_stream(wd + v), fw);
#pragma unroll
                    for (int q = 0; q < kTC; ++q) {
                        if (q < ntc) {
                            const float* ar = as + q * m + v * V;
#pragma unroll
                            for (int i = 0; i < V; ++i) acc[q] = fmaf(ar[i], fw[i], acc[q]);
                        }
                    }
                }
#pragma unroll
                for (int q = 0; q < kTC; ++q) {
                    if (q < ntc) {
                        const float y = warp_sum(acc[q]);
                        if (lane == 0) yslot[(size_t)(r0 + tc0 + q) * d + c] = gs[q] * y;
                    }
                }
            }
        }
    }
}

// out[t, c] = sum_{i kept, rank order} y[slot_pos[t*k+i], c]
template <typename T>
__global__ void __launch_bounds__(256) k_combine(const float* __restrict__ yslot,
                                                 const int32_t* __restrict__ slot_pos, T* __restrict__ out,
                                                 int n_tokens, int d, int k) {
    const int nq = d / 4;
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)n_tokens * nq) return;
    const int t = (int)(idx / nq), c4 = (int)(idx % nq);
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int i = 0; i < k; ++i) {
        const int r = slot_pos[(size_t)t * k + i];
        if (r < 0) continue;
        const float4 y = reinterpret_cast<const float4*>(yslot + (size_t)r * d)[c4];
        acc.x += y.x; acc.y += y.y; acc.z += y.z; acc.w += y.w;
    }
    T* o = out + (size_t)t * d + c4 * 4;
    o[0] = from_f32<T>(acc.x);
    o[1] = from_f32<T>(acc.y);
    o[2] = from_f32<T>(acc.z);
    o[3] = from_f32<T>(acc.w);
}

template <typename T>
cudaError_t run(const ace_layer* L, void* out, int T_, cudaStream_t s, cudaEvent_t* ev) {
    const ace_layer_desc& D = L->desc;
    const Workspace& W = L->ws;
    const int d = D.hidden, m = D.ffn, k = D.top_k;
    const int grid = L->num_sms * 4;
    const size_t smem1 = (size_t)kTC * d * sizeof(T);
    const size_t smem2 = (size_t)kTC * m * sizeof(float);
    if (ev) cudaEventRecord(ev[0], s);
    k_gemv_gateup<T><<<grid, 256, smem1, s>>>((const T*)W.h, (const T*)L->w_gate, (const T*)L->w_up,
                                              W.offsets, W.dlist, W.perm, W.meta, W.act, d, m, k);
    if (ev) cudaEventRecord(ev[1], s);
    k_gemv_down<T><<<grid, 256, smem2, s>>>(W.act, (const T*)L->w_down, W.ghat, W.offsets, W.dlist, W.perm,
                                            W.meta, W.yslot, d, m);
    const long long n = (long long)T_ * (d / 4);
    if (ev) cudaEventRecord(ev[2], s);
    k_combine<T><<<(int)((n + 255) / 256), 256, 0, s>>>(W.yslot, W.slot_pos, (T*)out, T_, d, k);
    if (ev) cudaEventRecord(ev[3], s);
    return cudaGetLastError();
}

}  // namespace

cudaError_t gemv_init(const ace_layer* L) {
    const int d = L->desc.hidden, m = L->desc.ffn;
    cudaError_t e;
    if (L->desc.dtype == ACE_BF16) {
        e = cudaFuncSetAttribute(k_gemv_gateup<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)(kTC * d * sizeof(__nv_bfloat16)));
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(k_gemv_down<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)(kTC * m * sizeof(float)));
    } else {
        e = cudaFuncSetAttribute(k_gemv_gateup<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)(kTC * d * sizeof(float)));
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(k_gemv_down<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)(kTC * m * sizeof(float)));
    }
    return e;
}

cudaError_t launch_experts_gemv(const ace_layer* L, void* out, int T, cudaStream_t s, cudaEvent_t* ev) {
    if (L->desc.dtype == ACE_BF16) return run<__nv_bfloat16>(L, out, T, s, ev);
    return run<float>(L, out, T, s, ev);
}

}  // namespace ace

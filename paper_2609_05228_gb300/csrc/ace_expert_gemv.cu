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

// Rows [lo, hi) of the flattened (distinct expert, weight row) space owned by
// this block: every block streams the same number of weight rows.
__device__ __forceinline__ void block_range(long long total, long long& lo, long long& hi) {
    lo = total * blockIdx.x / gridDim.x;
    hi = total * (blockIdx.x + 1) / gridDim.x;
}

// gate/up: one warp per row pair (W_gate[e, j], W_up[e, j]); each lane issues
// up to kCh 16-byte loads of each row before the dot products.
template <typename T>
__global__ void __launch_bounds__(256) k_gemv_gateup(const T* __restrict__ h, const T* __restrict__ w_gate,
                                                     const T* __restrict__ w_up,
                                                     const int32_t* __restrict__ offsets,
                                                     const int32_t* __restrict__ dlist,
                                                     const int32_t* __restrict__ perm,
                                                     const int32_t* __restrict__ meta,
                                                     float* __restrict__ act, int d, int m, int k) {
    constexpr int kCh = 8;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    uint4* hs = reinterpret_cast<uint4*>(smem_raw);     // [kTC][d / V] vectors
    constexpr int V = Vec16<T>::N;
    const int nvec = d / V;
    const int D = meta[kMetaDistinct];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
    long long lo, hi;
    block_range((long long)D * m, lo, hi);
    while (lo < hi) {
        const int e = dlist[lo / m];
        const int rb = (int)(lo % m);
        const int re = (int)min((long long)m, rb + (hi - lo));
        const int r0 = offsets[e], ne = offsets[e + 1] - r0;
        for (int tc0 = 0; tc0 < ne; tc0 += kTC) {
            const int ntc = min(kTC, ne - tc0);
            __syncthreads();
            for (int i = threadIdx.x; i < ntc * nvec; i += blockDim.x) {
                const int q = i / nvec, c = i % nvec;
                const int tok = perm[r0 + tc0 + q] / k;
                hs[i] = reinterpret_cast<const uint4*>(h + (size_t)tok * d)[c];
            }
            __syncthreads();
            for (int j = rb + warp; j < re; j += nwarps) {
                const uint4* wg = reinterpret_cast<const uint4*>(w_gate + ((size_t)e * m + j) * d);
                const uint4* wu = reinterpret_cast<const uint4*>(w_up + ((size_t)e * m + j) * d);
                float ag[kTC], au[kTC];
#pragma unroll
                for (int q = 0; q < kTC; ++q) { ag[q] = 0.f; au[q] = 0.f; }
                for (int c0 = 0; c0 < nvec; c0 += 32 * kCh) {
                    uint4 vg[kCh], vu[kCh];
#pragma unroll
                    for (int i = 0; i < kCh; ++i) {
                        const int c = c0 + lane + 32 * i;
                        const bool ok = c < nvec;
                        vg[i] = ok ? ld_stream(wg + c) : make_uint4(0, 0, 0, 0);
                        vu[i] = ok ? ld_stream(wu + c) : make_uint4(0, 0, 0, 0);
                    }
#pragma unroll
                    for (int i = 0; i < kCh; ++i) {
                        const int c = c0 + lane + 32 * i;
                        if (c >= nvec) break;
                        float fg[V], fu[V];
                        Vec16<T>::to_float(vg[i], fg);
                        Vec16<T>::to_float(vu[i], fu);
#pragma unroll
                        for (int q = 0; q < kTC; ++q) {
                            if (q < ntc) {
                                float fh[V];
                                Vec16<T>::to_float(hs[q * nvec + c], fh);
#pragma unroll
                                for (int t = 0; t < V; ++t) {
                                    ag[q] = fmaf(fh[t], fg[t], ag[q]);
                                    au[q] = fmaf(fh[t], fu[t], au[q]);
                                }
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
        lo += re - rb;
    }
}

// down: one warp per 4 rows W_down[e, c..c+3] (each m long); up to kCh
// 16-byte loads per row and lane are in flight before the dot products.
template <typename T>
__global__ void __launch_bounds__(256) k_gemv_down(const float* __restrict__ act, const T* __restrict__ w_down,
                                                   const float* __restrict__ ghat,
                                                   const int32_t* __restrict__ offsets,
                                                   const int32_t* __restrict__ dlist,
                                                   const int32_t* __restrict__ perm,
                                                   const int32_t* __restrict__ meta,
                                                   float* __restrict__ yslot, int d, int m) {
    constexpr int kCh = 4;
    constexpr int kRows = 4;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    float* as = reinterpret_cast<float*>(smem_raw);      // [kTC][m]
    __shared__ float gs[kTC];
    constexpr int V = Vec16<T>::N;
    const int nvec = m / V;
    const int D = meta[kMetaDistinct];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
    long long lo, hi;
    block_range((long long)D * d, lo, hi);
    while (lo < hi) {
        const int e = dlist[lo / d];
        const int rb = (int)(lo % d);
        const int re = (int)min((long long)d, rb + (hi - lo));
        const int r0 = offsets[e], ne = offsets[e + 1] - r0;
        for (int tc0 = 0; tc0 < ne; tc0 += kTC) {
            const int ntc = min(kTC, ne - tc0);
            __syncthreads();
            for (int i = threadIdx.x; i < ntc * (m / 4); i += blockDim.x) {
                const int q = i / (m / 4), c = i % (m / 4);
                reinterpret_cast<float4*>(as)[i] = reinterpret_cast<const float4*>(act + (size_t)(r0 + tc0 + q) * m)[c];
            }
            if (threadIdx.x < kTC) gs[threadIdx.x] = threadIdx.x < ntc ? ghat[perm[r0 + tc0 + threadIdx.x]] : 0.f;
            __syncthreads();
            for (int c = rb + warp * kRows; c < re; c += nwarps * kRows) {
                float acc[kRows][kTC];
#pragma unroll
                for (int r = 0; r < kRows; ++r)
#pragma unroll
                    for (int q = 0; q < kTC; ++q) acc[r][q] = 0.f;
                for (int v0 = 0; v0 < nvec; v0 += 32 * kCh) {
                    uint4 wv[kRows][kCh];
#pragma unroll
                    for (int r = 0; r < kRows; ++r) {
                        const uint4* wd = reinterpret_cast<const uint4*>(w_down + ((size_t)e * d + c + r) * m);
#pragma unroll
                        for (int i = 0; i < kCh; ++i) {
                            const int v = v0 + lane + 32 * i;
                            wv[r][i] = (c + r < re && v < nvec) ? ld_stream(wd + v) : make_uint4(0, 0, 0, 0);
                        }
                    }
#pragma unroll
                    for (int i = 0; i < kCh; ++i) {
                        const int v = v0 + lane + 32 * i;
                        if (v >= nvec) break;
#pragma unroll
                        for (int q = 0; q < kTC; ++q) {
                            if (q < ntc) {
                                float a[V];
                                const float4* ap = reinterpret_cast<const float4*>(as + q * m + v * V);
#pragma unroll
                                for (int t = 0; t < V / 4; ++t) {
                                    const float4 f = ap[t];
                                    a[4 * t] = f.x; a[4 * t + 1] = f.y; a[4 * t + 2] = f.z; a[4 * t + 3] = f.w;
                                }
#pragma unroll
                                for (int r = 0; r < kRows; ++r) {
                                    float fw[V];
                                    Vec16<T>::to_float(wv[r][i], fw);
#pragma unroll
                                    for (int t = 0; t < V; ++t) acc[r][q] = fmaf(a[t], fw[t], acc[r][q]);
                                }
                            }
                        }
                    }
                }
#pragma unroll
                for (int r = 0; r < kRows; ++r) {
#pragma unroll
                    for (int q = 0; q < kTC; ++q) {
                        if (q < ntc) {
                            const float y = warp_sum(acc[r][q]);
                            if (lane == 0 && c + r < re) yslot[(size_t)(r0 + tc0 + q) * d + c + r] = gs[q] * y;
                        }
                    }
                }
            }
        }
        lo += re - rb;
    }
}

// out[t, c] = sum_{i kept, rank order} y[slot_pos[t*k+i], c]
template <typename T>
__global__ void __launch_bounds__(256) k_combine(const float* __restrict__ yslot,
                                                 const int32_t* __restrict__ slot_pos, const T* __restrict__ resid,
                                                 T* __restrict__ out, int n_tokens, int d, int k) {
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
    if (resid) {
        const T* xr = resid + (size_t)t * d + c4 * 4;
        acc.x = to_f32(xr[0]) + acc.x;
        acc.y = to_f32(xr[1]) + acc.y;
        acc.z = to_f32(xr[2]) + acc.z;
        acc.w = to_f32(xr[3]) + acc.w;
    }
    T* o = out + (size_t)t * d + c4 * 4;
    o[0] = from_f32<T>(acc.x);
    o[1] = from_f32<T>(acc.y);
    o[2] = from_f32<T>(acc.z);
    o[3] = from_f32<T>(acc.w);
}

template <typename T>
cudaError_t run(const ace_layer* L, const void* x, void* out, int T_, cudaStream_t s, cudaEvent_t* ev) {
    const T* resid = L->desc.add_residual ? static_cast<const T*>(x) : nullptr;
    const ace_layer_desc& D = L->desc;
    const Workspace& W = L->ws;
    const int d = D.hidden, m = D.ffn, k = D.top_k;
    const int grid = L->num_sms * 2;
    const size_t smem1 = (size_t)kTC * d * sizeof(T);
    const size_t smem2 = (size_t)kTC * m * sizeof(float);
    k_gemv_gateup<T><<<grid, 256, smem1, s>>>((const T*)W.h, (const T*)L->w_gate, (const T*)L->w_up,
                                              W.offsets, W.dlist, W.perm, W.meta, W.act, d, m, k);
    if (ev) ace::record_stage(ev[1], s);
    k_gemv_down<T><<<grid, 256, smem2, s>>>(W.act, (const T*)L->w_down, W.ghat, W.offsets, W.dlist, W.perm,
                                            W.meta, W.yslot, d, m);
    const long long n = (long long)T_ * (d / 4);
    if (ev) ace::record_stage(ev[2], s);
    k_combine<T><<<(int)((n + 255) / 256), 256, 0, s>>>(W.yslot, W.slot_pos, resid, (T*)out, T_, d, k);
    if (ev) ace::record_stage(ev[3], s);
    return cudaGetLastError();
}

}  // namespace

cudaError_t gemv_init(const ace_layer* L) {
    const int d = L->desc.hidden, m = L->desc.ffn;
    cudaError_t e;
    if (L->desc.dtype == ACE_BF16) {
        e = raise_smem_limit(k_gemv_gateup<__nv_bfloat16>, (int)(kTC * d * sizeof(__nv_bfloat16)));
        if (e != cudaSuccess) return e;
        e = raise_smem_limit(k_gemv_down<__nv_bfloat16>, (int)(kTC * m * sizeof(float)));
    } else {
        e = raise_smem_limit(k_gemv_gateup<float>, (int)(kTC * d * sizeof(float)));
        if (e != cudaSuccess) return e;
        e = raise_smem_limit(k_gemv_down<float>, (int)(kTC * m * sizeof(float)));
    }
    return e;
}

cudaError_t launch_experts_gemv(const ace_layer* L, const void* x, void* out, int T, cudaStream_t s, cudaEvent_t* ev) {
    if (L->desc.dtype == ACE_BF16) return run<__nv_bfloat16>(L, x, out, T, s, ev);
    return run<float>(L, x, out, T, s, ev);
}

}  // namespace ace

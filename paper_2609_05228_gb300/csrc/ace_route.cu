// ace_route.cu — RMSNorm, router logits, top-k + gates, the Algorithm 4 skip
// decision, the App. B.1 per-batch threshold and the compaction of retained
// slots into per-expert groups.
//
// Two launch shapes share the same device functions (and so the same bits):
//   T <= kSmallT: k_route_fused, one launch for RMSNorm, router, top-k,
//                 decision, threshold and compaction;
//   larger T:     k_rmsnorm, router GEMM, k_topk_score, [k_sel_collect, k_sel_final],
//                 k_compact_count (+ the ratio-mode decision), k_compact_scan, k_compact_place.
#include <math.h>

#include "ace_device.cuh"
#include "ace_internal.h"

namespace ace {
namespace {

constexpr int kSmallT = 256;

// --------------------------------------------------------------------------
// RMSNorm (§3.1: expert and router input x = x_bar Gamma). One warp per token.
// h = x / sqrt(mean(x^2) + rms_eps) * gamma, computed in float, stored as T.
// --------------------------------------------------------------------------
// The row is read once into registers (all 16-byte loads issued before any
// arithmetic), then normalised from registers; supports d <= 32 * 16 * V.
constexpr int kNormVec = 16;

template <typename T, int NV = kNormVec>
__device__ __forceinline__ void rmsnorm_row(const T* __restrict__ xr, const T* __restrict__ gamma, T* hr, int d,
                                            float rms_eps, int lane) {
    constexpr int V = Vec16<T>::N;
    const int nvec = d / V;
    const uint4* xv = reinterpret_cast<const uint4*>(xr);
    const uint4* gv = reinterpret_cast<const uint4*>(gamma);
    uint4 xs[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        const int c = lane + 32 * i;
        xs[i] = c < nvec ? xv[c] : make_uint4(0, 0, 0, 0);
    }
    // sum of squares: one partial per 16-byte chunk (an fma chain from 0),
    // the lane's partials added in chunk order, then the warp butterfly --
    // the order every RMSNorm of the library uses
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        float f[V];
        Vec16<T>::to_float(xs[i], f);
        float part = 0.f;
#pragma unroll
        for (int j = 0; j < V; ++j) part = fmaf(f[j], f[j], part);
        ss += part;
    }
    ss = warp_sum(ss);
    const float inv = 1.0f / sqrtf(ss / (float)d + rms_eps);
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        const int c = lane + 32 * i;
        if (c < nvec) {
            float f[V], gm[V];
            Vec16<T>::to_float(xs[i], f);
            Vec16<T>::to_float(gv[c], gm);
            T o[V];
#pragma unroll
            for (int j = 0; j < V; ++j) o[j] = from_f32<T>(f[j] * inv * gm[j]);
            reinterpret_cast<uint4*>(hr)[c] = *reinterpret_cast<const uint4*>(o);
        }
    }
}

__device__ __forceinline__ void cp_async16_row(uint32_t dst, const void* src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}

// A warp per row. The row comes into shared memory by cp.async (d x sizeof(T)
// bytes per warp of dynamic shared memory), so no registers are held per load
// and more rows are in flight per SM; each lane reads back only its own
// 16-byte chunks (lane + 32 i), in the order and with the arithmetic of
// rmsnorm_row, so the bits are the same. NV bounds the chunks per lane.
template <typename T, int NV>
__global__ void __launch_bounds__(256) k_rmsnorm(const T* __restrict__ x, const T* __restrict__ gamma,
                                                 T* __restrict__ h, int n_tokens, int d, float rms_eps) {
    extern __shared__ __align__(16) unsigned char rn_rows[];      // [warps][d] staged rows
    pdl_wait();
    const int wib = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int row = blockIdx.x * (blockDim.x >> 5) + wib;
    if (row >= n_tokens) return;
    constexpr int V = Vec16<T>::N;
    const int nvec = d / V;
    const uint4* xv = reinterpret_cast<const uint4*>(x + (size_t)row * d);
    const uint4* rs = reinterpret_cast<const uint4*>(rn_rows + (size_t)wib * d * sizeof(T));
    const uint32_t rs_addr = (uint32_t)__cvta_generic_to_shared(rs);
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        const int c = lane + 32 * i;
        if (c < nvec) cp_async16_row(rs_addr + (uint32_t)c * 16u, xv + c);
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        const int c = lane + 32 * i;
        if (c < nvec) {
            float f[V];
            Vec16<T>::to_float(rs[c], f);
            float part = 0.f;
#pragma unroll
            for (int j = 0; j < V; ++j) part = fmaf(f[j], f[j], part);
            ss += part;
        }
    }
    ss = warp_sum(ss);
    const float inv = 1.0f / sqrtf(ss / (float)d + rms_eps);
    const uint4* gv = reinterpret_cast<const uint4*>(gamma);
    uint4* hv = reinterpret_cast<uint4*>(h + (size_t)row * d);
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        const int c = lane + 32 * i;
        if (c < nvec) {
            float f[V], gm[V];
            Vec16<T>::to_float(rs[c], f);
            Vec16<T>::to_float(gv[c], gm);
            T o[V];
#pragma unroll
            for (int j = 0; j < V; ++j) o[j] = from_f32<T>(f[j] * inv * gm[j]);
            hv[c] = *reinterpret_cast<const uint4*>(o);
        }
    }
}

// --------------------------------------------------------------------------
// Router logits z[t,e] = (h_t . w_e + b_e) / temp  (§3.2 logit). A block
// covers kRouterTok tokens x 8 experts (one expert row per warp): the token
// rows of h sit in shared memory and every lane issues its share of the
// expert row (up to 8 x 16 bytes) before the dot products. With FUSE_NORM
// the block computes the RMSNorm of its tokens from x itself, and blocks
// with blockIdx.y == 0 also store h for the experts.
// --------------------------------------------------------------------------
constexpr int kRouterTok = 16;
constexpr int kRouterExp = 8;

template <typename T, bool FUSE_NORM>
__global__ void __launch_bounds__(256) k_router(const T* __restrict__ src, const T* __restrict__ gamma,
                                                T* __restrict__ h_out, const T* __restrict__ w,
                                                const float* __restrict__ b, float* __restrict__ z,
                                                int n_tokens, int d, int n_exp, float inv_temp,
                                                int use_temp, float rms_eps) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    uint4* hs = reinterpret_cast<uint4*>(smem_raw);
    const int t0 = blockIdx.x * kRouterTok;
    const int nt = min(kRouterTok, n_tokens - t0);
    constexpr int V = Vec16<T>::N;
    const int nvec = d / V;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (FUSE_NORM) {
        T* hsr = reinterpret_cast<T*>(smem_raw);
        for (int r = warp; r < kRouterTok; r += blockDim.x >> 5) {
            if (r < nt) {
                rmsnorm_row(src + (size_t)(t0 + r) * d, gamma, hsr + (size_t)r * d, d, rms_eps, lane);
            } else {
                for (int c = lane; c < nvec; c += 32) hs[r * nvec + c] = make_uint4(0, 0, 0, 0);
            }
        }
        __syncthreads();
        if (blockIdx.y == 0) {
            for (int i = threadIdx.x; i < nt * nvec; i += blockDim.x) {
                const int r = i / nvec, c = i % nvec;
                reinterpret_cast<uint4*>(h_out + (size_t)(t0 + r) * d)[c] = hs[i];
            }
        }
    } else {
        for (int i = threadIdx.x; i < kRouterTok * nvec; i += blockDim.x) {
            const int r = i / nvec, c = i % nvec;
            uint4 v = make_uint4(0, 0, 0, 0);
            if (r < nt) v = reinterpret_cast<const uint4*>(src + (size_t)(t0 + r) * d)[c];
            hs[i] = v;
        }
        __syncthreads();
    }
    const int e = blockIdx.y * kRouterExp + warp;
    if (e >= n_exp) return;
    const uint4* we = reinterpret_cast<const uint4*>(w + (size_t)e * d);
    float acc[kRouterTok];
#pragma unroll
    for (int r = 0; r < kRouterTok; ++r) acc[r] = 0.f;
    constexpr int CH = 8;
    for (int c0 = 0; c0 < nvec; c0 += 32 * CH) {
        uint4 wv[CH];
#pragma unroll
        for (int i = 0; i < CH; ++i) {
            const int c = c0 + lane + 32 * i;
            wv[i] = c < nvec ? we[c] : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int i = 0; i < CH; ++i) {
            const int c = c0 + lane + 32 * i;
            if (c >= nvec) break;
            float wf[V];
            Vec16<T>::to_float(wv[i], wf);
#pragma unroll
            for (int r = 0; r < kRouterTok; ++r) {
                if (r < nt) {
                    float hf[V];
                    Vec16<T>::to_float(hs[r * nvec + c], hf);
#pragma unroll
                    for (int j = 0; j < V; ++j) acc[r] = fmaf(hf[j], wf[j], acc[r]);
                }
            }
        }
    }
#pragma unroll
    for (int r = 0; r < kRouterTok; ++r)
        if (r < nt) acc[r] = warp_sum(acc[r]);
    if (lane < nt) {
        float v = acc[0];
#pragma unroll
        for (int r = 1; r < kRouterTok; ++r) if (lane == r) v = acc[r];
        v = v + b[e];
        if (use_temp) v = v * inv_temp;
        z[(size_t)(t0 + lane) * n_exp + e] = v;
    }
}

// --------------------------------------------------------------------------
// Per-token decision, float32 in a fixed operation order (Algorithm 4).
// Lane i < k holds slot i (rank i). Every sum is taken sequentially in rank
// order through shuffles, so all lanes hold identical totals.
// --------------------------------------------------------------------------
struct SlotScore {
    float g;   // gate
    float c;   // score of the skip rule (ACE: max(p_gsp, p_rcr))
};

// Top-k over one token's logits (one warp). Lane l owns experts l + 32 j,
// j < NPL, held in registers. Order: larger logit first; ties to the lower
// expert index. NaN ranks last (as -inf), -0 equals +0. On return lane i < k
// holds (id, z) of rank i. Each round takes two warp reductions: the largest
// key (the logit mapped to an order-preserving unsigned integer), then the
// lowest expert index holding it.
__device__ __forceinline__ uint32_t order_key(float f) {
    const uint32_t u = __float_as_uint(__fadd_rn(f, 0.0f));     // -0 -> +0
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float key_value(uint32_t k) {
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

template <int NPL>
__device__ __forceinline__ void warp_topk(const float* __restrict__ zrow, int n_exp, int k, int lane,
                                          int& my_id, float& my_z, bool& saw_nan) {
    uint32_t v[NPL];
    saw_nan = false;
#pragma unroll
    for (int j = 0; j < NPL; ++j) {
        const int e = lane + 32 * j;
        if (e < n_exp) {
            float z = __ldcg(zrow + e);
            if (z != z) { saw_nan = true; z = -INFINITY; }
            v[j] = order_key(z);
        } else {
            v[j] = 0u;                       // below every real key: never chosen
        }
    }
    my_id = -1;
    my_z = 0.f;
    if (NPL <= 8) {
        // sort the lane's keys once (larger first, lower j first on ties: a
        // stable insertion network), then each round takes the largest head
        int jj[NPL];
#pragma unroll
        for (int j = 0; j < NPL; ++j) jj[j] = j;
#pragma unroll
        for (int a = 1; a < NPL; ++a) {
#pragma unroll
            for (int b = a; b > 0; --b) {
                const bool sw = v[b] > v[b - 1];
                const uint32_t tv = sw ? v[b] : v[b - 1];
                v[b] = sw ? v[b - 1] : v[b];
                v[b - 1] = tv;
                const int tj = sw ? jj[b] : jj[b - 1];
                jj[b] = sw ? jj[b - 1] : jj[b];
                jj[b - 1] = tj;
            }
        }
        for (int r = 0; r < k; ++r) {
            const uint32_t top = __reduce_max_sync(0xffffffffu, v[0]);
            const uint32_t e = __reduce_min_sync(0xffffffffu, (v[0] == top && top != 0u) ? (uint32_t)(lane + 32 * jj[0])
                                                                                       : 0xffffffffu);
            if ((int)(e & 31u) == lane) {
#pragma unroll
                for (int j = 0; j < NPL - 1; ++j) { v[j] = v[j + 1]; jj[j] = jj[j + 1]; }
                v[NPL - 1] = 0u;
            }
            if (lane == r) { my_id = (int)e; my_z = key_value(top); }
        }
    } else {
        unsigned taken = 0u;   // bit j: expert lane + 32*j chosen already
        for (int r = 0; r < k; ++r) {
            uint32_t bk = 0u;
            int bj = -1;
#pragma unroll
            for (int j = 0; j < NPL; ++j)
                if (!((taken >> j) & 1u) && v[j] != 0u && (bj < 0 || v[j] > bk)) { bk = v[j]; bj = j; }
            const uint32_t top = __reduce_max_sync(0xffffffffu, bj >= 0 ? bk : 0u);
            const uint32_t e = __reduce_min_sync(0xffffffffu, (bj >= 0 && bk == top) ? (uint32_t)(lane + 32 * bj)
                                                                                      : 0xffffffffu);
            if ((int)(e & 31u) == lane) taken |= 1u << (e >> 5);
            if (lane == r) { my_id = (int)e; my_z = key_value(top); }
        }
    }
}

// c of a skip rule from the two views and the gate (ace_fusion).
__device__ __forceinline__ float fuse_views(float pg, float pr, float g, int fusion) {
    switch (fusion) {
        case ACE_FUSION_MIN: return fminf(pg, pr);
        case ACE_FUSION_MEAN: return __fmul_rn(__fadd_rn(pg, pr), 0.5f);
        case ACE_FUSION_GSP: return pg;
        case ACE_FUSION_RCR: return pr;
        case ACE_FUSION_SCORE: return g;
        default: return fmaxf(pg, pr);                          // Eq. ace_contribution
    }
}

// Gates and c for the slot held by this lane (lanes >= k return zeros).
__device__ __forceinline__ SlotScore score_slot(int lane, int k, float z_i, float z_0, int id,
                                                const float* __restrict__ a_gsp,
                                                const float* __restrict__ a_rcr, float eps, int fusion) {
    const bool on = lane < k;
    const float e_i = on ? ace_exp32(__fsub_rn(z_i, z_0)) : 0.f;
    float s = __shfl_sync(0xffffffffu, e_i, 0);
    for (int j = 1; j < k; ++j) s = __fadd_rn(s, __shfl_sync(0xffffffffu, e_i, j));
    const float g = on ? __fdiv_rn(e_i, s) : 0.f;
    const float sg = on ? __fmul_rn(g, a_gsp[id]) : 0.f;       // Eq. gsp_contribution
    const float sr = on ? __fmul_rn(g, a_rcr[id]) : 0.f;       // Eq. rcr_contribution
    float zg = __shfl_sync(0xffffffffu, sg, 0);
    float zr = __shfl_sync(0xffffffffu, sr, 0);
    for (int j = 1; j < k; ++j) {
        zg = __fadd_rn(zg, __shfl_sync(0xffffffffu, sg, j));
        zr = __fadd_rn(zr, __shfl_sync(0xffffffffu, sr, j));
    }
    zg = __fadd_rn(zg, eps);
    zr = __fadd_rn(zr, eps);
    const float pg = on ? __fdiv_rn(sg, zg) : 0.f;              // Eq. gsp_probability
    const float pr = on ? __fdiv_rn(sr, zr) : 0.f;              // Eq. rcr_probability
    return SlotScore{g, on ? fuse_views(pg, pr, g, fusion) : 0.f};
}

// Slots excluded from the threshold search (App. B.1): rank 0 (the top-1)
// and the m_min-1 highest-c other slots, the ones Algorithm 4 restores first.
__device__ __forceinline__ bool slot_protected(int lane, int k, float c, int m_min) {
    bool prot = lane == 0;
    const int extra = min(m_min, k) - 1;
    if (extra > 0) {
        int better = 0;   // non-top-1 slots ahead of this one in (c desc, rank asc)
        for (int j = 1; j < k; ++j) {
            const float cj = __shfl_sync(0xffffffffu, c, j);
            if (j != lane && (cj > c || (cj == c && j < lane))) ++better;
        }
        if (lane != 0 && better < extra) prot = true;
    }
    return prot;
}

// Skip flag and g_hat for the slot of this lane, given tau.
__device__ __forceinline__ void decide_slot(int lane, int k, float g, float c, float tau, int m_min,
                                            float eps, bool& skip_out, float& ghat_out) {
    const bool on = lane < k;
    // candidate when c < tau (for ACE, Eq. ace_candidate_intersection via max);
    // slot 0 is the top-1 and is kept.
    bool skip = on && lane != 0 && (c < tau);
    const unsigned sk = __ballot_sync(0xffffffffu, skip);
    const int active = k - __popc(sk);
    if (active < m_min) {
        // restore skipped slots in c-descending order, lower rank first on ties
        int need = m_min - active;
        unsigned rem = sk;
        while (need > 0 && rem) {
            float best = -1.f;
            int bi = -1;
            for (unsigned mm = rem; mm; mm &= mm - 1) {
                const int j = __ffs(mm) - 1;
                const float cj = __shfl_sync(0xffffffffu, c, j);
                if (bi < 0 || cj > best) { best = cj; bi = j; }
            }
            rem &= ~(1u << bi);
            if (lane == bi) skip = false;
            --need;
        }
    }
    const unsigned keep = __ballot_sync(0xffffffffu, on && !skip);
    float zs = 0.f;
    for (int j = 0; j < k; ++j) {
        const float gj = __shfl_sync(0xffffffffu, g, j);
        if ((keep >> j) & 1u) zs = __fadd_rn(zs, gj);
    }
    zs = __fadd_rn(zs, eps);
    skip_out = skip;
    ghat_out = (on && !skip) ? __fdiv_rn(g, zs) : 0.f;
}

// The same decision with one thread per token: the token's k gates and c
// values sit in registers (loops fully unrolled over kMaxTopK), and every
// step -- the skip test, the restore order, the rank-order sum and the
// division -- is the one decide_slot takes, so the bits agree.
__device__ __forceinline__ void decide_token(const float* g_in, const float* c_in, int k, float tau, int m_min,
                                             float eps, uint8_t* skip_out, float* ghat_out,
                                             uint8_t* skip_copy) {
    float g[kMaxTopK], c[kMaxTopK];
    unsigned sk = 0u;
#pragma unroll
    for (int j = 0; j < kMaxTopK; ++j) {
        g[j] = j < k ? g_in[j] : 0.f;
        c[j] = j < k ? c_in[j] : 0.f;
        if (j < k && j != 0 && c[j] < tau) sk |= 1u << j;   // candidate: c < tau
    }
    int need = m_min - (k - __popc(sk));
    while (need > 0 && sk) {
        // restore the skipped slot of largest c, lower rank first on ties
        float best = -1.f;
        int bi = -1;
#pragma unroll
        for (int j = 0; j < kMaxTopK; ++j)
            if (((sk >> j) & 1u) && (bi < 0 || c[j] > best)) { best = c[j]; bi = j; }
        sk &= ~(1u << bi);
        --need;
    }
    float zs = 0.f;
#pragma unroll
    for (int j = 0; j < kMaxTopK; ++j)
        if (j < k && !((sk >> j) & 1u)) zs = __fadd_rn(zs, g[j]);
    zs = __fadd_rn(zs, eps);
#pragma unroll
    for (int j = 0; j < kMaxTopK; ++j) {
        if (j < k) {
            const bool s = (sk >> j) & 1u;
            skip_out[j] = s ? 1 : 0;
            if (skip_copy) skip_copy[j] = s ? 1 : 0;
            ghat_out[j] = s ? 0.f : __fdiv_rn(g[j], zs);
        }
    }
}

// --------------------------------------------------------------------------
// App. B.1 threshold for m candidates to skip: the (m+1)-th smallest
// candidate key v (radix select over the non-negative float bits, 8 bits per
// pass), lo = #{c < v}, hi = #{c <= v}; tau = v when lo == m or when lo is at
// least as close to m as hi, else the next float above v. Whole block;
// requires 0 < m < #candidates. Keys 0xffffffff are protected slots.
// --------------------------------------------------------------------------
// One shared 256-bin histogram per pass, filled with one atomic per distinct
// bin of a warp (the keys cluster: c lies in [0, 1]); a block-wide scan
// (thread b owns bin b; blockDim.x == 256) finds the digit.
template <int NW>
struct SelectSmem {
    int hist[256];
    int wtot[NW];
    uint32_t prefix;
    int want, below, last_cnt;
    float tau;
};

template <int NW>
__device__ float block_select_tau(const uint32_t* keys, int n, int m, SelectSmem<NW>& S) {
    static_assert(NW * 32 == 256, "one thread per bin");
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    uint32_t prefix = 0u, mask = 0u;
    int want = m, below = 0, last_cnt = 0;
    for (int pass = 0; pass < 4; ++pass) {
        const int shift = 24 - 8 * pass;
        S.hist[tid] = 0;
        __syncthreads();
        for (int i0 = 0; i0 < n; i0 += 256) {
            const int i = i0 + tid;
            const uint32_t key = i < n ? keys[i] : 0xffffffffu;
            if (key != 0xffffffffu && (key & mask) == prefix) {
                const int bin = (int)((key >> shift) & 255u);
                const unsigned peers = __match_any_sync(__activemask(), bin);
                if (lane == __ffs(peers) - 1) atomicAdd(&S.hist[bin], __popc(peers));
            }
        }
        __syncthreads();
        const int v = S.hist[tid];
        int inc = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= o) inc += y;
        }
        if (lane == 31) S.wtot[warp] = inc;
        __syncthreads();
        int base = 0;
#pragma unroll
        for (int w = 0; w < NW; ++w) base += w < warp ? S.wtot[w] : 0;
        const int exc = base + inc - v;
        // the owner of `want`; the last bin if want lies past every count
        if ((exc <= want && want < exc + v) || (tid == 255 && want >= exc + v)) {
            S.prefix = prefix | ((uint32_t)tid << shift);
            S.want = want - exc;
            S.below = below + exc;
            S.last_cnt = v;
        }
        __syncthreads();
        prefix = S.prefix;
        want = S.want;
        below = S.below;
        last_cnt = S.last_cnt;
        mask |= 255u << shift;
        __syncthreads();                     // S is rewritten by the next pass
    }
    const int lo = below, hi = below + last_cnt;
    float tau = __uint_as_float(prefix);
    if (!(lo == m || (m - lo) <= (hi - m))) tau = __uint_as_float(prefix + 1u);
    return tau;
}

// The same threshold for at most blockDim.x keys, by counting ranks: key i
// (not protected) is v when lt_i <= m < le_i, with lt_i = #{keys < key i} and
// le_i = #{keys <= key i} (a protected 0xffffffff key is above every
// candidate, so it counts in neither); then lo = lt_i and hi = le_i. One pass
// over the keys and one barrier, against the radix select's four passes of
// five barriers each: faster up to about 128 keys. The caller sets S.prefix /
// S.below / S.last_cnt beforehand and synchronises (the values stay if no key
// qualifies, which 0 < m < #candidates rules out).
template <int NW>
__device__ float block_select_tau_rank(const uint32_t* keys, int n, int m, SelectSmem<NW>& S) {
    const int i = threadIdx.x;
    const uint32_t ki = i < n ? keys[i] : 0xffffffffu;
    int lt = 0, le = 0;
#pragma unroll 8
    for (int j = 0; j < n; ++j) {
        const uint32_t kj = keys[j];
        lt += kj < ki;
        le += kj <= ki;
    }
    if (ki != 0xffffffffu && lt <= m && m < le) {
        S.prefix = ki;
        S.below = lt;
        S.last_cnt = le - lt;
    }
    __syncthreads();
    const uint32_t v = S.prefix;
    const int lo = S.below, hi = S.below + S.last_cnt;
    float tau = __uint_as_float(v);
    if (!(lo == m || (m - lo) <= (hi - m))) tau = __uint_as_float(v + 1u);
    return tau;
}

// Exclusive scan of cnt[0..n_exp) by the whole block (called by every
// thread; blockDim.x a multiple of 32, at most 1024): offsets[e],
// offsets[n_exp] = total, the distinct-expert list (increasing) and the meta
// totals; also off_s (shared) when given. With tok_tile > 0 it also writes
// tt_off[j] = sum over distinct experts before j of ceil(count / tok_tile)
// (the token-tile schedule of the tensor-core experts) and tt_off[D].
// Each thread scans a contiguous run of experts; the three running sums are
// combined by warp shuffles and one pass over the per-warp totals in wsum
// (shared, 3 x 32 ints).
__device__ void scan_counts_block(const int* cnt, int n_exp, int32_t* __restrict__ offsets,
                                  int32_t* __restrict__ dlist, int32_t* __restrict__ meta, int* off_s,
                                  int tok_tile, int32_t* __restrict__ tt_off, int* wsum) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
    const int per = (n_exp + blockDim.x - 1) / blockDim.x;
    const int e0 = min(tid * per, n_exp), e1 = min(e0 + per, n_exp);
    const int tt = tok_tile > 0 ? tok_tile : 1;
    int s = 0, dcount = 0, tiles = 0;
    for (int e = e0; e < e1; ++e) {
        const int c = cnt[e];
        s += c;
        dcount += c > 0;
        tiles += (c + tt - 1) / tt;
    }
    int xs = s, xd = dcount, xt = tiles;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int ys = __shfl_up_sync(0xffffffffu, xs, o);
        const int yd = __shfl_up_sync(0xffffffffu, xd, o);
        const int yt = __shfl_up_sync(0xffffffffu, xt, o);
        if (lane >= o) { xs += ys; xd += yd; xt += yt; }
    }
    if (lane == 31) { wsum[warp] = xs; wsum[32 + warp] = xd; wsum[64 + warp] = xt; }
    __syncthreads();
    if (warp == 0) {
        int vs = lane < nw ? wsum[lane] : 0, vd = lane < nw ? wsum[32 + lane] : 0, vt = lane < nw ? wsum[64 + lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int ys = __shfl_up_sync(0xffffffffu, vs, o);
            const int yd = __shfl_up_sync(0xffffffffu, vd, o);
            const int yt = __shfl_up_sync(0xffffffffu, vt, o);
            if (lane >= o) { vs += ys; vd += yd; vt += yt; }
        }
        wsum[lane] = vs;
        wsum[32 + lane] = vd;
        wsum[64 + lane] = vt;
    }
    __syncthreads();
    int run = xs - s + (warp ? wsum[warp - 1] : 0);
    int drun = xd - dcount + (warp ? wsum[32 + warp - 1] : 0);
    int trun = xt - tiles + (warp ? wsum[64 + warp - 1] : 0);
    for (int e = e0; e < e1; ++e) {
        const int c = cnt[e];
        offsets[e] = run;
        if (off_s) off_s[e] = run;
        run += c;
        if (c > 0) {
            if (tok_tile > 0) tt_off[drun] = trun;
            trun += (c + tt - 1) / tt;
            dlist[drun++] = e;
        }
    }
    if (tid == blockDim.x - 1) {       // its running sums end at the totals
        offsets[n_exp] = run;
        if (off_s) off_s[n_exp] = run;
        if (tok_tile > 0) tt_off[drun] = trun;
        meta[kMetaRetained] = run;
        meta[kMetaDistinct] = drun;
        meta[kMetaTokTiles] = tok_tile > 0 ? trun : 0;
    }
    __syncthreads();                   // wsum may be reused by the caller
}

// After scan_counts_block and a block barrier: the flat token-tile table of
// the tensor-core experts, tt_tab[tt] = (expert, first row, rows, 0).
// tt_cap: entries allocated in tt_tab (checked by the debug build).
__device__ void fill_tile_table(const int32_t* offsets, const int32_t* dlist, const int32_t* tt_off,
                                const int32_t* meta, int tok_tile, int4* tt_tab, int n_exp, int tt_cap, int* err) {
    if (tok_tile <= 0) return;
    const int D = meta[kMetaDistinct];
    for (int j = threadIdx.x; j < D; j += blockDim.x) {
        const int e = dlist[j];
        if (!ACE_IDX_OK((unsigned)e < (unsigned)n_exp, err)) continue;
        const int beg = offsets[e], cnt = offsets[e + 1] - beg, base = tt_off[j];
        for (int b = 0; b * tok_tile < cnt; ++b) {
            if (!ACE_IDX_OK(base + b >= 0 && base + b < tt_cap, err)) break;
            tt_tab[base + b] = make_int4(e, beg + b * tok_tile, min(tok_tile, cnt - b * tok_tile), 0);
        }
    }
}

// --------------------------------------------------------------------------
// Large-T kernels
// --------------------------------------------------------------------------

// Pass 1: top-k, gates, c; one warp per token, 32 tokens per block.
// THRESHOLD mode also decides. RATIO mode writes the candidate keys (float
// bits of c, or 0xffffffff for protected slots) and adds the block's
// histogram of their top 12 bits (shared memory first, then one global
// atomic per non-empty bin) to ghist, the first digit of the threshold select.
constexpr int kTopkWarps = 32;
constexpr int kHistBins = 4096;

template <int NPL>
__global__ void __launch_bounds__(kTopkWarps * 32) k_topk_score(float* __restrict__ logits, int n_tokens,
                                                                int n_exp, int k, const float* __restrict__ a_gsp,
                                                                const float* __restrict__ a_rcr, float eps,
                                                                int m_min, int mode, float tau,
                                                                int32_t* __restrict__ ids, float* __restrict__ gates,
                                                                float* __restrict__ cval, uint32_t* __restrict__ keys,
                                                                uint8_t* __restrict__ skip, float* __restrict__ ghat,
                                                                float* __restrict__ tau_out, int* __restrict__ err,
                                                                int32_t* __restrict__ ghist,
                                                                const float* __restrict__ part, int n_split,
                                                                const float* __restrict__ bias, float inv_temp,
                                                                int use_temp, int fusion) {
    __shared__ int hist[kHistBins];
    const bool ratio = mode == ACE_SKIP_RATIO;
    if (ratio)
        for (int i = threadIdx.x; i < kHistBins; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    pdl_wait();
    if (!ratio && blockIdx.x == 0 && threadIdx.x == 0) *tau_out = tau;
    const int t = blockIdx.x * kTopkWarps + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (t < n_tokens) {
        if (n_split > 1) {
            // split-K router: z = (sum of the slices in order + b) / temp
            const size_t stride = (size_t)n_tokens * n_exp;
            for (int e = lane; e < n_exp; e += 32) {
                const size_t o = (size_t)t * n_exp + e;
                float z = __ldcg(part + o);
                for (int sp = 1; sp < n_split; ++sp) z += __ldcg(part + sp * stride + o);
                z = z + bias[e];
                if (use_temp) z = z * inv_temp;
                logits[o] = z;
            }
            __syncwarp();
        }
        int id;
        float zv;
        bool nan;
        warp_topk<NPL>(logits + (size_t)t * n_exp, n_exp, k, lane, id, zv, nan);
        if (lane < k && !ACE_IDX_OK((unsigned)id < (unsigned)n_exp, err)) id = 0;   // tables are read at id
        const float z0 = __shfl_sync(0xffffffffu, zv, 0);
        if (__any_sync(0xffffffffu, nan) && lane == 0) atomicOr(err, kErrNumeric);
        const SlotScore sc = score_slot(lane, k, zv, z0, lane < k ? id : 0, a_gsp, a_rcr, eps, fusion);
        const size_t base = (size_t)t * k;
        if (lane < k) {
            ids[base + lane] = id;
            gates[base + lane] = sc.g;
            cval[base + lane] = sc.c;
        }
        if (!ratio) {
            bool sk;
            float gh;
            decide_slot(lane, k, sc.g, sc.c, tau, m_min, eps, sk, gh);
            if (lane < k) {
                skip[base + lane] = sk ? 1 : 0;
                ghat[base + lane] = gh;
            }
        } else {
            const bool prot = slot_protected(lane, k, sc.c, m_min);
            const uint32_t key = prot ? 0xffffffffu : __float_as_uint(sc.c);
            if (lane < k) keys[base + lane] = key;
            if (lane < k && !prot) {
                const int bin = (int)(key >> 20);
                const unsigned peers = __match_any_sync(__activemask(), bin);
                if (lane == __ffs(peers) - 1) atomicAdd(&hist[bin], __popc(peers));
            }
        }
    }
    if (ratio) {
        __syncthreads();
        for (int i = threadIdx.x; i < kHistBins; i += blockDim.x)
            if (hist[i]) atomicAdd(&ghist[i], hist[i]);
    }
}

// Exclusive prefix of v over a 1024-thread block (thread order); total = sum.
__device__ __forceinline__ int block_exscan_1024(int v, int* wtot, int& total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += y;
    }
    if (lane == 31) wtot[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        int wi = wtot[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += y;
        }
        wtot[lane] = wi;
    }
    __syncthreads();
    const int exc = inc - v + (warp ? wtot[warp - 1] : 0);
    total = wtot[31];
    __syncthreads();
    return exc;
}

// App. B.1 threshold for large T: the (m+1)-th smallest candidate key v,
// lo = #{c < v}, hi = #{c <= v}; tau = v when lo == m or lo is at least as
// close to m as hi, else the next float above v. The key is taken as three
// digits (bits 31..20, 19..10, 9..0):
//   k_topk_score  adds the digit-1 histogram (4096 bins, hist1);
//   k_sel_collect (many blocks) finds digit 1 from hist1 (every block, the
//                 same way), appends the keys inside it to cand and adds
//                 their digit-2 histogram (1024 bins, hist2); KPT keys per
//                 thread, chosen so the grid spans the SMs (its time is the
//                 latency of the hist1 and key loads, not bandwidth);
//   k_sel_final   (one block) finds digit 2, then digit 3 over cand, writes
//                 tau and re-zeroes hist1, hist2 and the candidate count.

// Block-wide digit search over `bins` = 1024 * per counts held per thread:
// the owner of rank `want` records prefix | digit << shift in S.
struct SelShared {
    int wtot[32];
    uint32_t prefix;
    int want, below, last;
};

template <int PER>
__device__ __forceinline__ void find_digit(const int (&b)[PER], int want, uint32_t prefix, int shift, int below,
                                           SelShared& S) {
    int total;
    int loc = 0;
#pragma unroll
    for (int j = 0; j < PER; ++j) loc += b[j];
    const int exc = block_exscan_1024(loc, S.wtot, total);
    if ((exc <= want && want < exc + loc) || (threadIdx.x == 1023 && want >= total)) {
        int cum = exc, j = 0;
        while (j < PER - 1 && cum + b[j] <= want) { cum += b[j]; ++j; }
        S.prefix = prefix | ((uint32_t)(PER * threadIdx.x + j) << shift);
        S.want = want - cum;
        S.below = below + cum;
        S.last = b[j];
    }
    __syncthreads();
}

template <int KPT>
__global__ void __launch_bounds__(1024) k_sel_collect(const uint32_t* __restrict__ keys, int n, int m,
                                                      const int32_t* __restrict__ hist1,
                                                      int32_t* __restrict__ hist2, uint32_t* __restrict__ cand,
                                                      int32_t* __restrict__ meta, int* err) {
    __shared__ SelShared S;
    __shared__ int h2[1024];
    const int tid = threadIdx.x, lane = tid & 31;
    h2[tid] = 0;
    pdl_wait();
    int b[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) b[j] = __ldcg(hist1 + 4 * tid + j);
    find_digit<4>(b, m, 0u, 20, 0, S);
    const uint32_t prefix = S.prefix;
    if (blockIdx.x == 0 && tid == 0) {
        meta[kMetaSelPrefix] = (int32_t)prefix;
        meta[kMetaSelWant] = S.want;
        meta[kMetaSelBelow] = S.below;
    }
    // this block's keys: KPT per thread (16-byte loads when KPT is a multiple of 4)
    const int base = (blockIdx.x * 1024 + tid) * KPT;
    uint32_t kv[KPT];
    if (KPT % 4 == 0 && base + KPT <= n) {
#pragma unroll
        for (int j = 0; j + 3 < KPT; j += 4) {
            const uint4 v = __ldcg(reinterpret_cast<const uint4*>(keys + base + j));
            kv[j] = v.x; kv[j + 1] = v.y; kv[j + 2] = v.z; kv[j + 3] = v.w;
        }
    } else {
#pragma unroll
        for (int j = 0; j < KPT; ++j) kv[j] = base + j < n ? __ldcg(keys + base + j) : 0xffffffffu;
    }
#pragma unroll
    for (int j = 0; j < KPT; ++j) {
        const bool in = kv[j] != 0xffffffffu && (kv[j] & 0xFFF00000u) == prefix;
        const unsigned bal = __ballot_sync(0xffffffffu, in);
        if (!bal) continue;
        int pos = 0;
        if (lane == 0) pos = atomicAdd(&meta[kMetaSelCount], __popc(bal));
        pos = __shfl_sync(0xffffffffu, pos, 0) + __popc(bal & lanemask_lt());
        if (in && ACE_IDX_OK(pos < n, err)) {
            cand[pos] = kv[j];
            const int bin = (int)((kv[j] >> 10) & 1023u);
            const unsigned peers = __match_any_sync(bal, bin);
            if (lane == __ffs(peers) - 1) atomicAdd(&h2[bin], __popc(peers));
        }
    }
    __syncthreads();
    if (h2[tid]) atomicAdd(&hist2[tid], h2[tid]);
}

__global__ void __launch_bounds__(1024) k_sel_final(int m, int32_t* __restrict__ hist1, int32_t* __restrict__ hist2,
                                                    const uint32_t* __restrict__ cand, int32_t* __restrict__ meta,
                                                    float* __restrict__ tau_out) {
    __shared__ SelShared S;
    __shared__ int h3[1024];
    const int tid = threadIdx.x, lane = tid & 31;
    h3[tid] = 0;
    pdl_wait();
    const uint32_t prefix1 = (uint32_t)__ldcg(meta + kMetaSelPrefix);
    const int want1 = __ldcg(meta + kMetaSelWant), below1 = __ldcg(meta + kMetaSelBelow);
    const int nc = __ldcg(meta + kMetaSelCount);
    int b[1] = {__ldcg(hist2 + tid)};
    find_digit<1>(b, want1, prefix1, 10, below1, S);
    const uint32_t prefix2 = S.prefix;
    const int want2 = S.want, below2 = S.below;
    for (int i0 = 0; i0 < nc; i0 += 1024 * 4) {
        uint32_t kv[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int i = i0 + j * 1024 + tid;
            kv[j] = i < nc ? __ldcg(cand + i) : 0xffffffffu;
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            if (kv[j] != 0xffffffffu && (kv[j] & 0xFFFFFC00u) == prefix2) {
                const int bin = (int)(kv[j] & 1023u);
                const unsigned peers = __match_any_sync(__activemask(), bin);
                if (lane == __ffs(peers) - 1) atomicAdd(&h3[bin], __popc(peers));
            }
        }
    }
    __syncthreads();
    int b3[1] = {h3[tid]};
    find_digit<1>(b3, want2, prefix2, 0, below2, S);
    // ready for the next call
#pragma unroll
    for (int j = 0; j < 4; ++j) hist1[4 * tid + j] = 0;
    hist2[tid] = 0;
    if (tid == 0) {
        meta[kMetaSelCount] = 0;
        const int lo = S.below, hi = S.below + S.last;
        float tau = __uint_as_float(S.prefix);
        if (!(lo == m || (m - lo) <= (hi - m))) tau = __uint_as_float(S.prefix + 1u);
        *tau_out = tau;
    }
}

// Compaction (Algorithm 1 "evaluate only the experts indexed by I"): retained
// slots grouped by expert, tokens increasing inside a group.
// Pass A (k_compact_count): per-chunk per-expert counts, stored expert-major
//   (counts[e * n_chunks + c]).
// Pass B (k_compact_scan, a block per expert): exclusive scan of expert e's
//   row, so counts[e][c] becomes the first row of chunk c's expert-e slots
//   within the expert's group; the last block to finish (atomic ticket) scans
//   the row totals into offsets[N+1], the distinct-expert list and the
//   token-tile table.
// Pass C (k_compact_place): each chunk places its slots at offsets[e] +
//   counts[e][c] + rank, the rank within (chunk, expert) from a per-expert
//   token bitmap, so the order is deterministic.
// With DECIDE (ratio mode) pass A first takes each token's decision from the
// stored g, c and the device tau (decide_token).
template <bool DECIDE>
__global__ void __launch_bounds__(kChunk) k_compact_count(int n_tokens, int k, int n_exp, int n_chunks,
                                                          const int32_t* __restrict__ ids,
                                                          uint8_t* __restrict__ skip,
                                                          const float* __restrict__ gates,
                                                          const float* __restrict__ cval,
                                                          const float* __restrict__ tau_dev, int m_min, float eps,
                                                          float* __restrict__ ghat,
                                                          int32_t* __restrict__ chunk_counts, int* err) {
    __shared__ int cnt[kMaxExperts];
    for (int e = threadIdx.x; e < n_exp; e += blockDim.x) cnt[e] = 0;
    __syncthreads();
    pdl_wait();
    const int t = blockIdx.x * kChunk + threadIdx.x;
    if (t < n_tokens) {
        const size_t base = (size_t)t * k;
        if (DECIDE)
            decide_token(gates + base, cval + base, k, __ldcg(tau_dev), m_min, eps, skip + base, ghat + base, nullptr);
        for (int i = 0; i < k; ++i) {
            const int e = ids[base + i];
            if (!skip[base + i] && ACE_IDX_OK((unsigned)e < (unsigned)n_exp, err)) atomicAdd(&cnt[e], 1);
        }
    }
    __syncthreads();
    for (int e = threadIdx.x; e < n_exp; e += blockDim.x)
        chunk_counts[(size_t)e * n_chunks + blockIdx.x] = cnt[e];
}

constexpr int kScanThreads = 256;   // k_compact_scan block: 4 counts per thread per round

// Exclusive prefix of v over the block (thread order, blockDim.x a multiple
// of 32); total = the block's sum. wtot: 32 ints of shared memory.
__device__ __forceinline__ int block_exscan(int v, int* wtot, int& total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += y;
    }
    if (lane == 31) wtot[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        int wi = lane < nw ? wtot[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += y;
        }
        wtot[lane] = wi;
    }
    __syncthreads();
    const int exc = inc - v + (warp ? wtot[warp - 1] : 0);
    total = wtot[nw - 1];
    __syncthreads();
    return exc;
}

// Block e: exclusive scan of counts[e][0 .. n_chunks) in place, row total to
// offsets[e]. The last block (ticket in meta) turns the totals into
// offsets[N+1], the distinct-expert list, the meta totals and the token-tile
// table, and re-zeroes the ticket.
__global__ void __launch_bounds__(kScanThreads) k_compact_scan(int n_exp, int n_chunks, int32_t* __restrict__ counts,
                                                               int32_t* __restrict__ offsets,
                                                               int32_t* __restrict__ dlist,
                                                               int32_t* __restrict__ meta, int tok_tile,
                                                               int32_t* __restrict__ tt_off, int4* __restrict__ tt_tab,
                                                               int tt_cap, int* err) {
    __shared__ int wtot[32];
    __shared__ int wsum[96];
    __shared__ int cnt[kMaxExperts];
    __shared__ int s_last;
    pdl_wait();
    const int tid = threadIdx.x;
    int32_t* row = counts + (size_t)blockIdx.x * n_chunks;
    int carry = 0;
    for (int c0 = 0; c0 < n_chunks; c0 += 4 * kScanThreads) {
        int v[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int c = c0 + 4 * tid + j;
            v[j] = c < n_chunks ? __ldcg(row + c) : 0;
        }
        int total;
        int run = carry + block_exscan(v[0] + v[1] + v[2] + v[3], wtot, total);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int c = c0 + 4 * tid + j;
            if (c < n_chunks) row[c] = run;
            run += v[j];
        }
        carry += total;
    }
    if (tid == 0) offsets[blockIdx.x] = carry;
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = atomicAdd(&meta[kMetaTicket], 1) == (int)gridDim.x - 1;
    __syncthreads();
    if (!s_last) return;
    if (tid == 0) meta[kMetaTicket] = 0;
    __threadfence();
    for (int e = tid; e < n_exp; e += blockDim.x) cnt[e] = __ldcg(offsets + e);
    __syncthreads();
    scan_counts_block(cnt, n_exp, offsets, dlist, meta, nullptr, tok_tile, tt_off, wsum);
    __syncthreads();
    fill_tile_table(offsets, dlist, tt_off, meta, tok_tile, tt_tab, n_exp, tt_cap, err);
}

__global__ void __launch_bounds__(kChunk) k_compact_place(int n_tokens, int k, int n_exp, int n_chunks,
                                                          const int32_t* __restrict__ ids,
                                                          const uint8_t* __restrict__ skip,
                                                          const int32_t* __restrict__ offsets,
                                                          const int32_t* __restrict__ chunk_base,
                                                          int32_t* __restrict__ perm,
                                                          int32_t* __restrict__ slot_pos, int* err) {
    constexpr int W = kChunk / 32;
    __shared__ uint32_t bm[kMaxExperts * W];
    for (int i = threadIdx.x; i < n_exp * W; i += blockDim.x) bm[i] = 0u;
    __syncthreads();
    pdl_wait();
    const int t = blockIdx.x * kChunk + threadIdx.x;
    const int w = threadIdx.x >> 5;
    const unsigned bit = 1u << (threadIdx.x & 31);
    if (t < n_tokens) {
        for (int i = 0; i < k; ++i) {
            const int e = ids[(size_t)t * k + i];
            if (!skip[(size_t)t * k + i] && ACE_IDX_OK((unsigned)e < (unsigned)n_exp, err)) atomicOr(&bm[e * W + w], bit);
        }
    }
    __syncthreads();
    if (t < n_tokens) {
        const unsigned lt = lanemask_lt();
        for (int i = 0; i < k; ++i) {
            const size_t s = (size_t)t * k + i;
            if (skip[s]) { slot_pos[s] = -1; continue; }
            const int e = ids[s];
            if (!ACE_IDX_OK((unsigned)e < (unsigned)n_exp, err)) { slot_pos[s] = -1; continue; }
            int rank = __popc(bm[e * W + w] & lt);
            for (int ww = 0; ww < w; ++ww) rank += __popc(bm[e * W + ww]);
            const int r = __ldcg(offsets + e) + __ldcg(chunk_base + (size_t)e * n_chunks + blockIdx.x) + rank;
            if (!ACE_IDX_OK(r >= 0 && (size_t)r < (size_t)n_tokens * k, err)) { slot_pos[s] = -1; continue; }
            perm[r] = (int32_t)s;
            slot_pos[s] = r;
        }
    }
}

// --------------------------------------------------------------------------
// Small-T fused kernel (T <= kSmallT): RMSNorm + router logits + top-k +
// decision + threshold + compaction in one launch.
//   phase A (every block, LOGITS only): block (bx, by) normalises tokens
//     [8 bx, 8 bx + 8) into fp32 shared memory (blocks with by == 0 also
//     store h for the experts) and computes their logits for experts
//     [8 by, 8 by + 8), one expert row per warp;
//   phase B (last block of each token tile, by an atomic ticket): top-k,
//     gates and c for the tile's tokens (and the decision in threshold mode);
//   phase C (the globally last block): the App. B.1 threshold in ratio mode
//     (by counting ranks up to kRankSelectMax slots, else a radix select),
//     the decision, and the compaction of retained slots.
// With one token tile (T <= 8) phases B and C run in the same block, which
// passes phase B's results to phase C in shared memory. Tickets are reset by
// the block that consumed them. No block waits on another. The kernel lets
// its dependent launch at entry; that kernel reads nothing of this one before
// its own griddepcontrol.wait.
// --------------------------------------------------------------------------
constexpr int kFuseTok = 8;
constexpr int kFuseWarps = 8;
constexpr int kRowPad = 16;    // bytes appended to each row staged by phase A
constexpr int kRankSelectMax = 128;   // slots up to which phase C counts ranks instead of a radix select
static_assert(kFuseTok == 8 && kFuseWarps == 8, "phase A's MMA takes 8 token rows x 8 router rows");
constexpr long long kRoutePrefetchBytes = 48LL << 20;   // decode: leading W_gu bytes pulled towards L2 while routing

struct FusedArgs {
    const void* x;
    const void* gamma;
    void* h_out;
    const void* w_r;
    const float* b_r;
    float inv_temp;
    int use_temp;
    float rms_eps;
    int d;
    float* logits;
    int n_tokens, n_exp, k;
    const float* a_gsp;
    const float* a_rcr;
    float eps;
    int m_min, mode, fusion;
    float tau_in;
    int m_q;
    int32_t* ids;
    float* gates;
    float* cval;
    uint32_t* keys;
    uint8_t* skip;
    float* ghat;
    float* tau_out;
    int32_t* offsets;
    int32_t* dlist;
    int32_t* perm;
    int32_t* slot_pos;
    int32_t* meta;
    int* err;
    int tok_tile;
    int32_t* tt_off;
    int4* tt_tab;
    int tt_cap;                 // entries allocated in tt_tab
    int32_t* tile_cnt;
    const uint8_t* pf_base;     // expert weights to start pulling into L2 while routing runs
    long long pf_bytes;         // (a multiple of 256 bytes; 0 = none)
    int* dec_done;              // the decode expert kernel's per-token-tile counters, zeroed here (or nullptr)
};

__host__ __device__ inline size_t fused_phase_c_bytes(int T, int k, int n_exp) {
    const size_t ns = (size_t)T * k;
    return 16 + ns * 16 + (size_t)n_exp * 4 + (size_t)(n_exp + 1) * 4 + (size_t)n_exp * 32 + ns + 16;
}

template <typename T, int NPL, bool LOGITS>
__global__ void __launch_bounds__(kFuseWarps * 32) k_route_fused(const __grid_constant__ FusedArgs a) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ SelectSmem<kFuseWarps> S;
    __shared__ int s_last;
    __shared__ float s_tab[LOGITS ? 2 * kMaxExperts : 1];   // the layer's GSP / RCR tables (phase B)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int t0 = blockIdx.x * kFuseTok;
    const int nt = min(kFuseTok, a.n_tokens - t0);
    const int n_exp = a.n_exp, k = a.k;
    // the expert kernel may launch now: its prologue (TMEM, barriers) overlaps the
    // routing, and it reads nothing of ours before its griddepcontrol.wait
    pdl_trigger();
    // one token tile: phases B and C run in the same block, which hands phase B's
    // results to phase C in shared memory (no fence, ticket or reload)
    const bool solo = gridDim.x == 1;
    const float* tab_gsp = a.a_gsp;
    const float* tab_rcr = a.a_rcr;
    if (LOGITS) {
        // A layer's tables were written when it was created: every block copies them
        // into shared memory before the dependency wait, so that phase B (whichever
        // block runs it) reads its experts' entries without a dependent global load.
        for (int i = threadIdx.x; i < n_exp; i += blockDim.x) {
            s_tab[i] = __ldg(a.a_gsp + i);
            s_tab[kMaxExperts + i] = __ldg(a.a_rcr + i);
        }
        tab_gsp = s_tab;
        tab_rcr = s_tab + kMaxExperts;
    } else if (blockIdx.y == 0) {
        // caller-owned tables (read after the wait): pull their lines towards L2
        const int lines = (n_exp + 31) / 32;
        if ((int)threadIdx.x < 2 * lines) {
            const float* tab = (int)threadIdx.x < lines ? a.a_gsp : a.a_rcr;
            const int l = (int)threadIdx.x % lines;
            asm volatile("prefetch.global.L2 [%0];" ::"l"(tab + min(l * 32, n_exp - 1)) : "memory");
        }
    }
    if (LOGITS) {
        // ---------------- phase A: RMSNorm + logits for 8 tokens x 8 experts.
        // Warp 0 bulk-copies gamma and the block's 8 router rows (layer
        // constants, before the dependency wait) and the tile's x rows into
        // shared memory, one row per lane, so the block waits for one round
        // trip; the rows are then normalised in place and the dot products
        // read shared memory. Staged rows are kRowPad bytes longer than a row,
        // which spreads the 8 rows of an MMA operand load over all 32 banks.
        const int d = a.d;
        constexpr int V = Vec16<T>::N;
        const int nvec = d / V;
        const uint32_t row_bytes = (uint32_t)(d * sizeof(T));
        const uint32_t rs = row_bytes + kRowPad;                  // staged row stride
        uint64_t* bar = reinterpret_cast<uint64_t*>(smem_raw);
        unsigned char* xs = smem_raw + 16;                        // [kFuseTok] rows -> h in place
        unsigned char* gs = xs + (size_t)kFuseTok * rs;           // gamma
        unsigned char* wsm = gs + rs;                             // [kFuseWarps] router rows
        float* red = reinterpret_cast<float*>(wsm + (size_t)kFuseWarps * rs);   // [warps][8][8] partial logits
        const int e0 = blockIdx.y * kFuseWarps;
        const int ne = min(kFuseWarps, n_exp - e0);
        const bool mma_path = sizeof(T) == 2 && d % (16 * kFuseWarps) == 0;
        // the router bias of this thread's output column (MMA path: column tid & 7 of
        // the 8 x 8 block; FMA path: the warp's expert), read before the dependency wait
        const int bj = mma_path ? (int)(threadIdx.x & 7) : warp;
        const float bias = bj < ne ? __ldg(a.b_r + e0 + bj) : 0.f;
        if (threadIdx.x == 0) {
            mbar_init(bar, 1);
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        }
        __syncthreads();
        if (warp == 0) {
            if (lane == 0) {
                mbar_expect_tx(bar, (uint32_t)(nt + 1 + ne) * row_bytes);
                bulk_g2s(gs, a.gamma, row_bytes, bar);
            }
            __syncwarp();
            if (lane < ne) bulk_g2s(wsm + (size_t)lane * rs, static_cast<const T*>(a.w_r) + (size_t)(e0 + lane) * d,
                                    row_bytes, bar);
            pdl_wait();                                           // x is the predecessor's output
            if (lane < nt) bulk_g2s(xs + (size_t)lane * rs, static_cast<const T*>(a.x) + (size_t)(t0 + lane) * d,
                                    row_bytes, bar);
        } else {
            pdl_wait();
        }
        if (!mbar_wait(bar, 0, a.err)) return;
        const uint4* gv = reinterpret_cast<const uint4*>(gs);
        if (warp < nt) {
            // h = x / sqrt(mean(x^2) + eps) * gamma, rounded to T (the stored h feeds the router)
            uint4* xr = reinterpret_cast<uint4*>(xs + (size_t)warp * rs);
            float ss = 0.f;                                   // chunk partials, as rmsnorm_row
#pragma unroll 1
            for (int c = lane; c < nvec; c += 32) {
                float f[V];
                Vec16<T>::to_float(xr[c], f);
                float part = 0.f;
#pragma unroll
                for (int j = 0; j < V; ++j) part = fmaf(f[j], f[j], part);
                ss += part;
            }
            ss = warp_sum(ss);
            const float inv = 1.0f / sqrtf(ss / (float)d + a.rms_eps);
            uint4* hg = blockIdx.y == 0 ? reinterpret_cast<uint4*>(static_cast<T*>(a.h_out) + (size_t)(t0 + warp) * d)
                                        : nullptr;
#pragma unroll 1
            for (int c = lane; c < nvec; c += 32) {
                float f[V], gm[V];
                Vec16<T>::to_float(xr[c], f);
                Vec16<T>::to_float(gv[c], gm);
                T o[V];
#pragma unroll
                for (int j = 0; j < V; ++j) o[j] = from_f32<T>(f[j] * inv * gm[j]);
                const uint4 ov = *reinterpret_cast<const uint4*>(o);
                xr[c] = ov;
                if (hg) hg[c] = ov;
            }
        }
        __syncthreads();
        if (threadIdx.x == 0) mbar_inval(bar);
        if (mma_path) {
            // bf16: warp w takes K slice w and runs mma.sync m16n8k16 over it
            // (A = the 8 token rows, zero-padded to 16; B = the 8 router rows;
            // products exact, fp32 accumulation); the 8 partial 8 x 8 blocks
            // are summed in warp order
            const int g = lane >> 2, tq = lane & 3;
            const int kslice = d / kFuseWarps;
            const unsigned char* xrow = xs + (size_t)g * rs;
            const unsigned char* wrow = wsm + (size_t)g * rs;
            float c0 = 0.f, c1 = 0.f, c2 = 0.f, c3 = 0.f;
#pragma unroll 4
            for (int ks = 0; ks < kslice; ks += 16) {
                const int kb = (warp * kslice + ks + 2 * tq) * 2;     // byte offset in the row
                const uint32_t a0 = *reinterpret_cast<const uint32_t*>(xrow + kb);
                const uint32_t a2 = *reinterpret_cast<const uint32_t*>(xrow + kb + 16);
                const uint32_t b0 = *reinterpret_cast<const uint32_t*>(wrow + kb);
                const uint32_t b1 = *reinterpret_cast<const uint32_t*>(wrow + kb + 16);
                asm volatile(
                    "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                    "{%0,%1,%2,%3};"
                    : "+f"(c0), "+f"(c1), "+f"(c2), "+f"(c3)
                    : "r"(a0), "r"(0u), "r"(a2), "r"(0u), "r"(b0), "r"(b1));
            }
            // c0, c1: token g, experts 2 tq and 2 tq + 1 (rows 8..15 are padding)
            red[(warp * 8 + g) * 8 + 2 * tq] = c0;
            red[(warp * 8 + g) * 8 + 2 * tq + 1] = c1;
            __syncthreads();
            if (threadIdx.x < 64) {
                const int r = threadIdx.x >> 3, j = threadIdx.x & 7;
                float v = 0.f;
#pragma unroll
                for (int w = 0; w < kFuseWarps; ++w) v += red[(w * 8 + r) * 8 + j];
                if (r < nt && j < ne) {
                    v = v + bias;
                    if (a.use_temp) v = v * a.inv_temp;
                    a.logits[(size_t)(t0 + r) * n_exp + e0 + j] = v;
                }
            }
        } else if (warp < ne) {
            const int e = e0 + warp;
            const uint4* wr = reinterpret_cast<const uint4*>(wsm + (size_t)warp * rs);
            float acc[kFuseTok];
#pragma unroll
            for (int r = 0; r < kFuseTok; ++r) acc[r] = 0.f;
#pragma unroll 1
            for (int c = lane; c < nvec; c += 32) {
                float wf[V];
                Vec16<T>::to_float(wr[c], wf);
#pragma unroll
                for (int r = 0; r < kFuseTok; ++r) {
                    float hf[V];
                    Vec16<T>::to_float(reinterpret_cast<const uint4*>(xs + (size_t)r * rs)[c], hf);
#pragma unroll
                    for (int j = 0; j < V; ++j) acc[r] = fmaf(hf[j], wf[j], acc[r]);
                }
            }
#pragma unroll
            for (int r = 0; r < kFuseTok; ++r) acc[r] = warp_sum(acc[r]);
            if (lane < nt) {
                float v = acc[0];
#pragma unroll
                for (int r = 1; r < kFuseTok; ++r) if (lane == r) v = acc[r];
                v = v + bias;
                if (a.use_temp) v = v * a.inv_temp;
                a.logits[(size_t)(t0 + lane) * n_exp + e] = v;
            }
        }
        __threadfence();
        __syncthreads();
        if (threadIdx.x == 0) {
            s_last = atomicAdd(&a.tile_cnt[blockIdx.x], 1) == (int)gridDim.y - 1;
            if (s_last) a.tile_cnt[blockIdx.x] = 0;
        }
        __syncthreads();
        if (!s_last) {
            if (a.pf_bytes > 0) {
                // HBM idles while the rest of the routing runs: the blocks
                // that leave here pull the leading expert-weight tiles towards
                // L2 (per-thread line prefetches: a bulk prefetch occupies the
                // SM's copy engine), off the path of the blocks that go on
                // (the lines of the continuing blocks' shares are left out)
                const long long units = a.pf_bytes >> 8;
                const long long nthr = (long long)gridDim.x * gridDim.y * blockDim.x;
                const long long b = (long long)blockIdx.y * gridDim.x + blockIdx.x;
                for (long long u = b * blockDim.x + threadIdx.x; u < units; u += nthr)
                    asm volatile("prefetch.global.L2::evict_last [%0];" ::"l"(a.pf_base + (u << 8)) : "memory");
            }
            return;
        }
        __threadfence();
    } else {
        pdl_wait();                                               // logits are the predecessor's output
    }
    // phase C's shared arrays (over phase A's staging rows, which no warp reads past the
    // ticket's barrier)
    const int n_tokens = a.n_tokens;
    const int ns = n_tokens * k;
    float* g_s = reinterpret_cast<float*>(smem_raw + 16);
    float* c_s = g_s + ns;
    uint32_t* key_s = reinterpret_cast<uint32_t*>(c_s + ns);
    int* id_s = reinterpret_cast<int*>(key_s + ns);
    int* cnt = id_s + ns;                                            // [n_exp]
    int* off_s = cnt + n_exp;                                        // [n_exp + 1]
    uint32_t* bm = reinterpret_cast<uint32_t*>(off_s + n_exp + 1);   // [n_exp * 8]
    uint8_t* skip_s = reinterpret_cast<uint8_t*>(bm + n_exp * 8);    // [ns]
    // ---------------- phase B: top-k, gates, c for this token tile
    const bool ratio = a.mode == ACE_SKIP_RATIO;
    for (int r = warp; r < nt; r += kFuseWarps) {
        const int t = t0 + r;
        int id;
        float zv;
        bool nan;
        warp_topk<NPL>(a.logits + (size_t)t * n_exp, n_exp, k, lane, id, zv, nan);
        if (lane < k && !ACE_IDX_OK((unsigned)id < (unsigned)n_exp, a.err)) id = 0;
        const float z0 = __shfl_sync(0xffffffffu, zv, 0);
        if (__any_sync(0xffffffffu, nan) && lane == 0) atomicOr(a.err, kErrNumeric);
        const SlotScore sc = score_slot(lane, k, zv, z0, lane < k ? id : 0, tab_gsp, tab_rcr, a.eps, a.fusion);
        const size_t base = (size_t)t * k;
        if (lane < k) {
            a.ids[base + lane] = id;
            a.gates[base + lane] = sc.g;
            a.cval[base + lane] = sc.c;
            if (solo) {
                id_s[base + lane] = id;
                g_s[base + lane] = sc.g;
                c_s[base + lane] = sc.c;
            }
        }
        if (!ratio) {
            bool sk;
            float gh;
            decide_slot(lane, k, sc.g, sc.c, a.tau_in, a.m_min, a.eps, sk, gh);
            if (lane < k) {
                a.skip[base + lane] = sk ? 1 : 0;
                a.ghat[base + lane] = gh;
                if (solo) skip_s[base + lane] = sk ? 1 : 0;
            }
        } else {
            const bool prot = slot_protected(lane, k, sc.c, a.m_min);
            const uint32_t key = prot ? 0xffffffffu : __float_as_uint(sc.c);
            if (lane < k) {
                a.keys[base + lane] = key;
                if (solo) key_s[base + lane] = key;
            }
        }
    }
    if (!solo) {
        __threadfence();
        __syncthreads();
        if (threadIdx.x == 0) {
            s_last = atomicAdd(&a.meta[kMetaTicket2], 1) == (int)gridDim.x - 1;
            if (s_last) a.meta[kMetaTicket2] = 0;
        }
        __syncthreads();
        if (!s_last) return;
        __threadfence();
    }
    // ---------------- phase C: threshold, decision, compaction (all tokens)
    for (int i = threadIdx.x; i < n_exp; i += blockDim.x) cnt[i] = 0;
    for (int i = threadIdx.x; i < n_exp * 8; i += blockDim.x) bm[i] = 0u;
    if (!solo) {
        for (int i = threadIdx.x; i < ns; i += blockDim.x) {
            id_s[i] = __ldcg(a.ids + i);
            if (ratio) {
                g_s[i] = __ldcg(a.gates + i);
                c_s[i] = __ldcg(a.cval + i);
                key_s[i] = __ldcg(a.keys + i);
            } else {
                skip_s[i] = __ldcg(a.skip + i);
            }
        }
    }
    if (threadIdx.x == 0) {
        S.prefix = 0u;
        S.below = 0;
        S.last_cnt = 0;
    }
    __syncthreads();
    if (ratio) {
        const float tau = ns <= kRankSelectMax ? block_select_tau_rank(key_s, ns, a.m_q, S)
                                               : block_select_tau(key_s, ns, a.m_q, S);
        if (threadIdx.x == 0) *a.tau_out = tau;
        for (int t = threadIdx.x; t < n_tokens; t += blockDim.x) {
            const int base = t * k;
            decide_token(g_s + base, c_s + base, k, tau, a.m_min, a.eps, a.skip + base, a.ghat + base,
                         skip_s + base);
        }
        __syncthreads();
    } else if (threadIdx.x == 0) {
        *a.tau_out = a.tau_in;
    }
    for (int s = threadIdx.x; s < ns; s += blockDim.x) {
        if (skip_s[s]) continue;
        const int e = id_s[s], t = s / k;
        if (!ACE_IDX_OK((unsigned)e < (unsigned)n_exp && (t >> 5) < 8, a.err)) continue;
        atomicAdd(&cnt[e], 1);
        atomicOr(&bm[e * 8 + (t >> 5)], 1u << (t & 31));
    }
    __syncthreads();
    scan_counts_block(cnt, n_exp, a.offsets, a.dlist, a.meta, off_s, a.tok_tile, a.tt_off, S.hist);
    __syncthreads();
    if (a.dec_done) {                     // the decode expert kernel counts up from zero
        for (int i = threadIdx.x; i < a.meta[kMetaTokTiles]; i += blockDim.x) a.dec_done[i] = 0;
        if (threadIdx.x == 0) a.meta[kMetaDecNext] = 0;
    }
    fill_tile_table(a.offsets, a.dlist, a.tt_off, a.meta, a.tok_tile, a.tt_tab, n_exp, a.tt_cap, a.err);
    for (int s = threadIdx.x; s < ns; s += blockDim.x) {
        if (skip_s[s]) { a.slot_pos[s] = -1; continue; }
        const int e = id_s[s], t = s / k, w = t >> 5;
        if (!ACE_IDX_OK((unsigned)e < (unsigned)n_exp && w < 8, a.err)) { a.slot_pos[s] = -1; continue; }
        int rank = __popc(bm[e * 8 + w] & ((1u << (t & 31)) - 1u));
        for (int ww = 0; ww < w; ++ww) rank += __popc(bm[e * 8 + ww]);
        const int r = off_s[e] + rank;
        if (!ACE_IDX_OK(r >= 0 && r < ns, a.err)) { a.slot_pos[s] = -1; continue; }
        a.perm[r] = s;
        a.slot_pos[s] = r;
    }
}

size_t fused_smem_bytes(const ace_layer* L, int T) {
    const size_t a = 16 + (size_t)(kFuseTok + 1 + kFuseWarps) * (L->desc.hidden * L->elem + kRowPad) +
                     (size_t)kFuseWarps * 64 * sizeof(float);
    const size_t c = fused_phase_c_bytes(T, L->desc.top_k, L->desc.n_experts);
    return a > c ? a : c;
}

__global__ void k_debug_exp(const float* __restrict__ x, float* __restrict__ y, int n) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) y[i] = ace_exp32(x[i]);
}

inline int cdiv(long long a, long long b) { return (int)((a + b - 1) / b); }

size_t router_smem(const ace_layer* L) { return (size_t)kRouterTok * L->desc.hidden * L->elem; }

template <typename T, bool FUSE>
cudaError_t router_launch(const ace_layer* L, const void* src, int T_, cudaStream_t s) {
    const int d = L->desc.hidden, n = L->desc.n_experts;
    const float temp = L->desc.router_temp;
    const dim3 blocks(cdiv(T_, kRouterTok), cdiv(n, kRouterExp));
    k_router<T, FUSE><<<blocks, 256, router_smem(L), s>>>((const T*)src, (const T*)L->gamma, (T*)L->ws.h,
                                                          (const T*)L->router_w, L->router_b, L->ws.logits, T_, d,
                                                          n, 1.0f / temp, temp != 1.0f, L->desc.rms_eps);
    return cudaGetLastError();
}

template <typename T>
cudaError_t set_router_attrs(size_t smem) {
    cudaError_t e = raise_smem_limit(k_router<T, true>, (int)smem);
    if (e != cudaSuccess) return e;
    return raise_smem_limit(k_router<T, false>, (int)smem);
}

int select_mq(const ace_layer* L, int T, ace_skip_ctl ctl, float* tau, bool* need_select) {
    const int k = L->desc.top_k;
    *tau = ctl.value;
    *need_select = false;
    if (ctl.mode != ACE_SKIP_RATIO) return 0;
    const long long n_all = (long long)T * k;
    const int prot = L->desc.min_active < 1 ? 1 : (L->desc.min_active > k ? k : L->desc.min_active);
    const long long n_cand = (long long)T * (k - prot);
    long long mq = llround((double)ctl.value * (double)n_all);
    if (mq < 0) mq = 0;
    if (mq > n_cand) mq = n_cand;
    if (mq == 0) *tau = 0.0f;
    else if (mq == n_cand) *tau = INFINITY;
    else *need_select = true;
    return (int)mq;
}

}  // namespace

bool small_path(int T) { return T <= kSmallT; }

namespace {
template <typename T, int NPL, bool LOGITS>
cudaError_t fused_launch(const ace_layer* L, const FusedArgs& a, int n_tok, cudaStream_t s) {
    const dim3 grid(cdiv(n_tok, kFuseTok), LOGITS ? cdiv(L->desc.n_experts, kFuseWarps) : 1);
    return launch_pdl(k_route_fused<T, NPL, LOGITS>, grid, dim3(kFuseWarps * 32), fused_smem_bytes(L, kSmallT), s, a);
}

template <typename T, bool LOGITS>
cudaError_t fused_dispatch(const ace_layer* L, const FusedArgs& a, int n_tok, cudaStream_t s) {
    const int n = L->desc.n_experts;
    if (n <= 128) return fused_launch<T, 4, LOGITS>(L, a, n_tok, s);
    if (n <= 256) return fused_launch<T, 8, LOGITS>(L, a, n_tok, s);
    return fused_launch<T, 32, LOGITS>(L, a, n_tok, s);
}

template <typename T, int NPL, bool LOGITS>
cudaError_t fused_attr(int smem) {
    return raise_smem_limit(k_route_fused<T, NPL, LOGITS>, smem);
}

template <typename T>
cudaError_t fused_attrs(int smem) {
    cudaError_t e;
    if ((e = fused_attr<T, 4, true>(smem)) != cudaSuccess) return e;
    if ((e = fused_attr<T, 8, true>(smem)) != cudaSuccess) return e;
    if ((e = fused_attr<T, 32, true>(smem)) != cudaSuccess) return e;
    if ((e = fused_attr<T, 4, false>(smem)) != cudaSuccess) return e;
    if ((e = fused_attr<T, 8, false>(smem)) != cudaSuccess) return e;
    return fused_attr<T, 32, false>(smem);
}
}  // namespace

// T <= kSmallT: the whole routing in one launch. x == nullptr: logits are given.
cudaError_t launch_route_fused(const ace_layer* L, const void* x, const float* logits, int T, ace_skip_ctl ctl,
                               cudaStream_t s) {
    const ace_layer_desc& D = L->desc;
    const Workspace& W = L->ws;
    FusedArgs a{};
    float tau;
    bool need_select;
    a.m_q = select_mq(L, T, ctl, &tau, &need_select);
    a.mode = need_select ? ACE_SKIP_RATIO : ACE_SKIP_THRESHOLD;
    a.fusion = ctl.fusion;
    a.tau_in = tau;
    a.x = x;
    a.gamma = L->gamma;
    a.h_out = W.h;
    a.w_r = L->router_w;
    a.b_r = L->router_b;
    a.inv_temp = 1.0f / D.router_temp;
    a.use_temp = D.router_temp != 1.0f;
    a.rms_eps = D.rms_eps;
    a.d = D.hidden;
    a.logits = const_cast<float*>(logits);
    a.n_tokens = T;
    a.n_exp = D.n_experts;
    a.k = D.top_k;
    a.a_gsp = L->a_gsp;
    a.a_rcr = L->a_rcr;
    a.eps = D.eps;
    a.m_min = D.min_active;
    a.ids = W.ids;
    a.gates = W.gates;
    a.cval = W.cval;
    a.keys = W.keys;
    a.skip = W.skip;
    a.ghat = W.ghat;
    a.tau_out = W.tau;
    a.offsets = W.offsets;
    a.dlist = W.dlist;
    a.perm = W.perm;
    a.slot_pos = W.slot_pos;
    a.meta = W.meta;
    a.err = W.err;
    a.tok_tile = L->tc ? tc_token_tile(L, T, ctl) : 0;
    a.tt_off = W.tt_off;
    a.tt_tab = W.tt_tab;
    a.tt_cap = L->tt_cap;
    a.tile_cnt = W.tile_cnt;
    if (x && L->tc) a.dec_done = W.dec_done;
    if (x && L->tc && L->w_gu) {
        const long long gu_bytes = 2LL * D.ffn * D.hidden * 2 * D.n_experts;
        const long long want = kRoutePrefetchBytes;
        a.pf_base = static_cast<const uint8_t*>(L->w_gu);
        a.pf_bytes = (want < gu_bytes ? want : gu_bytes) & ~255LL;
    }
    const bool bf = D.dtype == ACE_BF16;
    if (x) return bf ? fused_dispatch<__nv_bfloat16, true>(L, a, T, s) : fused_dispatch<float, true>(L, a, T, s);
    return bf ? fused_dispatch<__nv_bfloat16, false>(L, a, T, s) : fused_dispatch<float, false>(L, a, T, s);
}

template <typename E>
cudaError_t launch_rmsnorm_t(const ace_layer* L, const void* x, int T, cudaStream_t s) {
    const int d = L->desc.hidden;
    const int blocks = cdiv(T, 8);
    const int nv = cdiv(d / Vec16<E>::N, 32);      // vectors per lane (<= kNormVec, checked at create)
    const E* xt = static_cast<const E*>(x);
    const E* g = static_cast<const E*>(L->gamma);
    E* h = static_cast<E*>(L->ws.h);
    const float eps = L->desc.rms_eps;
    const size_t sm = (size_t)8 * d * sizeof(E);      // one staged row per warp
    if (nv <= 4) return launch_pdl(k_rmsnorm<E, 4>, dim3(blocks), dim3(256), sm, s, xt, g, h, T, d, eps);
    if (nv <= 8) return launch_pdl(k_rmsnorm<E, 8>, dim3(blocks), dim3(256), sm, s, xt, g, h, T, d, eps);
    return launch_pdl(k_rmsnorm<E, kNormVec>, dim3(blocks), dim3(256), sm, s, xt, g, h, T, d, eps);
}

cudaError_t launch_rmsnorm(const ace_layer* L, const void* x, int T, cudaStream_t s) {
    return L->desc.dtype == ACE_BF16 ? launch_rmsnorm_t<__nv_bfloat16>(L, x, T, s) : launch_rmsnorm_t<float>(L, x, T, s);
}

cudaError_t launch_router(const ace_layer* L, const void* x, int T, bool fuse_norm, cudaStream_t s) {
    const void* src = fuse_norm ? x : L->ws.h;
    if (L->desc.dtype == ACE_BF16)
        return fuse_norm ? router_launch<__nv_bfloat16, true>(L, src, T, s)
                         : router_launch<__nv_bfloat16, false>(L, src, T, s);
    return fuse_norm ? router_launch<float, true>(L, src, T, s) : router_launch<float, false>(L, src, T, s);
}

cudaError_t launch_route(const ace_layer* L, const float* logits, int T, ace_skip_ctl ctl, cudaStream_t s,
                         int n_split) {
    const ace_layer_desc& D = L->desc;
    const Workspace& W = L->ws;
    const int k = D.top_k, n = D.n_experts;
    float tau;
    bool need_select;
    const int m_q = select_mq(L, T, ctl, &tau, &need_select);
    const int mode = need_select ? ACE_SKIP_RATIO : ACE_SKIP_THRESHOLD;
    const int tok_tile = L->tc ? tc_token_tile(L, T, ctl) : 0;
    if (T <= kSmallT) return launch_route_fused(L, nullptr, logits, T, ctl, s);
    const int blocks = cdiv(T, kTopkWarps);
    cudaError_t e;
#define ACE_TOPK(NPL)                                                                                             \
    launch_pdl(k_topk_score<NPL>, dim3(blocks), dim3(kTopkWarps * 32), 0, s, const_cast<float*>(logits), T, n, k, \
               (const float*)L->a_gsp, (const float*)L->a_rcr, D.eps, D.min_active, mode, tau, W.ids, W.gates,    \
               W.cval, W.keys, W.skip, W.ghat, W.tau, W.err, W.sel_hist, (const float*)W.act_bf16, n_split,        \
               (const float*)L->router_b, 1.0f / D.router_temp, D.router_temp != 1.0f ? 1 : 0, ctl.fusion)
    if (n <= 128) e = ACE_TOPK(4);
    else if (n <= 256) e = ACE_TOPK(8);
    else e = ACE_TOPK(32);
#undef ACE_TOPK
    if (e != cudaSuccess) return e;
    if (mode == ACE_SKIP_RATIO) {
        const int nk = T * k;
        // fewest keys per thread that keep the grid within two 1024-thread blocks per SM
#define ACE_COLLECT(KPT)                                                                                          \
    launch_pdl(k_sel_collect<KPT>, dim3(cdiv(nk, 1024 * KPT)), dim3(1024), 0, s, (const uint32_t*)W.keys, nk, m_q, \
               (const int32_t*)W.sel_hist, W.sel_hist + kHistBins, W.sel_cand, W.meta, W.err)
        const long long slots = 2LL * 1024 * L->num_sms;
        if (nk <= slots) e = ACE_COLLECT(1);
        else if (nk <= 2 * slots) e = ACE_COLLECT(2);
        else if (nk <= 4 * slots) e = ACE_COLLECT(4);
        else e = ACE_COLLECT(8);
#undef ACE_COLLECT
        if (e != cudaSuccess) return e;
        e = launch_pdl(k_sel_final, dim3(1), dim3(1024), 0, s, m_q, W.sel_hist, W.sel_hist + kHistBins,
                       (const uint32_t*)W.sel_cand, W.meta, W.tau);
        if (e != cudaSuccess) return e;
    }
    const int n_chunks = cdiv(T, kChunk);
    const bool dec = mode == ACE_SKIP_RATIO;
    e = launch_pdl(dec ? k_compact_count<true> : k_compact_count<false>, dim3(n_chunks), dim3(kChunk), 0, s, T, k, n,
                   n_chunks, (const int32_t*)W.ids, W.skip, (const float*)W.gates, (const float*)W.cval,
                   (const float*)W.tau, D.min_active, D.eps, W.ghat, W.chunk_counts, W.err);
    if (e != cudaSuccess) return e;
    e = launch_pdl(k_compact_scan, dim3(n), dim3(kScanThreads), 0, s, n, n_chunks, W.chunk_counts, W.offsets, W.dlist,
                   W.meta, tok_tile, W.tt_off, W.tt_tab, L->tt_cap, W.err);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_compact_place, dim3(n_chunks), dim3(kChunk), 0, s, T, k, n, n_chunks, (const int32_t*)W.ids,
                      (const uint8_t*)W.skip, (const int32_t*)W.offsets, (const int32_t*)W.chunk_counts, W.perm,
                      W.slot_pos, W.err);
}

int route_launch_count(const ace_layer* L, int T, ace_skip_ctl ctl) {
    if (T <= kSmallT) return 1;   // fused with the router in the forward
    float tau;
    bool sel;
    select_mq(L, T, ctl, &tau, &sel);
    return sel ? 6 : 4;
}

cudaError_t route_init(const ace_layer* L) {
    cudaError_t e = set_router_attrs<__nv_bfloat16>(router_smem(L));
    if (e != cudaSuccess) return e;
    // k_rmsnorm stages one row per warp: 8 x d x element bytes
    const int rn = 8 * L->desc.hidden * (int)L->elem;
    const void* norms[] = {(const void*)k_rmsnorm<__nv_bfloat16, 4>, (const void*)k_rmsnorm<__nv_bfloat16, 8>,
                           (const void*)k_rmsnorm<__nv_bfloat16, kNormVec>, (const void*)k_rmsnorm<float, 4>,
                           (const void*)k_rmsnorm<float, 8>, (const void*)k_rmsnorm<float, kNormVec>};
    for (const void* kf : norms)
        if ((e = raise_smem_limit(kf, rn)) != cudaSuccess) return e;
    e = set_router_attrs<float>(router_smem(L));
    if (e != cudaSuccess) return e;
    const int sm = (int)fused_smem_bytes(L, kSmallT);
    if ((e = fused_attrs<__nv_bfloat16>(sm)) != cudaSuccess) return e;
    if ((e = fused_attrs<float>(sm)) != cudaSuccess) return e;
    const void* ks[] = {(const void*)k_route_fused<__nv_bfloat16, 4, true>, (const void*)k_route_fused<__nv_bfloat16, 8, true>,
                        (const void*)k_route_fused<__nv_bfloat16, 32, true>, (const void*)k_route_fused<float, 4, true>,
                        (const void*)k_route_fused<float, 8, true>, (const void*)k_route_fused<float, 32, true>,
                        (const void*)k_topk_score<4>, (const void*)k_topk_score<8>,
                        (const void*)k_topk_score<32>, (const void*)k_compact_count<true>,
                        (const void*)k_compact_count<false>, (const void*)k_compact_place,
                        (const void*)k_compact_scan};
    for (const void* kf : ks)
        if ((e = prefer_shared(kf)) != cudaSuccess) return e;
    return cudaSuccess;
}

// Decision-only launch of k_route_fused on scratch the caller owns (no layer).
size_t route_decide_smem(int T, int k, int n_exp) { return fused_phase_c_bytes(T, k, n_exp); }

cudaError_t route_decide_attr(int smem_bytes) {
    cudaError_t e;
    if ((e = raise_smem_limit(k_route_fused<__nv_bfloat16, 4, false>, smem_bytes)) != cudaSuccess) return e;
    if ((e = raise_smem_limit(k_route_fused<__nv_bfloat16, 8, false>, smem_bytes)) != cudaSuccess) return e;
    return raise_smem_limit(k_route_fused<__nv_bfloat16, 32, false>, smem_bytes);
}

cudaError_t launch_route_decide_scratch(const float* logits, int T, int n_exp, int k, const float* a_gsp,
                                        const float* a_rcr, float eps, int m_min, ace_skip_ctl ctl, int32_t* ids,
                                        uint8_t* skip, float* ghat, float* tau_out, const DecideScratch& sc,
                                        cudaStream_t s) {
    FusedArgs a{};
    float tau = ctl.value;
    bool need_select = false;
    int m_q = 0;
    if (ctl.mode == ACE_SKIP_RATIO) {
        const long long n_all = (long long)T * k;
        const int prot = m_min < 1 ? 1 : (m_min > k ? k : m_min);
        const long long n_cand = (long long)T * (k - prot);
        long long mq = llround((double)ctl.value * (double)n_all);
        mq = mq < 0 ? 0 : (mq > n_cand ? n_cand : mq);
        m_q = (int)mq;
        if (mq == 0) tau = 0.0f;
        else if (mq == n_cand) tau = INFINITY;
        else need_select = true;
    }
    a.mode = need_select ? ACE_SKIP_RATIO : ACE_SKIP_THRESHOLD;
    a.fusion = ctl.fusion;
    a.tau_in = tau;
    a.m_q = m_q;
    a.logits = const_cast<float*>(logits);
    a.n_tokens = T;
    a.n_exp = n_exp;
    a.k = k;
    a.a_gsp = a_gsp;
    a.a_rcr = a_rcr;
    a.eps = eps;
    a.m_min = m_min;
    a.ids = ids;
    a.gates = sc.gates;
    a.cval = sc.cval;
    a.keys = sc.keys;
    a.skip = skip;
    a.ghat = ghat;
    a.tau_out = tau_out;
    a.offsets = sc.offsets;
    a.dlist = sc.dlist;
    a.perm = sc.perm;
    a.slot_pos = sc.slot_pos;
    a.meta = sc.meta;
    a.err = sc.err;
    a.tok_tile = 0;
    a.tile_cnt = sc.tile_cnt;
    const size_t smem = route_decide_smem(T, k, n_exp);
    const dim3 grid(cdiv(T, kFuseTok), 1);
    if (n_exp <= 128) k_route_fused<__nv_bfloat16, 4, false><<<grid, kFuseWarps * 32, smem, s>>>(a);
    else if (n_exp <= 256) k_route_fused<__nv_bfloat16, 8, false><<<grid, kFuseWarps * 32, smem, s>>>(a);
    else k_route_fused<__nv_bfloat16, 32, false><<<grid, kFuseWarps * 32, smem, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_debug_exp(const float* x, float* y, int n, cudaStream_t s) {
    k_debug_exp<<<cdiv(n, 256), 256, 0, s>>>(x, y, n);
    return cudaGetLastError();
}

}  // namespace ace

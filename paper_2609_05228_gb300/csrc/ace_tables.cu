// ace_tables.cu — the offline expert tables of ACE on the GPU, from bf16
// weights in device memory.
//
// GSP (Algorithm 2; Eqs. gsp_up_path, gsp_gate_path, gsp_geometric_mean,
// gsp_layer_normalization). With G = Gamma W_gate, U = Gamma W_up (d x m) and
// W_down (m x d):
//   a_up = ||U||_F ||G W_down||_F,   a_gate = ||G||_F ||U W_down||_F,
//   a~_e = sqrt(a_up a_gate),        A^GSP(e) = a~_e / (mean_j a~_j + eps).
// ||Gamma W_p W_down||_F^2 = sum_i gamma_i^2 sum_j (sum_r W_p[i,r] W_down[r,j])^2
// is a d x d x m GEMM per expert and path whose d x d product never leaves
// the SM: k_gsp_frob runs it on the tensor cores (tcgen05.mma, bf16 operands
// exactly as stored, fp32 accumulators in TMEM) and its epilogue squares the
// accumulators, sums them per row, scales row i by gamma_i^2 (so Gamma is
// applied exactly, not rounded into a bf16 operand) and writes one fp64
// partial per (tile, warp). The nn.Linear layouts give W_p[i, r] =
// w_p[e][r][i] (the A operand, transposed into K-major tiles here) and
// W_down[r, j] = w_down[e][j][r] (the B operand, K-major as stored).
//
// RCR (Algorithm 3; Eqs. rcr_centered_router, rcr_direction_prototype,
// rcr_raw_amplification, rcr_layer_normalization): centred router rows
// w~_e = w_e - mean_j w_j, prototype q_e = w~_e / (RMS(w~_e) + eps) (rho = 1),
// a~_e = ||f_e(q_e)||_2 / (||q_e||_2 + eps), A^RCR(e) = a~_e / (mean a~ + eps),
// f_e(x) = (SiLU(x W_gate) * (x W_up)) W_down; q_e is scaled by gamma first
// when rcr_apply_gamma is set. One input row per expert makes this a GEMV
// over all expert weights: fp32 on the CUDA cores, bound by HBM.
//
// Every reduction is summed in a fixed order (per-thread, per-warp, per-tile
// partials combined by one thread per expert), so the tables are the same
// bits on every run.
#include <cuda.h>
#include <math.h>

#include <string>

#include "ace_device.cuh"
#include "ace_internal.h"
#include "ace_tc.cuh"

namespace ace {
namespace {

constexpr int kTabThreads = 192;
constexpr int kTabStages = 4;
constexpr int kTabA = 128 * kBK * 2;            // 16 KB: 128 rows i x 64 r
constexpr int kTabB = 256 * kBK * 2;            // 32 KB: 256 rows j x 64 r
constexpr int kTabStage = kTabA + kTabB;
constexpr int kTabSmem = kTabStages * kTabStage + 1024 + 256;
constexpr int kTile = 16384;                    // bytes of one 128 x 64 bf16 tile

// Fixed-order block sum of one double per thread (blockDim.x = 256).
__device__ __forceinline__ double block_sum_256(double v, double* sh) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = v;
    __syncthreads();
    double t = 0.0;
    if (threadIdx.x == 0)
        for (int w = 0; w < 8; ++w) t += sh[w];
    __syncthreads();
    return t;   // valid in thread 0
}

// ---------------------------------------------------------------- packing
//
// Tiles: block (e, t, kb) holds rows [128 t, 128 t + 128) and K columns
// [64 kb, 64 kb + 64) as 128 rows of 128 bytes; the 16-byte chunk c of row r
// sits at chunk position c ^ (r & 7) (the 128-byte swizzle that the
// tcgen05 shared-memory descriptor expects). Layout [e][t][kb].

// B operand: w_down[e] is [d][m] with K = m contiguous, so tiles are gathers.
__global__ void __launch_bounds__(256) k_pack_rows(const uint4* __restrict__ src, uint4* __restrict__ dst, int n_e,
                                                   int rows, int K) {
    const int cv = K / 8, kbs = K / 64, ts = rows / 128;
    const long long total = (long long)n_e * rows * cv;
    for (long long q = (long long)blockIdx.x * blockDim.x + threadIdx.x; q < total;
         q += (long long)gridDim.x * blockDim.x) {
        const long long blk = q >> 10;
        const int w = (int)(q & 1023);
        const int r = w >> 3, c = (w & 7) ^ (r & 7);
        const int kb = (int)(blk % kbs);
        const long long et = blk / kbs;
        const int t = (int)(et % ts);
        const long long e = et / ts;
        dst[q] = src[(e * rows + t * 128 + r) * cv + kb * 8 + c];
    }
}

// A operand: w_p[e] is [m][d] (K = m is the slow index), so each block
// transposes a 64 (r) x 128 (i) sub-matrix into one tile through shared
// memory: coalesced 16-byte reads into a row-major staging buffer; each warp
// then builds the 16-byte chunks of 32 consecutive tile rows i (one logical
// chunk c at a time, conflict-free column reads) and stores them at their
// swizzled positions in a second buffer (8 consecutive rows hit 8 distinct
// 16-byte bank groups); the finished tile leaves in coalesced 16-byte writes.
// The same pass accumulates the block's share of ||Gamma W_p||_F^2 =
// sum_{r,i} gamma_i^2 W_p[i, r]^2 (one fp64 partial per block, fixed order).
constexpr int kTrLd = 128 + 2;                  // staging row (bf16): 65 words, odd

__global__ void __launch_bounds__(256) k_pack_transposed(const __nv_bfloat16* __restrict__ src,
                                                         const float* __restrict__ gamma2,
                                                         uint4* __restrict__ dst, double* __restrict__ norm_part,
                                                         int d, int m) {
    __shared__ __align__(16) __nv_bfloat16 buf[64 * kTrLd];
    __shared__ __align__(16) uint4 tile[1024];
    __shared__ double sh[8];
    const int kbs = m / 64, ts = d / 128;
    const int kb = blockIdx.x % kbs;
    const int t = (blockIdx.x / kbs) % ts;
    const long long e = blockIdx.x / ((long long)kbs * ts);
    const __nv_bfloat16* s = src + (e * m + (long long)kb * 64) * d + (long long)t * 128;
    double acc = 0.0;
    for (int q = threadIdx.x; q < 64 * 16; q += 256) {
        const int r = q >> 4, c = q & 15;          // 16 chunks of 8 along i
        const uint4 v = *reinterpret_cast<const uint4*>(s + (long long)r * d + c * 8);
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
        float f[8];
        Vec16<__nv_bfloat16>::to_float(v, f);
        float sq = 0.f;
#pragma unroll
        for (int j = 0; j < 8; ++j) sq = fmaf(gamma2[t * 128 + c * 8 + j] * f[j], f[j], sq);
        acc += (double)sq;
        uint32_t* row = reinterpret_cast<uint32_t*>(&buf[r * kTrLd + c * 8]);   // 4-byte aligned (kTrLd even)
#pragma unroll
        for (int h = 0; h < 4; ++h) row[h] = w[h];
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int job = warp; job < 32; job += 8) {      // 4 groups of 32 rows x 8 logical chunks
        const int i = (job & 3) * 32 + lane, c = job >> 2;
        uint32_t w[4];
#pragma unroll
        for (int h = 0; h < 4; ++h) {
            const uint32_t lo = __bfloat16_as_ushort(buf[(8 * c + 2 * h) * kTrLd + i]);
            const uint32_t hi = __bfloat16_as_ushort(buf[(8 * c + 2 * h + 1) * kTrLd + i]);
            w[h] = lo | (hi << 16);
        }
        tile[i * 8 + (c ^ (i & 7))] = make_uint4(w[0], w[1], w[2], w[3]);
    }
    __syncthreads();
    uint4* out = dst + (long long)blockIdx.x * 1024;
    for (int q = threadIdx.x; q < 1024; q += 256) out[q] = tile[q];
    const double tot = block_sum_256(acc, sh);
    if (threadIdx.x == 0) norm_part[blockIdx.x] = tot;
}

// ---------------------------------------------------------------- GSP: Frobenius norms of the products

struct FrobParams {
    const uint8_t* a_tiles[2];   // gate, up: [n_e][d/128][m/64] tiles (rows i, K = r)
    const uint8_t* b_tiles;      // w_down:   [n_e][d/128][m/64] tiles (rows j, K = r)
    const float* gamma2;         // [d] gamma_i^2 (exact in fp32 for bf16 gamma)
    double* partial;             // [N][2][d/128 * d/256][4], indexed by the global expert
    int e0, n_e, d, m;
    int* err;
};

struct FrobItem {
    int el, path, tj, ti;
};

// Items in the order (expert, path, tj, ti): CTAs working at the same time
// share one expert's operands (L2-resident) and mostly the same B tile.
__device__ __forceinline__ FrobItem frob_item(const FrobParams& p, int item) {
    const int ti_n = p.d / 128, tj_n = p.d / 256;
    FrobItem it;
    it.ti = item % ti_n;
    item /= ti_n;
    it.tj = item % tj_n;
    item /= tj_n;
    it.path = item & 1;
    it.el = item >> 1;
    return it;
}

// 128 x 256 output tiles of C = A B^T, K = m, persistent over the items;
// warp 0 loads (bulk copies of pre-swizzled tiles), warp 1 issues the MMAs,
// warps 2..5 reduce the accumulators. Two 256-column accumulator buffers.
__global__ void __launch_bounds__(kTabThreads, 1) k_gsp_frob(const __grid_constant__ FrobParams p) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + kTabStages * kTabStage);
    uint64_t* empty = full + kTabStages;
    uint64_t* acc_full = empty + kTabStages;
    uint64_t* acc_empty = acc_full + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kTabStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&acc_full[a], 1);
            mbar_init(&acc_empty[a], 4);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(512u));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const int ti_n = p.d / 128, tj_n = p.d / 256, kblocks = p.m / kBK;
    const int n_items = p.n_e * 2 * ti_n * tj_n;

    if (warp == 0) {
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            long long issued = 0;
            for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
                const FrobItem it = frob_item(p, item);
                const uint8_t* a = p.a_tiles[it.path] + ((size_t)it.el * ti_n + it.ti) * kblocks * kTile;
                const uint8_t* b0 = p.b_tiles + ((size_t)it.el * ti_n + 2 * it.tj) * kblocks * kTile;
                const uint8_t* b1 = b0 + (size_t)kblocks * kTile;
                for (int kb = 0; kb < kblocks; ++kb) {
                    if (!mbar_wait(&empty[stage], phase ^ 1u, p.err) || *abort_flag) { ok = false; break; }
                    unsigned char* sa = smem + stage * kTabStage;
                    mbar_expect_tx(&full[stage], kTabStage);
                    bulk_g2s(sa, a + (size_t)kb * kTile, kTile, &full[stage]);
                    bulk_g2s(sa + kTabA, b0 + (size_t)kb * kTile, kTile, &full[stage]);
                    bulk_g2s(sa + kTabA + kTile, b1 + (size_t)kb * kTile, kTile, &full[stage]);
                    ++issued;
                    if (++stage == kTabStages) { stage = 0; phase ^= 1u; }
                }
            }
            if (!ok) {
                *abort_flag = 1;
                // let the copies already issued land before the CTA exits
                for (long long f = issued - 1; f >= 0 && f >= issued - kTabStages; --f)
                    if (!mbar_wait(&full[f % kTabStages], (uint32_t)((f / kTabStages) & 1), p.err)) break;
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(128, 256);
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
                if (!mbar_wait(&acc_empty[acc], acc_phase ^ 1u, p.err) || *abort_flag) { ok = false; break; }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * 256);
                for (int kb = 0; kb < kblocks; ++kb) {
                    if (!mbar_wait(&full[stage], phase, p.err) || *abort_flag) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t a_addr = smem_u32(smem + stage * kTabStage);
                    const uint32_t b_addr = a_addr + kTabA;
#pragma unroll
                    for (int kk = 0; kk < kBK / kUmmaK; ++kk)
                        mma_bf16(d_tmem, smem_desc_sw128(a_addr + kk * kUmmaK * 2),
                                 smem_desc_sw128(b_addr + kk * kUmmaK * 2), idesc, (kb > 0 || kk > 0) ? 1u : 0u);
                    mma_commit(&empty[stage]);
                    if (++stage == kTabStages) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
                mma_commit(&acc_full[acc]);
                if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
            }
            if (!ok) *abort_flag = 1;
        }
    } else {
        // warps 2..5: TMEM lanes 32 * (warp % 4) + lane hold rows i of the tile
        const int quad = warp & 3;
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
            bool ok = true;
            if (lane == 0) ok = mbar_wait(&acc_full[acc], acc_phase, p.err) && !*abort_flag;
            ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
            if (!ok) break;
            tc_fence_after();
            const FrobItem it = frob_item(p, item);
            const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(acc * 256);
            double row = 0.0;
#pragma unroll 1
            for (int c = 0; c < 16; c += 2) {
                uint32_t r0[16], r1[16];
                tmem_ld16(taddr + (uint32_t)(c * 16), r0);
                tmem_ld16(taddr + (uint32_t)(c * 16 + 16), r1);
                tmem_ld_wait();
                float s0 = 0.f, s1 = 0.f;
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const float v0 = __uint_as_float(r0[j]), v1 = __uint_as_float(r1[j]);
                    s0 = fmaf(v0, v0, s0);
                    s1 = fmaf(v1, v1, s1);
                }
                row += (double)s0;
                row += (double)s1;
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[acc]);
            const int i = it.ti * 128 + quad * 32 + lane;
            row *= (double)p.gamma2[i];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) row += __shfl_xor_sync(0xffffffffu, row, o);
            if (lane == 0) {
                const size_t tile = (size_t)it.tj * ti_n + it.ti;
                p.partial[(((size_t)(p.e0 + it.el) * 2 + it.path) * ti_n * tj_n + tile) * 4 + quad] = row;
            }
            if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(512u));
}

// ---------------------------------------------------------------- RCR

// Column means of the router weight: mean_i = (1/N) sum_e w_r[e, i].
__global__ void __launch_bounds__(256) k_rcr_colmean(const __nv_bfloat16* __restrict__ w_r, int n, int d,
                                                     double* __restrict__ mean) {
    const int i = blockIdx.x * 256 + threadIdx.x;
    if (i >= d) return;
    double s = 0.0;
    for (int e = 0; e < n; ++e) s += (double)__bfloat162float(w_r[(long long)e * d + i]);
    mean[i] = s / (double)n;
}

// Prototype of expert e (block e): x_e = q_e (* gamma), and ||q_e||_2.
__global__ void __launch_bounds__(256) k_rcr_proto(const __nv_bfloat16* __restrict__ w_r,
                                                   const double* __restrict__ mean,
                                                   const __nv_bfloat16* __restrict__ gamma, int apply_gamma, int d,
                                                   double eps, float* __restrict__ x, double* __restrict__ qnorm) {
    __shared__ double sh[8];
    __shared__ double s_inv;
    const long long e = blockIdx.x;
    const __nv_bfloat16* w = w_r + e * d;
    double ss = 0.0;
    for (int i = threadIdx.x; i < d; i += 256) {
        const double c = (double)__bfloat162float(w[i]) - mean[i];
        ss += c * c;
    }
    const double tot = block_sum_256(ss, sh);
    if (threadIdx.x == 0) s_inv = 1.0 / (sqrt(tot / (double)d) + eps);
    __syncthreads();
    const double inv = s_inv;
    double qq = 0.0;
    for (int i = threadIdx.x; i < d; i += 256) {
        const double q = ((double)__bfloat162float(w[i]) - mean[i]) * inv;
        qq += q * q;
        x[e * d + i] = (float)(apply_gamma ? q * (double)__bfloat162float(gamma[i]) : q);
    }
    const double qt = block_sum_256(qq, sh);
    if (threadIdx.x == 0) qnorm[e] = sqrt(qt);
}

// act_e[j] = SiLU(x_e . W_gate[e, j]) * (x_e . W_up[e, j]); grid (m / 64, N),
// each warp 8 rows j, one input row in shared memory.
__global__ void __launch_bounds__(256) k_rcr_gateup(const float* __restrict__ x, const __nv_bfloat16* __restrict__ w_gate,
                                                    const __nv_bfloat16* __restrict__ w_up, int d, int m,
                                                    float* __restrict__ act) {
    extern __shared__ __align__(16) float xs[];
    const long long e = blockIdx.y;
    for (int i = threadIdx.x; i < d; i += 256) xs[i] = x[e * d + i];
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int cv = d / 8;
    for (int t = 0; t < 8; ++t) {
        const int j = blockIdx.x * 64 + warp * 8 + t;
        const uint4* g = reinterpret_cast<const uint4*>(w_gate + (e * m + j) * (long long)d);
        const uint4* u = reinterpret_cast<const uint4*>(w_up + (e * m + j) * (long long)d);
        float sg = 0.f, su = 0.f;
        for (int q = lane; q < cv; q += 32) {
            float fg[8], fu[8];
            Vec16<__nv_bfloat16>::to_float(ld_stream(g + q), fg);
            Vec16<__nv_bfloat16>::to_float(ld_stream(u + q), fu);
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                sg = fmaf(fg[k], xs[q * 8 + k], sg);
                su = fmaf(fu[k], xs[q * 8 + k], su);
            }
        }
        sg = warp_sum(sg);
        su = warp_sum(su);
        if (lane == 0) act[e * m + j] = sg / (1.0f + expf(-sg)) * su;
    }
}

// y_e[c] = act_e . W_down[e, c]; grid (d / 64, N); each block writes the sum
// of its 64 y_c^2 (fixed order) to part[e][block].
__global__ void __launch_bounds__(256) k_rcr_down(const float* __restrict__ act, const __nv_bfloat16* __restrict__ w_down,
                                                  int d, int m, double* __restrict__ part) {
    extern __shared__ __align__(16) float as[];
    __shared__ double sh[8];
    const long long e = blockIdx.y;
    for (int j = threadIdx.x; j < m; j += 256) as[j] = act[e * m + j];
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int cv = m / 8;
    double y2 = 0.0;
    for (int t = 0; t < 8; ++t) {
        const int c = blockIdx.x * 64 + warp * 8 + t;
        const uint4* w = reinterpret_cast<const uint4*>(w_down + (e * d + c) * (long long)m);
        float s = 0.f;
        for (int q = lane; q < cv; q += 32) {
            float f[8];
            Vec16<__nv_bfloat16>::to_float(ld_stream(w + q), f);
#pragma unroll
            for (int k = 0; k < 8; ++k) s = fmaf(f[k], as[q * 8 + k], s);
        }
        s = warp_sum(s);
        y2 += (double)s * (double)s;   // identical in every lane
    }
    if (lane == 0) sh[warp] = y2;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < 8; ++w) t += sh[w];
        part[e * gridDim.x + blockIdx.x] = t;
    }
}

// ---------------------------------------------------------------- final normalisation

// Block e sums expert e's partials, each list in a fixed order (strided
// per-thread sums, then block_sum_256): raw[e] = {||G W_down||^2,
// ||U W_down||^2, ||G||^2, ||U||^2, ||f_e(q_e)||^2}.
__global__ void __launch_bounds__(256) k_tables_reduce(const double* __restrict__ frob, int frob_per,
                                                       const double* __restrict__ norms, int norm_per,
                                                       const double* __restrict__ rcr_part, int rcr_per, int n,
                                                       double* __restrict__ raw) {
    __shared__ double sh[8];
    const size_t e = blockIdx.x;
    const double* lists[5] = {frob + (e * 2 + 0) * frob_per, frob + (e * 2 + 1) * frob_per, norms + e * norm_per,
                              norms + ((size_t)n + e) * norm_per, rcr_part + e * rcr_per};
    const int lens[5] = {frob_per, frob_per, norm_per, norm_per, rcr_per};
    for (int l = 0; l < 5; ++l) {
        double v = 0.0;
        for (int i = threadIdx.x; i < lens[l]; i += 256) v += lists[l][i];
        const double t = block_sum_256(v, sh);
        if (threadIdx.x == 0) raw[e * 5 + l] = t;
    }
}

// One block of 1024 threads: the per-expert scores and the layer normalisation.
__global__ void __launch_bounds__(1024) k_tables_final(const double* __restrict__ raw,
                                                       const double* __restrict__ qnorm, int n, double eps,
                                                       float* __restrict__ gsp_out, float* __restrict__ rcr_out) {
    __shared__ double sg[1024], sr[1024];
    const int e = threadIdx.x;
    double ag = 0.0, ar = 0.0;
    if (e < n) {
        const double* r = raw + (size_t)e * 5;
        const double a_up = sqrt(r[3]) * sqrt(r[0]);      // ||U||_F ||G W_down||_F   (Eq. gsp_up_path)
        const double a_gate = sqrt(r[2]) * sqrt(r[1]);    // ||G||_F ||U W_down||_F   (Eq. gsp_gate_path)
        ag = sqrt(a_up * a_gate);                         // Eq. gsp_geometric_mean
        ar = sqrt(r[4]) / (qnorm[e] + eps);               // Eq. rcr_raw_amplification
    }
    sg[e] = ag;
    sr[e] = ar;
    __syncthreads();
    for (int o = 512; o > 0; o >>= 1) {
        if (e < o) {
            sg[e] += sg[e + o];
            sr[e] += sr[e + o];
        }
        __syncthreads();
    }
    if (e < n) {
        gsp_out[e] = (float)(ag / (sg[0] / n + eps));   // Eq. gsp_layer_normalization
        rcr_out[e] = (float)(ar / (sr[0] / n + eps));   // Eq. rcr_layer_normalization
    }
}

__global__ void k_gamma2(const __nv_bfloat16* __restrict__ g, float* __restrict__ g2, int d) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < d) {
        const float v = __bfloat162float(g[i]);
        g2[i] = v * v;
    }
}

ace_status tab_fail(ace_status st, const std::string& m) {
    set_last_error(m.c_str());
    return st;
}

}  // namespace
}  // namespace ace

extern "C" ace_status ace_offline_tables_device(int d, int N, int m, const void* gamma, const void* router_w,
                                                const void* w_gate, const void* w_up, const void* w_down, double eps,
                                                int rcr_apply_gamma, size_t tile_budget, float* gsp_out,
                                                float* rcr_out, void* stream) {
    using namespace ace;
    if (!gamma || !router_w || !w_gate || !w_up || !w_down || !gsp_out || !rcr_out)
        return tab_fail(ACE_ERR_INVALID_ARG, "ace_offline_tables_device: NULL pointer");
    if (d <= 0 || N <= 0 || m <= 0) return tab_fail(ACE_ERR_INVALID_ARG, "ace_offline_tables_device: sizes must be > 0");
    if (N > kMaxExperts) return tab_fail(ACE_ERR_UNSUPPORTED, "ace_offline_tables_device: N > 1024");
    if (d % 256 || m % 64 || d > 16384)
        return tab_fail(ACE_ERR_UNSUPPORTED,
                        "ace_offline_tables_device: d must be a multiple of 256 (<= 16384), m a multiple of 64");
    if (!(eps >= 0.0)) return tab_fail(ACE_ERR_INVALID_ARG, "ace_offline_tables_device: eps must be >= 0");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return tab_fail(ACE_ERR_CUDA, std::string("ace_offline_tables_device: ") + cudaGetErrorString(e));

    // experts per chunk: three tile copies (A gate, A up, B) within the budget
    const size_t per_expert = 3ull * d * m * 2;
    const size_t budget = tile_budget ? tile_budget : (1536ull << 20);
    long long chunk_ll = (long long)(budget / per_expert);
    int chunk = chunk_ll > N ? N : (int)chunk_ll;
    chunk = chunk < 1 ? 1 : chunk;
    const int ti_n = d / 128, tj_n = d / 256, frob_per = ti_n * tj_n * 4, rcr_per = d / 64;
    const int norm_per = ti_n * (m / 64);        // k_pack_transposed blocks per expert

    const size_t tiles_bytes = (size_t)chunk * d * m * 2;
    size_t off = 0;
    auto take = [&](size_t bytes) { const size_t o = off; off += (bytes + 255) & ~(size_t)255; return o; };
    const size_t o_a0 = take(tiles_bytes), o_a1 = take(tiles_bytes), o_b = take(tiles_bytes);
    const size_t o_frob = take((size_t)N * 2 * frob_per * 8), o_norm = take((size_t)N * 2 * norm_per * 8);
    const size_t o_raw = take((size_t)N * 5 * 8);
    const size_t o_mean = take((size_t)d * 8), o_x = take((size_t)N * d * 4), o_qn = take((size_t)N * 8);
    const size_t o_act = take((size_t)N * m * 4), o_rcr = take((size_t)N * rcr_per * 8);
    const size_t o_g2 = take((size_t)d * 4), o_out = take((size_t)2 * N * 4), o_err = take(4);
    unsigned char* base = nullptr;
    e = cudaMalloc(&base, off);
    if (e != cudaSuccess) return tab_fail(ACE_ERR_OOM, "ace_offline_tables_device: scratch allocation failed");
    ace_status st = ACE_OK;
    const __nv_bfloat16* wg = static_cast<const __nv_bfloat16*>(w_gate);
    const __nv_bfloat16* wu = static_cast<const __nv_bfloat16*>(w_up);
    const __nv_bfloat16* wd = static_cast<const __nv_bfloat16*>(w_down);
    float* g2 = reinterpret_cast<float*>(base + o_g2);
    int* err = reinterpret_cast<int*>(base + o_err);
    float* out = reinterpret_cast<float*>(base + o_out);
    int herr = 0;
#define TAB_CK(call)                                                                                      \
    do {                                                                                                  \
        cudaError_t e_ = (call);                                                                          \
        if (e_ != cudaSuccess) {                                                                          \
            st = tab_fail(ACE_ERR_CUDA, std::string("ace_offline_tables_device: ") + cudaGetErrorString(e_)); \
            goto done;                                                                                    \
        }                                                                                                 \
    } while (0)
    TAB_CK(cudaFuncSetAttribute(k_gsp_frob, cudaFuncAttributeMaxDynamicSharedMemorySize, kTabSmem));
    TAB_CK(ace::raise_smem_limit(k_rcr_gateup, d * 4));
    TAB_CK(ace::raise_smem_limit(k_rcr_down, m * 4));
    TAB_CK(cudaMemsetAsync(err, 0, 4, s));
    k_gamma2<<<(d + 255) / 256, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(gamma), g2, d);
    TAB_CK(cudaGetLastError());
    for (int e0 = 0; e0 < N; e0 += chunk) {
        const int n_e = N - e0 < chunk ? N - e0 : chunk;
        const size_t eo = (size_t)e0 * m * d;
        const int tblocks = n_e * ti_n * (m / 64);
        double* norm = reinterpret_cast<double*>(base + o_norm);   // [path][e][norm_per]
        k_pack_transposed<<<tblocks, 256, 0, s>>>(wg + eo, g2, reinterpret_cast<uint4*>(base + o_a0),
                                                  norm + (size_t)e0 * norm_per, d, m);
        TAB_CK(cudaGetLastError());
        k_pack_transposed<<<tblocks, 256, 0, s>>>(wu + eo, g2, reinterpret_cast<uint4*>(base + o_a1),
                                                  norm + ((size_t)N + e0) * norm_per, d, m);
        TAB_CK(cudaGetLastError());
        k_pack_rows<<<sms * 8, 256, 0, s>>>(reinterpret_cast<const uint4*>(wd + eo), reinterpret_cast<uint4*>(base + o_b),
                                            n_e, d, m);
        TAB_CK(cudaGetLastError());
        FrobParams p{};
        p.a_tiles[0] = base + o_a0;
        p.a_tiles[1] = base + o_a1;
        p.b_tiles = base + o_b;
        p.gamma2 = g2;
        p.partial = reinterpret_cast<double*>(base + o_frob);
        p.e0 = e0;
        p.n_e = n_e;
        p.d = d;
        p.m = m;
        p.err = err;
        const int items = n_e * 2 * ti_n * tj_n;
        k_gsp_frob<<<items < sms ? items : sms, kTabThreads, kTabSmem, s>>>(p);
        TAB_CK(cudaGetLastError());
    }
    k_rcr_colmean<<<(d + 255) / 256, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(router_w), N, d,
                                                  reinterpret_cast<double*>(base + o_mean));
    TAB_CK(cudaGetLastError());
    k_rcr_proto<<<N, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(router_w), reinterpret_cast<double*>(base + o_mean),
                                  static_cast<const __nv_bfloat16*>(gamma), rcr_apply_gamma, d, eps,
                                  reinterpret_cast<float*>(base + o_x), reinterpret_cast<double*>(base + o_qn));
    TAB_CK(cudaGetLastError());
    k_rcr_gateup<<<dim3(m / 64, N), 256, d * 4, s>>>(reinterpret_cast<const float*>(base + o_x), wg, wu, d, m,
                                                     reinterpret_cast<float*>(base + o_act));
    TAB_CK(cudaGetLastError());
    k_rcr_down<<<dim3(d / 64, N), 256, m * 4, s>>>(reinterpret_cast<const float*>(base + o_act), wd, d, m,
                                                   reinterpret_cast<double*>(base + o_rcr));
    TAB_CK(cudaGetLastError());
    k_tables_reduce<<<N, 256, 0, s>>>(reinterpret_cast<const double*>(base + o_frob), frob_per,
                                      reinterpret_cast<const double*>(base + o_norm), norm_per,
                                      reinterpret_cast<const double*>(base + o_rcr), rcr_per, N,
                                      reinterpret_cast<double*>(base + o_raw));
    TAB_CK(cudaGetLastError());
    k_tables_final<<<1, 1024, 0, s>>>(reinterpret_cast<const double*>(base + o_raw),
                                      reinterpret_cast<const double*>(base + o_qn), N, eps, out, out + N);
    TAB_CK(cudaGetLastError());
    TAB_CK(cudaMemcpyAsync(gsp_out, out, (size_t)N * 4, cudaMemcpyDeviceToHost, s));
    TAB_CK(cudaMemcpyAsync(rcr_out, out + N, (size_t)N * 4, cudaMemcpyDeviceToHost, s));
    TAB_CK(cudaMemcpyAsync(&herr, err, 4, cudaMemcpyDeviceToHost, s));
    TAB_CK(cudaStreamSynchronize(s));
    if (herr & kErrTimeout) st = tab_fail(ACE_ERR_TIMEOUT, "ace_offline_tables_device: a bounded device wait ran out");
#undef TAB_CK
done:
    cudaStreamSynchronize(s);
    cudaFree(base);
    return st;
}

// ace_expert_tc.cu — the SwiGLU experts (Eq. swiglu_expert) over retained
// slots only, as a persistent grouped GEMM on the 5th-generation tensor cores
// (tcgen05.mma, accumulators in TMEM, operands staged by TMA).
//
// One kernel template serves both projections and both batch regimes:
//   GEMM 1 (gate/up, K = d): act[r, j] = SiLU(h_r . W_gate[e, j]) * (h_r . W_up[e, j])
//   GEMM 2 (down,    K = m): y[r, c]   = g_hat(r) * (act[r] . W_down[e, c])
// where rows r are retained slots in expert-grouped order (the compaction's
// permutation) and e is the slot's expert.
//   * decode (SWAP): the 128-row MMA operand is a tile of weight rows and the
//     N = 16 operand is up to 16 token rows of one expert, so each weight tile
//     is streamed once and the MMA does the reduction the GEMV would do on
//     the CUDA cores;
//   * prefill: the 128-row operand is a tile of token rows, N = 256 weight rows.
// Gate and up rows are interleaved in blocks of 16 (W_gu packed at create
// time), so one accumulator tile holds matching gate and up outputs and the
// SiLU-and-product runs in the epilogue.
//
// Warp roles (192 threads): warp 0 issues TMA loads into a STAGES-deep ring,
// warp 1 owns TMEM and issues the MMAs (one thread), warps 2..5 run the
// epilogue from TMEM (each warp reads its 32-lane quadrant). Two accumulator
// buffers let the epilogue of one tile overlap the MMAs of the next. GEMM 1
// of a prefill batch on one CTA per tile and the decode kernel have four more
// warps (320 threads) that gather their token rows from h with 16-byte
// cp.async straight into the stage, so no permuted copy of h is written and
// read back; the CTA-pair GEMM 1 still loads rows gathered by k_gather_rows
// (gathering there was measured 2x slower: the partner CTA's rows need a
// relayed arrival per stage). Every mbarrier wait is bounded; on expiry the
// kernel sets kErrTimeout, stops issuing work and releases TMEM before
// returning.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <math.h>

#include "ace_device.cuh"
#include "ace_internal.h"
#include "ace_tc.cuh"

namespace ace {
namespace {

constexpr int kThreads = 192;

struct TcParams {
    CUtensorMap tm_tok;                 // token rows [rows, K] bf16
    CUtensorMap tm_w;                   // weight rows [N * w_rows, K] bf16
    const int32_t* offsets;             // [N+1]
    const int32_t* dlist;               // [N]
    const int4* tt_tab;                 // token tiles (expert, first row, rows, 0)
    const int32_t* meta;
    void* out;                          // act bf16 [rows, m], y [rows, d] (fp32 SWAP / bf16) or logits
    int K;                              // reduction length
    int w_rows;                         // weight rows per expert (2m or d)
    int w_tiles;                        // w_rows / weight tile
    const uint8_t* w_tiles_hbm;         // expert weights as pre-swizzled 16 KB tiles (nullptr: tm_w)
    int w_kb;                           // 64-column K blocks per weight row (tiled weights)
    int out_ld;                         // row length of out
    int* err;
    // single-group schedule (router logits): rows > 0 replaces the expert groups
    int single_rows;
    const float* bias;                  // [n_valid_cols] (EPI 2)
    float inv_temp;
    int use_temp;
    int n_valid_cols;                   // columns of out that exist (EPI 2)
    const int32_t* perm;                // [R] slot of row r (GEMM 2 epilogue)
    int k_splits;                       // router (EPI 2): K slices, each writing raw partials at split * split_stride
    long long split_stride;
    const float* ghat;                  // [T*k] g_hat by slot (GEMM 2 reads ghat[perm[r]])
    int k;
    const __nv_bfloat16* h_src;         // GEMM 1 of a prefill batch: h [T, K], rows gathered by the kernel
};

// ---------------------------------------------------------------- CTA-pair (cta_group::2) helpers

__device__ __forceinline__ uint32_t cluster_ctarank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// shared::cluster address of `p` (a shared::cta address) in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t mapa_shared(const void* p, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(p)), "r"(rank));
    return r;
}

// Tensor load whose completion is counted on an mbarrier of either CTA of the pair.
__device__ __forceinline__ void tma_load_2d_pair(void* smem_dst, const CUtensorMap* map, uint32_t bar_cluster, int x,
                                                 int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4}], [%2];"
        ::"r"(smem_u32(smem_dst)), "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(x), "r"(y)
        : "memory");
}

// A remote arrival that orders no memory operations: for a barrier whose waiter
// reads nothing the arriving threads wrote. An epilogue warp frees an
// accumulator this way once tcgen05.wait::ld has completed its TMEM loads
// (and tcgen05.fence::before_thread_sync has ordered them before the arrival),
// without first waiting for its own global stores of output rows.
__device__ __forceinline__ void mbar_arrive_cluster_relaxed(uint32_t bar_cluster) {
    asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster) : "memory");
}

__device__ __forceinline__ void mma_bf16_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                              uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate));
}

// Arrives on the mbarrier at the same offset in both CTAs of the pair once
// the pair's prior MMAs have completed.
__device__ __forceinline__ void mma_commit_pair(uint64_t* bar) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;"
        ::"r"(smem_u32(bar)), "h"((uint16_t)0x3)
        : "memory");
}



__device__ __forceinline__ float silu(float u) { return u / (1.0f + __expf(-u)); }

// ---------------------------------------------------------------- tile schedule

struct Tile {
    int e;        // expert
    int row0;     // first token row (perm order)
    int nrows;    // valid token rows
    int wrow0;    // first weight row in the [N * w_rows] map
    int wt;       // weight tile index within the expert
    int split;    // K slice (split-K router only, else 0)
    int kb0;      // first K block of the slice
};

// Tiles run K slice major: tile = split * n_base + (token tile * w_tiles + weight tile).
template <int TOKTILE, int WTILE>
__device__ __forceinline__ Tile tile_at(const TcParams& p, int tile, int n_base, int kblocks) {
    const int split = tile / n_base;
    tile -= split * n_base;
    const int tt = tile / p.w_tiles;
    const int wt = tile - tt * p.w_tiles;
    Tile t;
    if (p.single_rows > 0) {
        t.e = 0;
        t.row0 = tt * TOKTILE;
        t.nrows = min(TOKTILE, p.single_rows - t.row0);
    } else {
        const int4 v = p.tt_tab[tt];
        t.e = v.x;
        t.row0 = v.y;
        t.nrows = v.z;
    }
    t.wrow0 = t.e * p.w_rows + wt * WTILE;
    t.wt = wt;
    t.split = split;
    t.kb0 = split * kblocks;
    return t;
}


// Epilogue of a wide tile (this CTA's 128 token rows x 256 weight rows in
// TMEM at tbase): EPI 0 writes SiLU(gate) * up as bf16 act (gate and up
// columns interleaved in blocks of 16); EPI 1 writes the g_hat-scaled output
// row of the slot, rounded to bf16, at its expert-grouped row (the combine
// sums a token's rows in rank order). The calling warp holds tile rows
// [row_base, row_base + 32), one per lane; `gh` is the lane's g_hat (EPI 1,
// loaded before the accumulator wait so its latency overlaps the MMAs).
//
// EPI 1 writes twice the bytes per tile of EPI 0 after a K loop of m instead
// of d, so its stores bound the down GEMM. TMEM hands each lane one row, so
// the warp's values pass through `stg` (32 rows x 128 B of this warp's shared
// memory, 16-byte chunks XOR-swizzled by row so both the row-wise writes and
// the column-wise reads are free of bank conflicts) and leave as 128-byte row
// segments: each store instruction writes four whole lines instead of 32
// separate 16-byte pieces.
__device__ __forceinline__ void stage_chunk(unsigned char* stg, int lane, const uint4 (&v)[8]) {
#pragma unroll
    for (int g = 0; g < 8; ++g)
        *reinterpret_cast<uint4*>(stg + lane * 128 + ((g ^ (lane & 7)) << 4)) = v[g];
    __syncwarp();
}

// Rows [row_base, row_base + 32) of `stg`, 128 bytes each, to dst0 + row * ld_bytes.
__device__ __forceinline__ void store_chunk(const unsigned char* stg, int lane, unsigned char* dst0, size_t ld_bytes,
                                            int row_base, int nrows) {
    const int gg = lane & 7;
#pragma unroll
    for (int it = 0; it < 8; ++it) {
        const int r = it * 4 + (lane >> 3);
        const uint4 v = *reinterpret_cast<const uint4*>(stg + r * 128 + ((gg ^ (r & 7)) << 4));
        if (row_base + r < nrows) *reinterpret_cast<uint4*>(dst0 + (size_t)(row_base + r) * ld_bytes + gg * 16) = v;
    }
    __syncwarp();                                        // stg is rewritten by the next chunk
}

template <int EPI>
__device__ __forceinline__ void epilogue_wide(const TcParams& p, const Tile& t, uint32_t tbase, int row_base,
                                              int lane, float gh, unsigned char* stg) {
    constexpr int WT = 256;
    if (EPI == 0) {
        // direct 32-byte stores per row: staging these through shared memory
        // measured slower (the MMAs, not the stores, bound this GEMM)
        const int row = row_base + lane;
        __nv_bfloat16* act = static_cast<__nv_bfloat16*>(p.out);
#pragma unroll 1
        for (int blk = 0; blk < WT / 32; ++blk) {
            uint32_t g[16], u[16];
            tmem_ld16(tbase + blk * 32, g);
            tmem_ld16(tbase + blk * 32 + 16, u);
            tmem_ld_wait();
            if (row < t.nrows) {
                __align__(16) __nv_bfloat16 o[16];
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    o[i] = __float2bfloat16_rn(silu(__uint_as_float(g[i])) * __uint_as_float(u[i]));
                const int j0 = (t.wt * (WT / 32) + blk) * 16;
                uint4* dst = reinterpret_cast<uint4*>(act + (size_t)(t.row0 + row) * p.out_ld + j0);
                dst[0] = reinterpret_cast<const uint4*>(o)[0];
                dst[1] = reinterpret_cast<const uint4*>(o)[1];
            }
        }
    } else {
        unsigned char* y = static_cast<unsigned char*>(p.out) + (size_t)t.row0 * p.out_ld * 2;
#pragma unroll 1
        for (int c0 = 0; c0 < WT; c0 += 64) {
            uint32_t r[4][16];
#pragma unroll
            for (int q = 0; q < 4; ++q) tmem_ld16(tbase + c0 + 16 * q, r[q]);
            tmem_ld_wait();
            uint4 v[8];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                uint32_t w[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const __nv_bfloat162 b2 = __floats2bfloat162_rn(gh * __uint_as_float(r[q][2 * i]),
                                                                    gh * __uint_as_float(r[q][2 * i + 1]));
                    w[i] = *reinterpret_cast<const uint32_t*>(&b2);
                }
                v[2 * q] = make_uint4(w[0], w[1], w[2], w[3]);
                v[2 * q + 1] = make_uint4(w[4], w[5], w[6], w[7]);
            }
            stage_chunk(stg, lane, v);
            store_chunk(stg, lane, y + (size_t)(t.wt * WT + c0) * 2, (size_t)p.out_ld * 2, row_base, t.nrows);
        }
    }
}

// g_hat of a wide tile's row for EPI 1 (0 for rows past the tile's end).
template <int EPI>
__device__ __forceinline__ float wide_row_ghat(const TcParams& p, const Tile& t, int row) {
    if (EPI != 1 || row >= t.nrows) return 0.f;
    return p.ghat[p.perm[t.row0 + row]];
}

// ---------------------------------------------------------------- kernel

// SWAP: A (M = 128) = weight rows, B (N = TOKTILE) = token rows.
// !SWAP: A (M = 128) = token rows, B (N = WTILE) = weight rows.
// EPI 0: SwiGLU into act (bf16); EPI 1: g_hat-scaled down-projection rows
// per slot, into y (fp32 for SWAP, bf16 otherwise); EPI 2: router logits
// (fp32, + bias, / temperature), SWAP only.
template <bool SWAP, int EPI, int STAGES>
struct TcCfg {
    static constexpr int TOKTILE = SWAP ? 16 : 128;
    static constexpr int WTILE = SWAP ? 128 : 256;
    static constexpr int BM = 128;
    static constexpr int BN = SWAP ? TOKTILE : WTILE;
    static constexpr int A_ROWS = BM;
    static constexpr int B_ROWS = BN;
    static constexpr int A_BYTES = A_ROWS * kBK * 2;
    static constexpr int B_BYTES = B_ROWS * kBK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int ACC_COLS = BN;                       // fp32 columns per accumulator
    static constexpr int TMEM_COLS = (2 * ACC_COLS) < 32 ? 32 : 2 * ACC_COLS;
    static constexpr int STG_BYTES = (!SWAP && EPI == 1) ? 4 * 4096 : 0;   // EPI 1 staging, 4 KB per warp
    static constexpr int SMEM = STAGES * STAGE_BYTES + 1024 /*align*/ + 256 /*barriers*/ + STG_BYTES;
    // GEMM 1 of a prefill batch gathers its token rows itself: four more
    // warps copy them from h with 16-byte cp.async (no h_perm round trip)
    static constexpr bool GATHER = !SWAP && EPI == 0;
    static constexpr int THREADS = GATHER ? kThreads + 32 * 4 : kThreads;
};
constexpr int kGatherWarp0 = kThreads / 32;      // first token-gather warp (warps 6..9)

// 16-byte copy global -> shared through the L2 (cp.async.cg); src_bytes 0
// writes zeros without reading.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}

// Arrives on `bar` once this thread's earlier cp.async copies have landed
// (the barrier's expected count includes this arrival).
__device__ __forceinline__ void cp_async_arrive_noinc(uint64_t* bar) {
    asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(smem_u32(bar)) : "memory");
}

template <bool SWAP, int EPI, int STAGES>
__global__ void __launch_bounds__(TcCfg<SWAP, EPI, STAGES>::THREADS, 1) k_expert_tc(const __grid_constant__ TcParams p) {
    using C = TcCfg<SWAP, EPI, STAGES>;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * C::STAGE_BYTES);
    uint64_t* empty = full + STAGES;
    uint64_t* acc_full = empty + STAGES;
    uint64_t* acc_empty = acc_full + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int splits = p.k_splits > 1 ? p.k_splits : 1;
    const int kblocks = p.K / kBK / splits;          // K blocks per tile
    if (threadIdx.x == 0) {
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tm_tok)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tm_w)) : "memory");
    }

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], C::GATHER ? 1 + 128 : 1);     // + one arrival per gather thread
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&acc_full[a], 1);
            mbar_init(&acc_empty[a], 4);          // one arrival per epilogue warp
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"((uint32_t)C::TMEM_COLS));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    // everything above overlaps the predecessor kernel (PDL); its results are read below
    pdl_wait();
    const int n_base = (p.single_rows > 0 ? (p.single_rows + C::TOKTILE - 1) / C::TOKTILE : p.meta[kMetaTokTiles]) *
                       p.w_tiles;
    const int n_tiles = n_base * splits;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        // Lane 0 waits for free stages and loads the A and B tiles.
        int stage = 0;
        uint32_t phase = 0;
        bool ok = true;
        long long issued = 0;
        for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
            const Tile t = tile_at<C::TOKTILE, C::WTILE>(p, tile, n_base, kblocks);
            for (int kb = 0; kb < kblocks; ++kb) {
                int go = 1;
                if (lane == 0) go = mbar_wait_or_abort(&empty[stage], phase ^ 1u, p.err, abort_flag);
                if (!__shfl_sync(0xffffffffu, go, 0)) { ok = false; break; }
                unsigned char* sa = smem + stage * C::STAGE_BYTES;
                unsigned char* sb = sa + C::A_BYTES;
                if (lane == 0) {
                    // the gather threads' copies complete on this barrier by their own arrivals
                    mbar_expect_tx(&full[stage], C::GATHER ? C::B_BYTES : C::STAGE_BYTES);
                    const int kx = (t.kb0 + kb) * kBK;
                    if (SWAP) {
                        if (p.w_tiles_hbm)
                            bulk_g2s(sa, p.w_tiles_hbm + (((size_t)t.e * (p.w_rows / 128) + t.wt) * p.w_kb + (t.kb0 + kb)) * 16384,
                                     16384, &full[stage]);
                        else
                            tma_load_2d(sa, &p.tm_w, &full[stage], kx, t.wrow0);
                        tma_load_2d(sb, &p.tm_tok, &full[stage], kx, t.row0);
                    } else {
                        if (!C::GATHER) tma_load_2d(sa, &p.tm_tok, &full[stage], kx, t.row0);
                        if (p.w_tiles_hbm) {
                            const unsigned char* wt0 =
                                p.w_tiles_hbm + (((size_t)t.e * (p.w_rows / 128) + 2 * t.wt) * p.w_kb + (t.kb0 + kb)) * 16384;
                            bulk_g2s(sb, wt0, 16384, &full[stage]);
                            bulk_g2s(sb + 16384, wt0 + (size_t)p.w_kb * 16384, 16384, &full[stage]);
                        } else {
                            tma_load_2d(sb, &p.tm_w, &full[stage], kx, t.wrow0);
                        }
                    }
                }
                ++issued;
                if (++stage == STAGES) { stage = 0; phase ^= 1u; }
            }
        }
        if (!ok && lane == 0) {
            *abort_flag = 1;
            // our own copies must land before the block exits: wait (bounded)
            // on the full barrier of each of the last STAGES fills
            for (long long f = issued - 1; f >= 0 && f >= issued - STAGES; --f) {
                if (!mbar_wait(&full[f % STAGES], (uint32_t)((f / STAGES) & 1), p.err)) break;
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(C::BM, C::BN);
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
                if (!mbar_wait_or_abort(&acc_empty[acc], acc_phase ^ 1u, p.err, abort_flag)) { ok = false; break; }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * C::ACC_COLS);
                for (int kb = 0; kb < kblocks; ++kb) {
                    if (!mbar_wait_or_abort(&full[stage], phase, p.err, abort_flag)) { ok = false; break; }
                    // gathered rows were written by cp.async (generic proxy); the MMA reads
                    // them through the async proxy
                    if (C::GATHER) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    tc_fence_after();
                    const uint32_t a_addr = smem_u32(smem + stage * C::STAGE_BYTES);
                    const uint32_t b_addr = a_addr + C::A_BYTES;
                    // descriptors of the stage's first K step; a K step of 16 bf16 (32 B)
                    // adds 2 to the 14-bit start-address field
                    const uint64_t ad = smem_desc_sw128(a_addr), bd = smem_desc_sw128(b_addr);
#pragma unroll
                    for (int kk = 0; kk < kBK / kUmmaK; ++kk)
                        mma_bf16(d_tmem, ad + 2 * kk, bd + 2 * kk, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
                    mma_commit(&empty[stage]);           // frees the stage when these MMAs finish
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
                mma_commit(&acc_full[acc]);              // accumulator ready for the epilogue
                if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
            }
            if (!ok) *abort_flag = 1;
        }
    } else if (warp >= kGatherWarp0) {
        // ------------------------------------------------ token-row gather (GATHER: warps 6..9)
        // Thread g * 8 + c copies 16-byte chunk c of tile rows g, g + 16, ..., g + 112 for each
        // K block, into the 128-byte-swizzled layout the TMA would write (row r at 128 r, chunk
        // c at chunk c ^ (r & 7)); rows past the tile's end are zero-filled.
        if (C::GATHER) {
            const int gt = threadIdx.x - 32 * kGatherWarp0;
            const int c = gt & 7, g = gt >> 3;
            const uint32_t cx = (uint32_t)((c ^ (g & 7)) << 4);
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
                const Tile t = tile_at<C::TOKTILE, C::WTILE>(p, tile, n_base, kblocks);
                const __nv_bfloat16* src[8];
                uint32_t nb[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const int row = g + 16 * j;
                    const bool in = row < t.nrows;
                    const int tok = in ? p.perm[t.row0 + row] / p.k : 0;
                    src[j] = p.h_src + (size_t)tok * p.K + c * 8;
                    nb[j] = in ? 16u : 0u;
                }
                for (int kb = 0; kb < kblocks; ++kb) {
                    int go = 1;
                    if (lane == 0) go = mbar_wait_or_abort(&empty[stage], phase ^ 1u, p.err, abort_flag);
                    if (!__shfl_sync(0xffffffffu, go, 0)) { ok = false; break; }
                    const uint32_t sa = smem_u32(smem + stage * C::STAGE_BYTES) + (uint32_t)g * 128u + cx;
                    const int kx = (t.kb0 + kb) * kBK;
#pragma unroll
                    for (int j = 0; j < 8; ++j) cp_async16(sa + (uint32_t)j * 2048u, src[j] + kx, nb[j]);
                    cp_async_arrive_noinc(&full[stage]);
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                }
            }
            if (!ok) *abort_flag = 1;
            asm volatile("cp.async.wait_all;" ::: "memory");    // no copy in flight at exit
        }
    } else {
        // ------------------------------------------------ epilogue (warps 2..5)
        const int quad = warp & 3;                       // TMEM lane quadrant of this warp
        unsigned char* stg = smem + STAGES * C::STAGE_BYTES + 256 + quad * 4096;
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
            // the tile's rows and g_hat are read while its MMAs still run
            const Tile t = tile_at<C::TOKTILE, C::WTILE>(p, tile, n_base, kblocks);
            const float gh = SWAP ? 0.f : wide_row_ghat<EPI>(p, t, quad * 32 + lane);
            bool ok = true;
            if (lane == 0) ok = mbar_wait_or_abort(&acc_full[acc], acc_phase, p.err, abort_flag);
            ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
            if (!ok) break;
            tc_fence_after();
            const uint32_t tbase = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(acc * C::ACC_COLS);
            if (SWAP) {
                // lane = weight row (32 per warp), columns = TOKTILE (16) tokens
                uint32_t r[16];
                tmem_ld16(tbase, r);
                tmem_ld_wait();
                if (EPI == 0) {
                    // rows: 16 gate then 16 up of FFN block (4 * wt + quad)
                    const int j = (t.wt * 4 + quad) * 16 + (lane & 15);
                    __nv_bfloat16* act = static_cast<__nv_bfloat16*>(p.out);
#pragma unroll
                    for (int c = 0; c < 16; ++c) {
                        const float v = __uint_as_float(r[c]);
                        const float u = __shfl_xor_sync(0xffffffffu, v, 16);
                        if (lane < 16 && c < t.nrows)
                            act[(size_t)(t.row0 + c) * p.out_ld + j] = __float2bfloat16_rn(silu(v) * u);
                    }
                } else if (EPI == 1) {
                    const int col = t.wt * C::WTILE + quad * 32 + lane;
                    float* y = static_cast<float*>(p.out);
#pragma unroll
                    for (int c = 0; c < 16; ++c) {
                        if (c < t.nrows)
                            y[(size_t)(t.row0 + c) * p.out_ld + col] = p.ghat[p.perm[t.row0 + c]] * __uint_as_float(r[c]);
                    }
                } else {
                    // router logits: lane = expert, columns = tokens
                    const int e = t.wt * C::WTILE + quad * 32 + lane;
                    if (e < p.n_valid_cols) {
                        float* z = static_cast<float*>(p.out);
                        const float b = p.bias[e];
#pragma unroll
                        for (int c = 0; c < 16; ++c) {
                            if (c < t.nrows) {
                                float v = __uint_as_float(r[c]) + b;
                                if (p.use_temp) v = v * p.inv_temp;
                                z[(size_t)(t.row0 + c) * p.out_ld + e] = v;
                            }
                        }
                    }
                }
            } else {
                // lane = token row, columns = WTILE weight rows
                const int row = quad * 32 + lane;
                const bool valid = row < t.nrows;
                const size_t orow = (size_t)(t.row0 + row);
                if (EPI != 2) {
                    epilogue_wide<EPI>(p, t, tbase, quad * 32, lane, gh, stg);
                } else {
                    // split-K: raw partial sums per slice (bias and temperature added by the consumer)
                    float* z = static_cast<float*>(p.out) + (size_t)t.split * p.split_stride;
                    const bool raw = splits > 1;
#pragma unroll 1
                    for (int c0 = 0; c0 < C::WTILE; c0 += 16) {
                        const int col0 = t.wt * C::WTILE + c0;
                        if (col0 >= p.n_valid_cols) break;
                        uint32_t r[16];
                        tmem_ld16(tbase + c0, r);
                        tmem_ld_wait();
                        if (valid) {
                            float v[16];
#pragma unroll
                            for (int i = 0; i < 16; ++i) {
                                const int col = min(col0 + i, p.n_valid_cols - 1);
                                v[i] = __uint_as_float(r[i]);
                                if (!raw) {
                                    v[i] = v[i] + p.bias[col];
                                    if (p.use_temp) v[i] = v[i] * p.inv_temp;
                                }
                            }
                            float* zr = z + orow * p.out_ld + col0;
                            if (col0 + 16 <= p.n_valid_cols && (p.out_ld & 3) == 0) {
#pragma unroll
                                for (int i = 0; i < 16; i += 4)
                                    *reinterpret_cast<float4*>(zr + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
                            } else {
#pragma unroll
                                for (int i = 0; i < 16; ++i)
                                    if (col0 + i < p.n_valid_cols) zr[i] = v[i];
                            }
                        }
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[acc]);
            if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
        }
    }
    tc_fence_before();
    __syncthreads();
    pdl_trigger();
    tc_fence_after();
    if (warp == 1) {
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                     "r"((uint32_t)C::TMEM_COLS));
    }
}



// ---------------------------------------------------------------- decode: both GEMMs in one launch
//
// For batches of at most 256 tokens (16-token tiles, weights as the 128-row
// MMA operand) gate/up and down run in one persistent launch, so the SMs that
// finish their gate/up tiles start on down tiles instead of idling through
// the tail of a separate launch. Tiles 0 .. n1-1 are gate/up (token-tile
// major, so one token tile's gate/up tiles run together), n1 .. are down. A
// down tile's weights and act rows load after done[tt] shows that every
// gate/up epilogue warp of that token tile has written its act columns
// (release: store, proxy fence, fence, atomic; acquire: bounded spin on an
// acquiring load, then a proxy fence before the TMA). The producer takes the
// tiles from a counter (zeroed by the routing), so CTAs that drew light tiles
// draw more, and hands each index to the MMA, epilogue and gather warps
// through a ring in shared memory. Tiles leave the counter in index order and
// a CTA issues every stage of a tile before it takes the next, so a down
// tile's wait is on gate/up tiles already taken, whose MMAs and epilogues
// finish without their producers: the waits cannot form a cycle.
struct DecParams {
    CUtensorMap tm_act;                 // act rows, 16-row boxes
    const uint8_t* w_gu;                // tiled W_gu
    const uint8_t* w_down;              // tiled W_down
    const int4* tt_tab;
    const int32_t* meta;
    const int32_t* perm;
    const float* ghat;
    __nv_bfloat16* act;                 // [R, m]
    float* y;                           // [R, d]
    int* done;                          // [token tiles] gate/up epilogue warps finished (zeroed by the routing)
    int* tile_next;                     // the next tile to take (zeroed by the routing)
    int* err;
    int d, m, k;
    const __nv_bfloat16* h;             // [T, d] normalised rows: gate/up token rows are gathered from here
    long long ready_spin;               // bound (SM clock cycles) on the wait for a token tile's act rows
    int ready_extra;                    // added to that wait's target: 0, or unreachable (a test of the bound)
};

// A stage holds KBS K blocks: the KBS weight tiles of one (expert, weight
// tile) are adjacent in the tiled layout, so they arrive with one bulk copy
// of KBS x 16 KB, followed by KBS token boxes. Each stage costs a fixed
// producer / MMA / barrier round trip (measured about 0.2 us on one SM), so a
// lone SM streams about twice as fast with 36 KB stages as with 18 KB ones:
// batches that retain few experts, where few SMs have work, take KBS = 2;
// larger ones keep KBS = 1 (8 stages), which every SM streams at its share of
// the HBM bandwidth.
template <int KBS>
struct DecCfg {
    // warps 0-5 as in k_expert_tc; warps 6-9 gather the gate/up tiles' token
    // rows from h with cp.async (one 16-byte chunk of each row per thread and
    // K block) and arrive on every stage's full barrier
    static constexpr int THREADS = kThreads + 32 * 4;
    static constexpr int STAGES = KBS == 1 ? 8 : 6;
    static constexpr int A = KBS * 128 * kBK * 2;             // weight tiles
    static constexpr int B1 = 16 * kBK * 2;                   // one token box (16 rows x 64 bf16)
    static constexpr int STAGE = A + KBS * B1;
    static constexpr int SMEM = STAGES * STAGE + 1024 + 512;
};
constexpr int kDecRing = 8;             // tile indices in flight from the producer to the other roles
constexpr int kDecRingTakers = 1 + 4 + 4;   // the MMA thread, the epilogue and the gather warps
// Decode batches that take 2 K blocks per stage: few distinct retained experts.
constexpr int kDecWideStageTokens = 16;

__device__ __forceinline__ int ld_acquire(const int* p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void fence_proxy_async_global() {
    asm volatile("fence.proxy.async.global;" ::: "memory");
}

struct DecTile {
    int phase;    // 0 gate/up, 1 down
    int tt;       // token tile
    int e, row0, nrows;
    int wt;       // 128-row weight tile
    int kblocks;
};

__device__ __forceinline__ DecTile dec_tile(const DecParams& p, int tile, int n1) {
    DecTile t;
    const int wt1 = 2 * p.m / 128, wt2 = p.d / 128;
    if (tile < n1) {
        t.phase = 0;
        t.tt = tile / wt1;
        t.wt = tile - t.tt * wt1;
        t.kblocks = p.d / kBK;
    } else {
        const int j = tile - n1;
        t.phase = 1;
        t.tt = j / wt2;
        t.wt = j - t.tt * wt2;
        t.kblocks = p.m / kBK;
    }
    const int4 v = p.tt_tab[t.tt];
    t.e = v.x;
    t.row0 = v.y;
    t.nrows = v.z;
    return t;
}

template <int KBS>
__global__ void __launch_bounds__(DecCfg<KBS>::THREADS, 1) k_expert_decode(const __grid_constant__ DecParams p) {
    using C = DecCfg<KBS>;
    constexpr int kDecStages = C::STAGES, kDecStage = C::STAGE, kDecA = C::A;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + kDecStages * kDecStage);
    uint64_t* empty = full + kDecStages;
    uint64_t* acc_full = empty + kDecStages;
    uint64_t* acc_empty = acc_full + 2;
    uint64_t* ring_full = acc_empty + 2;
    uint64_t* ring_empty = ring_full + kDecRing;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(ring_empty + kDecRing);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    volatile int* ring = abort_flag + 1;        // [kDecRing] tile indices, -1 = no more
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tm_act)) : "memory");
        for (int s = 0; s < kDecStages; ++s) {
            mbar_init(&full[s], 1 + 128);           // the producer's arrival + one per gather thread
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&acc_full[a], 1);
            mbar_init(&acc_empty[a], 4);
        }
        for (int r = 0; r < kDecRing; ++r) {
            mbar_init(&ring_full[r], 1);
            mbar_init(&ring_empty[r], kDecRingTakers);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(32u));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    pdl_wait();
    const int ntt = p.meta[kMetaTokTiles];
    const int wt1 = 2 * p.m / 128;
    const int n1 = ntt * wt1, n_tiles = n1 + ntt * (p.d / 128);
    const int done_target = 4 * wt1 + p.ready_extra;

    if (warp == 0) {
        // ------------------------------------------------ producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            long long issued = 0;
            int ri = 0;
            uint32_t rph = 0;
            int tile = atomicAdd(p.tile_next, 1);
            while (ok) {
                // hand the tile (or the end) to the other roles
                if (!mbar_wait_or_abort(&ring_empty[ri], rph ^ 1u, p.err, abort_flag)) { ok = false; break; }
                ring[ri] = tile < n_tiles ? tile : -1;
                mbar_arrive(&ring_full[ri]);
                if (++ri == kDecRing) { ri = 0; rph ^= 1u; }
                if (tile >= n_tiles) break;
                const DecTile t = dec_tile(p, tile, n1);
                if (t.phase == 1) {
                    // the token tile's act rows: every gate/up epilogue warp has written
                    if (ld_acquire(p.done + t.tt) < done_target) {
                        const long long t0 = clock64();
                        while (ld_acquire(p.done + t.tt) < done_target) {
                            if (clock64() - t0 > p.ready_spin || *abort_flag) {
                                atomicOr(p.err, kErrTimeout);
                                ok = false;
                                break;
                            }
                        }
                    }
                    if (!ok) break;
                    fence_proxy_async_global();
                }
                const uint8_t* wbase = t.phase == 0 ? p.w_gu : p.w_down;
                const int wrows = t.phase == 0 ? 2 * p.m : p.d;
                for (int kb = 0; kb < t.kblocks; kb += KBS) {
                    if (!mbar_wait_or_abort(&empty[stage], phase ^ 1u, p.err, abort_flag)) { ok = false; break; }
                    unsigned char* sa = smem + stage * kDecStage;
                    // gate/up: the gather warps copy the token rows (their own arrivals)
                    mbar_expect_tx(&full[stage], t.phase == 0 ? kDecA : kDecStage);
                    bulk_g2s(sa, wbase + (((size_t)t.e * (wrows / 128) + t.wt) * t.kblocks + kb) * 16384,
                             KBS * 16384, &full[stage]);
                    if (t.phase == 1) {
#pragma unroll
                        for (int j = 0; j < KBS; ++j)
                            tma_load_2d(sa + kDecA + j * C::B1, &p.tm_act, &full[stage], (kb + j) * kBK, t.row0);
                    }
                    ++issued;
                    if (++stage == kDecStages) { stage = 0; phase ^= 1u; }
                }
                // the next tile, taken once this one's stages are out (its latency hides
                // behind the stages in flight)
                if (ok) tile = atomicAdd(p.tile_next, 1);
            }
            if (!ok) {
                *abort_flag = 1;
                for (long long f = issued - 1; f >= 0 && f >= issued - kDecStages; --f) {
                    if (!mbar_wait(&full[f % kDecStages], (uint32_t)((f / kDecStages) & 1), p.err)) break;
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(128, 16);
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            int ri = 0;
            uint32_t rph = 0;
            while (ok) {
                if (!mbar_wait_or_abort(&ring_full[ri], rph, p.err, abort_flag)) { ok = false; break; }
                const int tile = ring[ri];
                mbar_arrive(&ring_empty[ri]);
                if (++ri == kDecRing) { ri = 0; rph ^= 1u; }
                if (tile < 0) break;
                const DecTile t = dec_tile(p, tile, n1);
                if (!mbar_wait_or_abort(&acc_empty[acc], acc_phase ^ 1u, p.err, abort_flag)) { ok = false; break; }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * 16);
                for (int kb = 0; kb < t.kblocks; kb += KBS) {
                    if (!mbar_wait_or_abort(&full[stage], phase, p.err, abort_flag)) { ok = false; break; }
                    // gathered token rows were written by cp.async (generic proxy)
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    tc_fence_after();
                    const uint32_t s_addr = smem_u32(smem + stage * kDecStage);
#pragma unroll
                    for (int j = 0; j < KBS; ++j) {
                        const uint32_t a_addr = s_addr + j * 16384;               // weight tile kb + j
                        const uint32_t b_addr = s_addr + kDecA + j * C::B1;       // its token box
                        const uint64_t ad = smem_desc_sw128(a_addr), bd = smem_desc_sw128(b_addr);
#pragma unroll
                        for (int kk = 0; kk < kBK / kUmmaK; ++kk)
                            mma_bf16(d_tmem, ad + 2 * kk, bd + 2 * kk, idesc, (kb + j > 0 || kk > 0) ? 1u : 0u);
                    }
                    mma_commit(&empty[stage]);
                    if (++stage == kDecStages) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
                mma_commit(&acc_full[acc]);
                if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
            }
            if (!ok) *abort_flag = 1;
        }
    } else if (warp >= kGatherWarp0) {
        // ------------------------------------------------ token-row gather (warps 6..9)
        // Gate/up tiles: thread r * 8 + c copies chunk c of token row r (r < 16) of each K
        // block into the stage's token box, in the 128-byte-swizzled layout the TMA would
        // write; rows past the tile's end are zero-filled. Down tiles (act rows by TMA): the
        // threads only arrive, after the stage's slot is free, so every phase of the full
        // barrier gets its 128 arrivals.
        const int gt = threadIdx.x - 32 * kGatherWarp0;
        const int r = gt >> 3, c = gt & 7;
        const uint32_t off = (uint32_t)r * 128u + (uint32_t)((c ^ (r & 7)) << 4);
        int stage = 0;
        uint32_t phase = 0;
        bool ok = true;
        int ri = 0;
        uint32_t rph = 0;
        while (ok) {
            int tile = -1, go = 1;
            if (lane == 0) {
                go = mbar_wait_or_abort(&ring_full[ri], rph, p.err, abort_flag);
                if (go) tile = ring[ri];
            }
            go = __shfl_sync(0xffffffffu, go, 0);
            tile = __shfl_sync(0xffffffffu, tile, 0);
            if (!go) { ok = false; break; }
            if (lane == 0) mbar_arrive(&ring_empty[ri]);
            if (++ri == kDecRing) { ri = 0; rph ^= 1u; }
            if (tile < 0) break;
            const DecTile t = dec_tile(p, tile, n1);
            const bool in = t.phase == 0 && r < t.nrows;
            const __nv_bfloat16* src = p.h + (size_t)(in ? p.perm[t.row0 + r] / p.k : 0) * p.d + c * 8;
            for (int kb = 0; kb < t.kblocks; kb += KBS) {
                int go = 1;
                if (lane == 0) go = mbar_wait_or_abort(&empty[stage], phase ^ 1u, p.err, abort_flag);
                if (!__shfl_sync(0xffffffffu, go, 0)) { ok = false; break; }
                if (t.phase == 0) {
                    const uint32_t sb = smem_u32(smem + stage * kDecStage + kDecA) + off;
#pragma unroll
                    for (int j = 0; j < KBS; ++j) cp_async16(sb + j * C::B1, src + (kb + j) * kBK, in ? 16u : 0u);
                }
                cp_async_arrive_noinc(&full[stage]);
                if (++stage == kDecStages) { stage = 0; phase ^= 1u; }
            }
        }
        if (!ok) *abort_flag = 1;
        asm volatile("cp.async.wait_all;" ::: "memory");    // no copy in flight at exit
    } else {
        // ------------------------------------------------ epilogue (warps 2..5)
        const int quad = warp & 3;
        int acc = 0;
        uint32_t acc_phase = 0;
        int ri = 0;
        uint32_t rph = 0;
        while (true) {
            int tile = -1, go = 1;
            if (lane == 0) {
                go = mbar_wait_or_abort(&ring_full[ri], rph, p.err, abort_flag);
                if (go) tile = ring[ri];
            }
            go = __shfl_sync(0xffffffffu, go, 0);
            tile = __shfl_sync(0xffffffffu, tile, 0);
            if (!go) break;
            if (lane == 0) mbar_arrive(&ring_empty[ri]);
            if (++ri == kDecRing) { ri = 0; rph ^= 1u; }
            if (tile < 0) break;
            bool ok = true;
            if (lane == 0) ok = mbar_wait_or_abort(&acc_full[acc], acc_phase, p.err, abort_flag);
            ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
            if (!ok) break;
            tc_fence_after();
            const DecTile t = dec_tile(p, tile, n1);
            uint32_t r[16];
            tmem_ld16(tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(acc * 16), r);
            tmem_ld_wait();
            if (t.phase == 0) {
                // rows: 16 gate then 16 up of FFN block (4 * wt + quad); SwiGLU into act
                const int j = (t.wt * 4 + quad) * 16 + (lane & 15);
#pragma unroll
                for (int c = 0; c < 16; ++c) {
                    const float v = __uint_as_float(r[c]);
                    const float u = __shfl_xor_sync(0xffffffffu, v, 16);
                    if (lane < 16 && c < t.nrows)
                        p.act[(size_t)(t.row0 + c) * p.m + j] = __float2bfloat16_rn(silu(v) * u);
                }
                fence_proxy_async_global();          // act is read by the TMA of down tiles
                __threadfence();
                __syncwarp();
                if (lane == 0) atomicAdd(p.done + t.tt, 1);
            } else {
                const int col = t.wt * 128 + quad * 32 + lane;
#pragma unroll
                for (int c = 0; c < 16; ++c) {
                    if (c < t.nrows)
                        p.y[(size_t)(t.row0 + c) * p.d + col] = p.ghat[p.perm[t.row0 + c]] * __uint_as_float(r[c]);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[acc]);
            if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
        }
    }
    tc_fence_before();
    __syncthreads();
    pdl_trigger();
    tc_fence_after();
    if (warp == 1) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(32u));
}

// ---------------------------------------------------------------- CTA-pair kernel
//
// Wide tiles of 256 token rows x 256 weight rows for batches whose experts
// hold many tokens: a cluster of two CTAs issues tcgen05.mma.cta_group::2
// (M = 256, N = 256). CTA r stages token rows [128 r, 128 r + 128) and weight
// rows [128 r, 128 r + 128) of the tile, 32 KB per K block, and holds its 128
// rows of the fp32 accumulator in its own TMEM, so each SM loads two thirds of
// what a 128 x 256 tile on one SM loads for the same MACs.
//   * Both CTAs' producers load their halves; every load completes on the
//     leader's (rank 0) full barrier, which the leader arms for 64 KB.
//   * The leader's single MMA thread issues the pair's MMAs; its commits
//     arrive on the empty and acc_full barriers of both CTAs.
//   * Each CTA's epilogue drains its own TMEM rows and arrives on the
//     leader's acc_empty (count 8: four warps per CTA).
// Every mbarrier wait is bounded as in k_expert_tc; TMEM is allocated and
// freed by one warp in each CTA (cta_group::2).
constexpr int kPairStages = 6;
constexpr int kPairHalf = 128 * kBK * 2;                   // 16 KB: 128 rows x 64 bf16
constexpr int kPairStage = 2 * kPairHalf;                  // this CTA's A + B halves
constexpr int kPairSmem = kPairStages * kPairStage + 1024 + 256 + 4 * 4096;   // + epilogue staging

template <int EPI>
__global__ void __launch_bounds__(kThreads, 1) k_expert_pair(const __grid_constant__ TcParams p) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + kPairStages * kPairStage);
    uint64_t* empty = full + kPairStages;
    uint64_t* acc_full = empty + kPairStages;
    uint64_t* acc_empty = acc_full + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;
    const int unit = (int)(blockIdx.x >> 1), n_units = (int)(gridDim.x >> 1);
    const int kblocks = p.K / kBK;
    if (threadIdx.x == 0) {
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tm_tok)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tm_w)) : "memory");
        for (int s = 0; s < kPairStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&acc_full[a], 1);
            mbar_init(&acc_empty[a], 8);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(512u));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;");
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();                                          // both CTAs' barriers exist
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    pdl_wait();
    const int n_tiles = p.meta[kMetaTokTiles] * p.w_tiles;

    if (warp == 0) {
        // ------------------------------------------------ producer (both CTAs)
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            for (int tile = unit; tile < n_tiles && ok; tile += n_units) {
                const Tile t = tile_at<256, 256>(p, tile, n_tiles, kblocks);
                for (int kb = 0; kb < kblocks; ++kb) {
                    if (!mbar_wait_or_abort(&empty[stage], phase ^ 1u, p.err, abort_flag)) { ok = false; break; }
                    unsigned char* sa = smem + stage * kPairStage;
                    unsigned char* sb = sa + kPairHalf;
                    const uint32_t bar = mapa_shared(&full[stage], 0);
                    if (leader) mbar_expect_tx(&full[stage], 2 * kPairStage);
                    tma_load_2d_pair(sa, &p.tm_tok, bar, kb * kBK, t.row0 + 128 * (int)rank);
                    // weight block (e, 2 wt + rank, kb) of the tiled layout: rows of 128 B, no swizzle
                    const int blk = ((t.e * (p.w_rows / 128) + 2 * t.wt + (int)rank) * p.w_kb + kb);
                    tma_load_2d_pair(sb, &p.tm_w, bar, 0, blk * 128);
                    if (++stage == kPairStages) { stage = 0; phase ^= 1u; }
                }
            }
            if (!ok) *abort_flag = 1;
            // every fill's slot released again: no commit is still heading for this CTA
            for (int s = 0; s < kPairStages && ok; ++s) {
                if (!mbar_wait(&empty[stage], phase ^ 1u, p.err)) break;
                if (++stage == kPairStages) { stage = 0; phase ^= 1u; }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer (leader only)
        if (leader && lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(256, 256);
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            for (int tile = unit; tile < n_tiles && ok; tile += n_units) {
                if (!mbar_wait_or_abort(&acc_empty[acc], acc_phase ^ 1u, p.err, abort_flag)) { ok = false; break; }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * 256);
                for (int kb = 0; kb < kblocks; ++kb) {
                    if (!mbar_wait_or_abort(&full[stage], phase, p.err, abort_flag)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t a_addr = smem_u32(smem + stage * kPairStage);
                    const uint32_t b_addr = a_addr + kPairHalf;
                    const uint64_t ad = smem_desc_sw128(a_addr), bd = smem_desc_sw128(b_addr);
#pragma unroll
                    for (int kk = 0; kk < kBK / kUmmaK; ++kk)
                        mma_bf16_pair(d_tmem, ad + 2 * kk, bd + 2 * kk, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
                    mma_commit_pair(&empty[stage]);      // both CTAs may refill this stage
                    if (++stage == kPairStages) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
                mma_commit_pair(&acc_full[acc]);         // both CTAs' accumulator rows are ready
                if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
            }
            if (!ok) *abort_flag = 1;
        }
    } else {
        // ------------------------------------------------ epilogue (warps 2..5, both CTAs)
        const int quad = warp & 3;
        const int row_base = 128 * (int)rank + quad * 32;
        unsigned char* stg = smem + kPairStages * kPairStage + 256 + quad * 4096;
        const uint32_t acc_empty_leader[2] = {mapa_shared(&acc_empty[0], 0), mapa_shared(&acc_empty[1], 0)};
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int tile = unit; tile < n_tiles; tile += n_units) {
            // the tile's rows and g_hat are read while its MMAs still run
            const Tile t = tile_at<256, 256>(p, tile, n_tiles, kblocks);
            const float gh = wide_row_ghat<EPI>(p, t, row_base + lane);
            bool ok = true;
            if (lane == 0) ok = mbar_wait_or_abort(&acc_full[acc], acc_phase, p.err, abort_flag);
            ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
            if (!ok) break;
            tc_fence_after();
            const uint32_t tbase = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(acc * 256);
            epilogue_wide<EPI>(p, t, tbase, row_base, lane, gh, stg);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster_relaxed(acc_empty_leader[acc]);
            if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
        }
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();                                          // the pair is done with TMEM and barriers
    pdl_trigger();
    tc_fence_after();
    if (warp == 1) {
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(512u));
    }
}

// ---------------------------------------------------------------- helper kernels

// h_perm[r] = h[perm[r] / k]: token rows in expert-grouped order for the
// TMA tile loads of GEMM 1. One warp per row; d <= 4096 (16 vectors per lane).
__global__ void __launch_bounds__(256) k_gather_rows(const __nv_bfloat16* __restrict__ h,
                                                     const int32_t* __restrict__ perm,
                                                     const int32_t* __restrict__ meta,
                                                     __nv_bfloat16* __restrict__ h_perm,
                                                     int d, int k, int n_slots, int* __restrict__ err) {
    pdl_wait();
    const int R = meta[kMetaRetained];
    const int nvec = d / 8;
    const int lane = threadIdx.x & 31;
    const int wpb = blockDim.x >> 5;
    // h rows are read once per retained slot (k times a token at most): keep
    // them in L2; the h_perm rows are read once, by GEMM 1's TMA: stream them
    const uint64_t keep = l2_policy_evict_last();
    for (int r = blockIdx.x * wpb + (threadIdx.x >> 5); r < R; r += gridDim.x * wpb) {
        const int slot = perm[r];
        if (!ACE_IDX_OK(r < n_slots && slot >= 0 && slot < n_slots, err)) continue;
        const int tok = slot / k;
        const uint4* src = reinterpret_cast<const uint4*>(h + (size_t)tok * d);
        uint4* dst = reinterpret_cast<uint4*>(h_perm + (size_t)r * d);
        uint4 v[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const int c = lane + 32 * i;
            if (c < nvec) v[i] = ld_l2_keep(src + c, keep);
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const int c = lane + 32 * i;
            if (c < nvec) st_stream(dst + c, v[i]);
        }
    }
}

// out[t, c] = (x[t, c] +) sum_{i kept, rank order} y[slot_pos[t*k+i], c]
// (Eq. ace_sparse_output; y rows already carry g_hat). One thread per 8
// columns of a token, so a warp reads 256 contiguous columns of each row.
// The token's k row indices are read first and all k row loads are issued
// before the sum, which still runs in rank order.
template <typename Y>
struct Row8;
template <>
struct Row8<float> {
    float4 a, b;
    __device__ __forceinline__ void load(const float* p) {
        a = reinterpret_cast<const float4*>(p)[0];
        b = reinterpret_cast<const float4*>(p)[1];
    }
    __device__ __forceinline__ void add_to(float* acc) const {
        acc[0] += a.x; acc[1] += a.y; acc[2] += a.z; acc[3] += a.w;
        acc[4] += b.x; acc[5] += b.y; acc[6] += b.z; acc[7] += b.w;
    }
};
template <>
struct Row8<__nv_bfloat16> {
    uint4 v;
    __device__ __forceinline__ void load(const __nv_bfloat16* p) { v = *reinterpret_cast<const uint4*>(p); }
    __device__ __forceinline__ void add_to(float* acc) const {
        float f[8];
        Vec16<__nv_bfloat16>::to_float(v, f);
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[j] += f[j];
    }
};

template <typename Y, int KMAX>
__global__ void __launch_bounds__(256) k_combine_bf16(const Y* __restrict__ y, const int32_t* __restrict__ slot_pos,
                                                      const __nv_bfloat16* __restrict__ resid,
                                                      __nv_bfloat16* __restrict__ out, int n_tokens, int d, int k,
                                                      int y_rows, int* __restrict__ err) {
    pdl_wait();
    const int nq = d / 8;
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)n_tokens * nq) return;
    const int t = (int)(idx / nq), c8 = (int)(idx % nq);
    int r[KMAX];
#pragma unroll
    for (int i = 0; i < KMAX; ++i) {
        r[i] = i < k ? __ldg(slot_pos + (size_t)t * k + i) : -1;
        if (!ACE_IDX_OK(r[i] >= -1 && r[i] < y_rows, err)) r[i] = -1;
    }
    Row8<Y> v[KMAX];
#pragma unroll
    for (int i = 0; i < KMAX; ++i)
        if (r[i] >= 0) v[i].load(y + (size_t)r[i] * d + 8 * c8);
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int i = 0; i < KMAX; ++i)
        if (r[i] >= 0) v[i].add_to(acc);
    if (resid) {
        float xr[8];
        Vec16<__nv_bfloat16>::to_float(reinterpret_cast<const uint4*>(resid + (size_t)t * d)[c8], xr);
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] = xr[i] + acc[i];
    }
    __align__(16) __nv_bfloat16 o[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) o[i] = __float2bfloat16_rn(acc[i]);
    reinterpret_cast<uint4*>(out + (size_t)t * d)[c8] = *reinterpret_cast<const uint4*>(o);
}

// The combine of a layer in a stack fused with the next layer's RMSNorm
// (bf16 slot rows, T > 256): one block per token and one thread per 8-element
// chunk (blockDim = d / 8). Each thread forms its chunk of the output row as
// k_combine_bf16 does (slot rows in rank order, then the residual, rounded to
// bf16) and the sum of squares of the rounded values as one fma chain; warp 0
// then adds, for lane l, the partials of chunks l, l + 32, l + 64, ... in that
// order and reduces across lanes by the butterfly -- the order of the
// stand-alone RMSNorm, so h_next = out / sqrt(mean(out^2) + eps) * gamma_next
// has the same bits as that kernel applied to the output. A thread's 16-byte
// chunks of the slot rows come through shared memory by cp.async (k x d x 2
// bytes of dynamic shared memory per block), so no registers are held per
// load: more blocks, and so more tokens' rows, are in flight per SM.
template <int KMAX>
__global__ void __launch_bounds__(512) k_combine_norm(const __nv_bfloat16* __restrict__ y,
                                                      const int32_t* __restrict__ slot_pos,
                                                      const __nv_bfloat16* __restrict__ resid,
                                                      __nv_bfloat16* __restrict__ out,
                                                      const __nv_bfloat16* __restrict__ gamma_next,
                                                      __nv_bfloat16* __restrict__ h_next, float eps_next, int d,
                                                      int k, int y_rows, int* __restrict__ err) {
    extern __shared__ __align__(16) unsigned char cn_rows[];   // [k][blockDim.x] 16-byte chunks
    __shared__ float part_s[512];
    __shared__ float inv_s;
    pdl_wait();
    const int t = blockIdx.x, c8 = threadIdx.x;
    int r[KMAX];
#pragma unroll
    for (int i = 0; i < KMAX; ++i) {
        r[i] = i < k ? __ldg(slot_pos + (size_t)t * k + i) : -1;
        if (!ACE_IDX_OK(r[i] >= -1 && r[i] < y_rows, err)) r[i] = -1;
    }
    const uint32_t sb = smem_u32(cn_rows) + (uint32_t)c8 * 16u;
#pragma unroll
    for (int i = 0; i < KMAX; ++i)
        if (r[i] >= 0) cp_async16(sb + (uint32_t)(i * blockDim.x) * 16u, y + (size_t)r[i] * d + 8 * c8, 16u);
    asm volatile("cp.async.wait_all;" ::: "memory");   // each thread reads back only its own chunks
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int i = 0; i < KMAX; ++i)
        if (r[i] >= 0) {
            float f[8];
            Vec16<__nv_bfloat16>::to_float(
                *reinterpret_cast<const uint4*>(cn_rows + ((size_t)i * blockDim.x + c8) * 16), f);
#pragma unroll
            for (int j = 0; j < 8; ++j) acc[j] += f[j];
        }
    if (resid) {
        float xr[8];
        Vec16<__nv_bfloat16>::to_float(reinterpret_cast<const uint4*>(resid + (size_t)t * d)[c8], xr);
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[j] = xr[j] + acc[j];
    }
    __align__(16) __nv_bfloat16 o[8];
    float f[8], part = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        o[j] = __float2bfloat16_rn(acc[j]);
        f[j] = __bfloat162float(o[j]);
        part = fmaf(f[j], f[j], part);
    }
    reinterpret_cast<uint4*>(out + (size_t)t * d)[c8] = *reinterpret_cast<const uint4*>(o);
    part_s[c8] = part;
    __syncthreads();
    if (threadIdx.x < 32) {
        float ss = 0.f;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) ss += part_s[threadIdx.x + 32 * w];
        ss = warp_sum(ss);
        if (threadIdx.x == 0) inv_s = 1.0f / sqrtf(ss / (float)d + eps_next);
    }
    __syncthreads();
    const float inv = inv_s;
    float gm[8];
    Vec16<__nv_bfloat16>::to_float(reinterpret_cast<const uint4*>(gamma_next)[c8], gm);
#pragma unroll
    for (int j = 0; j < 8; ++j) o[j] = __float2bfloat16_rn(f[j] * inv * gm[j]);
    reinterpret_cast<uint4*>(h_next + (size_t)t * d)[c8] = *reinterpret_cast<const uint4*>(o);
}

template <int KMAX>
cudaError_t launch_combine_norm(const __nv_bfloat16* y, const int32_t* sp, const __nv_bfloat16* resid,
                                __nv_bfloat16* out, const ace_layer* next, int T, int d, int k, int y_rows, int* err,
                                cudaStream_t s) {
    // d is a multiple of 256 (tensor-core layers) and at most 4096: d / 8 threads, whole warps
    return launch_pdl(k_combine_norm<KMAX>, dim3(T), dim3(d / 8), (size_t)k * d * 2, s, y, sp, resid, out,
                      static_cast<const __nv_bfloat16*>(next->gamma), static_cast<__nv_bfloat16*>(next->ws.h),
                      next->desc.rms_eps, d, k, y_rows, err);
}

// ---------------------------------------------------------------- host side

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

cudaError_t get_encoder() {
    if (g_encode) return cudaSuccess;
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess) return e;
    if (q != cudaDriverEntryPointSuccess || !fn) return cudaErrorNotSupported;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    return cudaSuccess;
}

// 2-D bf16 map over [rows, cols] (row-major), box [box_rows, 64], 128-byte swizzle.
// With swizzle == false the map copies rows verbatim (the tiled expert weights
// are stored already swizzled).
cudaError_t make_map(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows,
                     bool swizzle = true) {
    cudaError_t e = get_encoder();
    if (e != cudaSuccess) return e;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {cols * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kBK, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t set_pair_attr(const void* k) {
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, kPairSmem);
    if (e != cudaSuccess) return e;
    return prefer_shared(k);
}

// Pair clusters that fit at once (one CTA per SM, clusters of two).
cudaError_t max_pair_clusters(const void* k, int* n) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kPairSmem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaOccupancyMaxActiveClusters(n, k, &cfg);
}

template <int EPI>
cudaError_t launch_pair(const ace_layer* L, const TcParams& p, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * L->pair_clusters);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kPairSmem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, k_expert_pair<EPI>, p);
}

constexpr int kStagesSwap = 8;
constexpr int kStagesWide = 4;

template <bool SWAP, int EPI>
constexpr int stages_for() { return SWAP ? kStagesSwap : kStagesWide; }

template <bool SWAP, int EPI>
cudaError_t set_attr() {
    constexpr int S = stages_for<SWAP, EPI>();
    cudaError_t e = cudaFuncSetAttribute(k_expert_tc<SWAP, EPI, S>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         TcCfg<SWAP, EPI, S>::SMEM);
    if (e != cudaSuccess) return e;
    return prefer_shared(k_expert_tc<SWAP, EPI, S>);
}

template <bool SWAP, int EPI>
cudaError_t launch_gemm(const ace_layer* L, const TcParams& p, cudaStream_t s) {
    constexpr int S = stages_for<SWAP, EPI>();
    return launch_pdl(k_expert_tc<SWAP, EPI, S>, dim3(L->num_sms), dim3(TcCfg<SWAP, EPI, S>::THREADS),
                      TcCfg<SWAP, EPI, S>::SMEM, s, p);
}

// Expert weights as tiles in HBM: block (e, t, kb) holds weight rows
// [128 t, 128 t + 128) x columns [64 kb, 64 kb + 64) of expert e, 16 KB,
// already in the 128-byte-swizzled order of a shared-memory operand tile
// (row r at 128 r, its 16-byte chunk c at chunk c ^ (r & 7)). A stage's
// weights then arrive with one contiguous 16 KB bulk copy. Blocks are stored
// [e][t][kb]. For W_gu the rows interleave gate and up in blocks of 16:
// row 32b + i is W_gate row 16b + i (i < 16) or W_up row 16b + i - 16.
template <bool GU>
__global__ void __launch_bounds__(256) k_pack_tiles(const uint4* __restrict__ src0, const uint4* __restrict__ src1,
                                                    uint4* __restrict__ dst, int n_exp, int rows, int cols) {
    const int cv = cols / 8;                      // 16-byte chunks per source row
    const int kbs = cols / 64, wts = rows / 128;
    const long long total = (long long)n_exp * rows * cv;
    for (long long q = (long long)blockIdx.x * blockDim.x + threadIdx.x; q < total;
         q += (long long)gridDim.x * blockDim.x) {
        const long long blk = q >> 10;            // 1024 chunks per 16 KB block
        const int w = (int)(q & 1023);
        const int r = w >> 3, c = (w & 7) ^ (r & 7);
        const int kb = (int)(blk % kbs);
        const long long et = blk / kbs;
        const int t = (int)(et % wts), e = (int)(et / wts);
        const int row = t * 128 + r, chunk = kb * 8 + c;
        uint4 v;
        if (GU) {
            const int b = row >> 5, li = row & 31;
            const int j = b * 16 + (li & 15);
            v = (li < 16 ? src0 : src1)[((long long)e * (rows / 2) + j) * cv + chunk];
        } else {
            v = src0[((long long)e * rows + row) * cv + chunk];
        }
        dst[q] = v;
    }
}

}  // namespace

cudaError_t tc_pack_weights(ace_layer* L, const void* w_gate, const void* w_up, const void* w_down, cudaStream_t s) {
    const ace_layer_desc& D = L->desc;
    k_pack_tiles<true><<<L->num_sms * 8, 256, 0, s>>>((const uint4*)w_gate, (const uint4*)w_up, (uint4*)L->w_gu,
                                                      D.n_experts, 2 * D.ffn, D.hidden);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_pack_tiles<false><<<L->num_sms * 8, 256, 0, s>>>((const uint4*)w_down, nullptr, (uint4*)L->w_down,
                                                       D.n_experts, D.hidden, D.ffn);
    return cudaGetLastError();
}

// Expected retained slots per expert (ratio mode: the requested skip ratio;
// threshold mode: none skipped) decide the wide-tile kernel: CTA pairs with
// 256-row tiles once experts average 256 or more slots, else one CTA per
// 128-row tile.
bool tc_use_pair(const ace_layer* L, int T, ace_skip_ctl ctl) {
    if (T <= kTcSmallT || L->pair_clusters < 1) return false;
    const ace_layer_desc& D = L->desc;
    const double keep = ctl.mode == ACE_SKIP_RATIO ? 1.0 - (double)ctl.value : 1.0;
    return (double)T * D.top_k * keep >= 256.0 * D.n_experts;
}

int tc_token_tile(const ace_layer* L, int T, ace_skip_ctl ctl) {
    return T <= kTcSmallT ? 16 : (tc_use_pair(L, T, ctl) ? 256 : 128);
}

bool tc_supported(const ace_layer* L) {
    const ace_layer_desc& D = L->desc;
    return D.dtype == ACE_BF16 && D.ffn % 128 == 0 && D.hidden % 256 == 0;
}

cudaError_t tc_init(ace_layer* L) {
    if (!tc_supported(L)) return cudaSuccess;
    const ace_layer_desc& D = L->desc;
    cudaError_t e;
    if ((e = set_attr<true, 0>()) != cudaSuccess) return e;
    if ((e = set_attr<true, 1>()) != cudaSuccess) return e;
    if ((e = set_attr<false, 0>()) != cudaSuccess) return e;
    if ((e = set_attr<false, 1>()) != cudaSuccess) return e;
    if ((e = set_attr<false, 2>()) != cudaSuccess) return e;
    if ((e = cudaFuncSetAttribute(k_expert_decode<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  DecCfg<1>::SMEM)) != cudaSuccess)
        return e;
    if ((e = prefer_shared(k_expert_decode<1>)) != cudaSuccess) return e;
    if ((e = cudaFuncSetAttribute(k_expert_decode<2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  DecCfg<2>::SMEM)) != cudaSuccess)
        return e;
    if ((e = prefer_shared(k_expert_decode<2>)) != cudaSuccess) return e;
    if ((e = set_pair_attr((const void*)k_expert_pair<0>)) != cudaSuccess) return e;
    if ((e = set_pair_attr((const void*)k_expert_pair<1>)) != cudaSuccess) return e;
    int c0 = 0, c1 = 0;
    if ((e = max_pair_clusters((const void*)k_expert_pair<0>, &c0)) != cudaSuccess) return e;
    if ((e = max_pair_clusters((const void*)k_expert_pair<1>, &c1)) != cudaSuccess) return e;
    L->pair_clusters = c0 < c1 ? c0 : c1;
    if ((e = prefer_shared(k_gather_rows)) != cudaSuccess) return e;
    // the stack's combine stages k slot-row chunks per thread: k x d x 2 bytes per block
    if ((e = raise_smem_limit(k_combine_norm<8>, 8 * D.hidden * 2)) != cudaSuccess) return e;
    if ((e = raise_smem_limit(k_combine_norm<kMaxTopK>, kMaxTopK * D.hidden * 2)) != cudaSuccess) return e;
    if ((e = prefer_shared(k_combine_norm<8>)) != cudaSuccess) return e;
    if ((e = prefer_shared(k_combine_norm<kMaxTopK>)) != cudaSuccess) return e;

    // row counts as allocated at create time (padded to at least 256 rows)
    const uint64_t rows = (uint64_t)D.max_tokens * D.top_k < 256 ? 256 : (uint64_t)D.max_tokens * D.top_k;
    const uint64_t h_rows = D.max_tokens < 256 ? 256 : (uint64_t)D.max_tokens;
    const uint64_t n_pad = ((uint64_t)D.n_experts + 255) / 256 * 256;
    const uint64_t n = D.n_experts, d = D.hidden, m = D.ffn;
    // token maps: h_perm (GEMM 1) and act (GEMM 2), tiles of 16 / 128 rows
    if ((e = make_map(&L->tcm.tok1_big, L->ws.h_perm, rows, d, 128)) != cudaSuccess) return e;
    if ((e = make_map(&L->tcm.tok2_small, L->ws.act_bf16, rows, m, 16)) != cudaSuccess) return e;
    if ((e = make_map(&L->tcm.tok2_big, L->ws.act_bf16, rows, m, 128)) != cudaSuccess) return e;
    // weight maps: W_gu [N * 2m, d] and W_down [N * d, m]
    // router: h [Tmax, d] in 128-row boxes, W_r [N, d] in 256-row boxes
    if ((e = make_map(&L->tcm.h_rows_big, L->ws.h, h_rows, d, 128)) != cudaSuccess) return e;
    // tiled expert weights as rows of 64 bf16 (16 KB tiles = 128 rows), copied verbatim
    if ((e = make_map(&L->tcm.wgu_rows, L->w_gu, n * 2 * m * d / 64, 64, 128, false)) != cudaSuccess) return e;
    if ((e = make_map(&L->tcm.wd_rows, L->w_down, n * d * m / 64, 64, 128, false)) != cudaSuccess) return e;
    if ((e = make_map(&L->tcm.tok1_small, L->ws.h_perm, rows, d, 16)) != cudaSuccess) return e;
    if ((e = make_map(&L->tcm.w_router_big, L->router_w, n_pad, d, 256)) != cudaSuccess) return e;
    return cudaSuccess;
}

// Router logits on the tensor cores for batches over 256 tokens (smaller
// ones are routed by the fused kernel): 128 tokens x 256 experts per tile,
// so W_r (N padded to 256 rows) is re-read from L2 once per 128 tokens.
int router_splits(const ace_layer* L, int T) {
    const ace_layer_desc& D = L->desc;
    const int base = ((T + 127) / 128) * ((D.n_experts + 255) / 256);
    const int kblocks = D.hidden / kBK;
    int sp = 1;
    // the partials [splits, T, N] fp32 live in act_bf16 ([T*k, m] bf16), idle while routing
    while (sp < 8 && 2 * sp * base <= L->num_sms && kblocks % (2 * sp) == 0 && kblocks / (2 * sp) >= 4 &&
           (size_t)2 * sp * D.n_experts * 4 <= (size_t)D.top_k * D.ffn * 2)
        sp *= 2;
    return sp;
}

cudaError_t launch_router_tc(const ace_layer* L, int T, cudaStream_t s) {
    const ace_layer_desc& D = L->desc;
    TcParams p{};
    p.tm_tok = L->tcm.h_rows_big;
    p.tm_w = L->tcm.w_router_big;
    p.k_splits = router_splits(L, T);
    p.split_stride = (long long)T * D.n_experts;
    p.out = p.k_splits > 1 ? L->ws.act_bf16 : (void*)L->ws.logits;
    p.K = D.hidden;
    p.w_rows = D.n_experts;
    p.w_tiles = (D.n_experts + 255) / 256;
    p.out_ld = D.n_experts;
    p.err = L->ws.err;
    p.single_rows = T;
    p.bias = L->router_b;
    p.inv_temp = 1.0f / D.router_temp;
    p.use_temp = D.router_temp != 1.0f;
    p.n_valid_cols = D.n_experts;
    return launch_gemm<false, 2>(L, p, s);
}

cudaError_t launch_experts_tc(const ace_layer* L, const void* x, void* out, int T, ace_skip_ctl ctl, cudaStream_t s,
                              cudaEvent_t* ev, const ace_layer* next) {
    const bool pair = tc_use_pair(L, T, ctl);
    const __nv_bfloat16* resid = L->desc.add_residual ? static_cast<const __nv_bfloat16*>(x) : nullptr;
    const ace_layer_desc& D = L->desc;
    const Workspace& W = L->ws;
    const int d = D.hidden, m = D.ffn, k = D.top_k;
    const bool small = T <= kTcSmallT;
    cudaError_t e = cudaSuccess;
    // token rows in expert-grouped order for the CTA-pair GEMM 1's 256-row TMA tiles;
    // the decode kernel and the single-CTA prefill GEMM 1 gather their rows themselves
    if (pair) {
        e = launch_pdl(k_gather_rows, dim3(L->num_sms * 4), dim3(256), 0, s, (const __nv_bfloat16*)W.h,
                       (const int32_t*)W.perm, (const int32_t*)W.meta, (__nv_bfloat16*)W.h_perm, d, k,
                       T * k, W.err);
        if (e != cudaSuccess) return e;
    }
    if (small) {
        // both GEMMs in one persistent launch (k_expert_decode), then the combine
        if (ev) ace::record_stage(ev[0], s);
        DecParams q{};
        q.tm_act = L->tcm.tok2_small;
        q.w_gu = static_cast<const uint8_t*>(L->w_gu);
        q.w_down = static_cast<const uint8_t*>(L->w_down);
        q.tt_tab = W.tt_tab;
        q.meta = W.meta;
        q.perm = W.perm;
        q.ghat = W.ghat;
        q.act = static_cast<__nv_bfloat16*>(W.act_bf16);
        q.y = W.yslot;
        q.done = W.dec_done;
        q.tile_next = W.meta + kMetaDecNext;
        q.h = static_cast<const __nv_bfloat16*>(W.h);
        q.err = W.err;
        q.d = d;
        q.m = m;
        q.k = k;
        q.ready_spin = L->dbg_ready_spin > 0 ? L->dbg_ready_spin : kSpinCycles;
        q.ready_extra = L->dbg_ready_spin > 0 ? (1 << 30) : 0;
        // K blocks are even: d is a multiple of 256 and m of 128 on this path
        e = T <= kDecWideStageTokens
                ? launch_pdl(k_expert_decode<2>, dim3(L->num_sms), dim3(DecCfg<2>::THREADS), DecCfg<2>::SMEM, s, q)
                : launch_pdl(k_expert_decode<1>, dim3(L->num_sms), dim3(DecCfg<1>::THREADS), DecCfg<1>::SMEM, s, q);
        if (e != cudaSuccess) return e;
        if (ev) {                           // gate/up and down share one launch: the down stage reads 0
            ace::record_stage(ev[1], s);
            ace::record_stage(ev[2], s);
        }
        const long long nthreads = (long long)T * (d / 8);
        const dim3 grid((unsigned)((nthreads + 255) / 256));
        const int yr = T * k;                 // fp32 slot rows of this batch
        e = k <= 8 ? launch_pdl(k_combine_bf16<float, 8>, grid, dim3(256), 0, s, (const float*)W.yslot,
                                (const int32_t*)W.slot_pos, resid, (__nv_bfloat16*)out, T, d, k, yr, W.err)
                   : launch_pdl(k_combine_bf16<float, kMaxTopK>, grid, dim3(256), 0, s, (const float*)W.yslot,
                                (const int32_t*)W.slot_pos, resid, (__nv_bfloat16*)out, T, d, k, yr, W.err);
        if (ev) ace::record_stage(ev[3], s);
        return e;
    }
    if (ev) ace::record_stage(ev[0], s);
    TcParams p1{};
    p1.tm_tok = small ? L->tcm.tok1_small : L->tcm.tok1_big;
    p1.w_tiles_hbm = static_cast<const uint8_t*>(L->w_gu);
    p1.w_kb = d / kBK;
    p1.offsets = W.offsets;
    p1.dlist = W.dlist;
    p1.tt_tab = W.tt_tab;
    p1.meta = W.meta;
    p1.perm = W.perm;
    p1.ghat = W.ghat;
    p1.k = k;
    p1.out = W.act_bf16;
    p1.h_src = static_cast<const __nv_bfloat16*>(W.h);
    p1.K = d;
    p1.w_rows = 2 * m;
    p1.w_tiles = 2 * m / (small ? 128 : 256);
    p1.out_ld = m;
    p1.err = W.err;
    if (pair) {
        TcParams q = p1;
        q.tm_w = L->tcm.wgu_rows;
        q.w_tiles = 2 * m / 256;
        e = launch_pair<0>(L, q, s);
    } else {
        e = small ? launch_gemm<true, 0>(L, p1, s) : launch_gemm<false, 0>(L, p1, s);
    }
    if (e != cudaSuccess) return e;
    if (ev) ace::record_stage(ev[1], s);
    TcParams p2 = p1;
    p2.tm_tok = small ? L->tcm.tok2_small : L->tcm.tok2_big;
    p2.w_tiles_hbm = static_cast<const uint8_t*>(L->w_down);
    p2.w_kb = m / kBK;
    // y per slot: fp32 rows for SWAP tiles; bf16 rows otherwise, written over
    // h_perm, which GEMM 1 (complete before GEMM 2 reads anything) no longer needs
    p2.out = small ? (void*)W.yslot : W.h_perm;
    p2.K = m;
    p2.w_rows = d;
    p2.w_tiles = d / (small ? 128 : 256);
    p2.out_ld = d;
    if (pair) {
        TcParams q = p2;
        q.tm_w = L->tcm.wd_rows;
        q.w_tiles = d / 256;
        e = launch_pair<1>(L, q, s);
    } else {
        e = small ? launch_gemm<true, 1>(L, p2, s) : launch_gemm<false, 1>(L, p2, s);
    }
    if (e != cudaSuccess) return e;
    if (ev) ace::record_stage(ev[2], s);
    const long long nthreads = (long long)T * (d / 8);
    const dim3 grid((unsigned)((nthreads + 255) / 256));
    const int32_t* sp = W.slot_pos;
    __nv_bfloat16* o = static_cast<__nv_bfloat16*>(out);
    const int yr = T * k;                     // slot rows of this batch
    if (small) {
        const float* y = W.yslot;
        e = k <= 8 ? launch_pdl(k_combine_bf16<float, 8>, grid, dim3(256), 0, s, y, sp, resid, o, T, d, k, yr, W.err)
                   : launch_pdl(k_combine_bf16<float, kMaxTopK>, grid, dim3(256), 0, s, y, sp, resid, o, T, d, k, yr,
                                W.err);
    } else if (next) {
        const __nv_bfloat16* y = static_cast<const __nv_bfloat16*>(W.h_perm);
        e = k <= 8 ? launch_combine_norm<8>(y, sp, resid, o, next, T, d, k, yr, W.err, s)
                   : launch_combine_norm<kMaxTopK>(y, sp, resid, o, next, T, d, k, yr, W.err, s);
    } else {
        const __nv_bfloat16* y = static_cast<const __nv_bfloat16*>(W.h_perm);
        e = k <= 8 ? launch_pdl(k_combine_bf16<__nv_bfloat16, 8>, grid, dim3(256), 0, s, y, sp, resid, o, T, d, k, yr,
                                W.err)
                   : launch_pdl(k_combine_bf16<__nv_bfloat16, kMaxTopK>, grid, dim3(256), 0, s, y, sp, resid, o, T, d,
                                k, yr, W.err);
    }
    if (ev) ace::record_stage(ev[3], s);
    return e;
}

}  // namespace ace

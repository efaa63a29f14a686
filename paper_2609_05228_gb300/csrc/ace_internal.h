// ace_internal.h — layer object, workspace layout and kernel launchers of
// libace.so. Host and device code of the library share it; nothing outside
// csrc/ includes it.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>
#include <vector>

#include "ace.h"

namespace ace {

// Device error word bits (ace_layer::ws.err).
enum : int {
    kErrNumeric = 1,   // a router logit was NaN / the gate sum was not finite
    kErrTimeout = 2,   // a bounded device wait ran out
    kErrBounds = 4,    // an index check failed (debug-style guard, access skipped)
};

// meta[] slots (int32, device): written by the compaction's last block.
enum : int {
    kMetaRetained = 0,     // R
    kMetaTicket = 1,       // last-block ticket (reset by the last block)
    kMetaDistinct = 2,     // D, experts with >= 1 retained slot
    kMetaSlice1 = 3,       // gate/up GEMV: rows of m per work item
    kMetaSlice2 = 4,       // down GEMV: rows of d per work item
    kMetaTiles1 = 5,       // tensor-core GEMM 1 tiles
    kMetaTiles2 = 6,       // tensor-core GEMM 2 tiles
    kMetaTicket2 = 7,      // second ticket (fused small-T routing)
    kMetaTokTiles = 8,     // token tiles of the tensor-core expert schedule
    kMetaSelCount = 9,     // large-T threshold select: candidates collected (kept zero between calls)
    kMetaSelPrefix = 10,   //   first digit, as the key prefix
    kMetaSelWant = 11,     //   rank still wanted inside the first digit
    kMetaSelBelow = 12,    //   candidates below the first digit
    kMetaDecNext = 13,     // decode expert kernel: the next tile to take (zeroed by the routing)
    kMetaCount = 16,
};

constexpr int kChunk = 64;            // tokens per compaction block (large-T route)
constexpr int kTcSmallT = 256;       // tensor-core experts: decode tiling up to this many tokens
constexpr int kMaxExperts = 1024;
constexpr int kMaxTopK = 16;
constexpr int kGemvTokenChunk = 8;   // tokens processed per weight pass in the GEMVs

struct Workspace {
    void* h = nullptr;           // [Tmax, d] dtype: RMSNorm output
    float* logits = nullptr;     // [Tmax, N]
    int32_t* ids = nullptr;      // [Tmax, k] rank order
    float* gates = nullptr;      // [Tmax, k] g
    float* cval = nullptr;       // [Tmax, k] c of the skip rule (ACE: max(p_gsp, p_rcr))
    uint32_t* keys = nullptr;    // [Tmax, k] ratio-mode candidate keys
    uint8_t* skip = nullptr;     // [Tmax, k]
    float* ghat = nullptr;       // [Tmax, k]
    float* tau = nullptr;        // [1]
    int32_t* chunk_counts = nullptr;  // [n_chunks, N] counts, then per-chunk bases
    int32_t* offsets = nullptr;  // [N+1]
    int32_t* dlist = nullptr;    // [N] distinct retained experts, increasing
    int32_t* perm = nullptr;     // [Tmax*k]
    int32_t* slot_pos = nullptr; // [Tmax*k] row of slot t*k+i in perm order, -1 if skipped
    int32_t* meta = nullptr;     // [kMetaCount]
    float* act = nullptr;        // [Tmax*k, m] fp32 (CUDA-core path)
    float* yslot = nullptr;      // [Tmax*k, d] fp32: g_hat-scaled expert outputs per retained slot
    void* h_perm = nullptr;      // [Tmax*k, d] bf16: h rows in expert-grouped order (tensor path); for
                                 // batches over 256 tokens GEMM 2 then writes its bf16 y rows over it
    void* act_bf16 = nullptr;    // [Tmax*k, m] bf16 (tensor path)
    int32_t* tt_off = nullptr;   // [N+1] token-tile prefix over distinct experts
    int32_t* dec_done = nullptr; // [tiles of tt_tab] gate/up warps finished per token tile (decode kernel)
    int4* tt_tab = nullptr;      // [N + Tmax*k/16 + 1] token tiles: (expert, first row, rows, 0)
    int32_t* tile_cnt = nullptr; // [Tmax/8 + 1] per-token-tile tickets of the fused small-T kernel
    int32_t* sel_hist = nullptr; // [4096 + 1024] digit histograms of the threshold keys (kept zero between calls)
    uint32_t* sel_cand = nullptr;// [Tmax*k] keys of the chosen first digit (large-T threshold select)
    int* err = nullptr;          // device error word
    void* x_stage = nullptr;     // [Tmax, d] dtype: host-API staging
    void* out_stage = nullptr;   // [Tmax, d]
};

// Tensor maps of the tensor-core expert path (built once at create time).
struct TcMaps {
    CUtensorMap tok1_small, tok1_big;   // h_perm, boxes of 16 / 128 rows
    CUtensorMap tok2_small, tok2_big;   // act_bf16, boxes of 16 / 128 rows
    CUtensorMap h_rows_big, w_router_big;   // router GEMM (batches over 256 tokens): 128-row / 256-row boxes
    CUtensorMap wgu_rows, wd_rows;      // tiled W_gu / W_down as 128-B rows (CTA-pair kernel), no swizzle
};

}  // namespace ace

// A host-buffer forward (copy in, forward, copy out) captured as a CUDA
// graph and replayed while the call's arguments stay the same.
struct AceHostGraph {
    cudaGraphExec_t exec = nullptr;
    cudaStream_t own = nullptr;          // used for calls on the legacy default stream
    cudaStream_t stream = nullptr;       // the stream the graph was captured for
    const void* x_host = nullptr;
    void* out_host = nullptr;
    const void* x_mapped = nullptr;      // device addresses of the page-locked host buffers at capture
    void* out_mapped = nullptr;
    int T = -1;
    ace_skip_ctl ctl{0, 0.f, 0};
    bool profiling = false;
    int* err_host = nullptr;             // pinned copies of the device error words, written by the graph
    int n_err = 0;
};

struct ace_stack {
    AceHostGraph hg;
    std::vector<ace_layer*> layers;
    void* buf[2] = {nullptr, nullptr};   // [max_tokens, d] bf16: alternating layer outputs
    int max_tokens = 0;
    int hidden = 0;
};

// Debug build (ACE_DEBUG_CHECKS): every device array of a layer is
// allocated kCanaryBytes longer and the tail filled with kCanaryByte; the
// synchronising calls check that no kernel wrote past an array's end.
namespace ace {
constexpr size_t kCanaryBytes = 256;
constexpr unsigned char kCanaryByte = 0xA5;
struct Canary {
    const char* name;   // the array's field name
    unsigned char* at;  // first byte past the array
};
}  // namespace ace

struct ace_layer {
    ace_layer_desc desc;
    int device = 0;
    int num_sms = 0;
    int pair_clusters = 0;       // CTA pairs of the wide-tile expert kernel resident at once
    int tt_cap = 0;              // entries allocated in ws.tt_tab
    std::vector<ace::Canary> canaries;   // debug build only
    size_t elem = 2;             // bytes per element of dtype
    // layer-owned weights
    void* router_w = nullptr;    // [N, d]
    float* router_b = nullptr;   // [N] (zeros when there is no bias)
    void* w_gate = nullptr;      // [N, m, d] (CUDA-core path only)
    void* w_up = nullptr;        // [N, m, d] (CUDA-core path only)
    void* w_gu = nullptr;        // tensor path: [N][2m/128][d/64] tiles of 128 x 64 bf16 (16 KB, 128-byte
                                 // swizzled), gate/up rows interleaved in blocks of 16
    bool tc = false;             // tensor-core expert path in use
    ace::TcMaps tcm;
    void* w_down = nullptr;      // [N, d, m]; tensor path: [N][d/128][m/64] tiles like w_gu
    void* gamma = nullptr;       // [d]
    float* a_gsp = nullptr;      // [N]
    float* a_rcr = nullptr;      // [N]
    ace::Workspace ws;
    // last call
    int last_T = -1;
    ace_skip_ctl last_ctl{0, 0.f};
    cudaStream_t last_stream = nullptr;
    bool last_has_logits = false;
    // stage timing (ace_layer_set_profiling)
    bool profiling = false;
    cudaEvent_t ev[10] = {};
    int n_stages = 0;
    int last_launches = 0;       // kernels launched by the last forward / route call
    AceHostGraph hg;             // ace_moe_forward_host
    long long dbg_ready_spin = 0;  // ace_debug_set_wait_budget: 0 = off
};

namespace ace {

// ---- launchers (ace_route.cu) ----
cudaError_t route_init(const ace_layer* L);   // per-layer kernel attributes
// Small batches (T <= 256) fuse RMSNorm into the router and run the whole
// decision + compaction in one block.
bool small_path(int T);
cudaError_t launch_rmsnorm(const ace_layer* L, const void* x, int T, cudaStream_t s);
cudaError_t launch_router(const ace_layer* L, const void* x, int T, bool fuse_norm, cudaStream_t s);
// Runs top-k / gates / decision / threshold / compaction from `logits`.
cudaError_t launch_route(const ace_layer* L, const float* logits, int T, ace_skip_ctl ctl, cudaStream_t s,
                         int n_split = 1);
int route_launch_count(const ace_layer* L, int T, ace_skip_ctl ctl);
// T <= 256: RMSNorm + router + decision + compaction in one launch; with
// x == nullptr the logits are taken from `logits` instead.
cudaError_t launch_route_fused(const ace_layer* L, const void* x, const float* logits, int T, ace_skip_ctl ctl,
                               cudaStream_t s);
cudaError_t launch_debug_exp(const float* x, float* y, int n, cudaStream_t s);

// Caller-provided scratch for the decision-only launch of the fused small-T
// kernel (used by the entry point that allocates nothing).
struct DecideScratch {
    float* gates;        // [T*k]
    float* cval;         // [T*k]
    uint32_t* keys;      // [T*k]
    int32_t* offsets;    // [N+1]
    int32_t* dlist;      // [N]
    int32_t* perm;       // [T*k]
    int32_t* slot_pos;   // [T*k]
    int32_t* meta;       // [kMetaCount], tickets must start at zero
    int32_t* tile_cnt;   // [T/8 + 1], must start at zero
    int* err;            // [1]
};
void set_last_error(const char* msg);   // the thread-local text of ace_last_error_message()
size_t route_decide_smem(int T, int k, int n_exp);
cudaError_t route_decide_attr(int smem_bytes);
cudaError_t launch_route_decide_scratch(const float* logits, int T, int n_exp, int k, const float* a_gsp,
                                        const float* a_rcr, float eps, int m_min, ace_skip_ctl ctl, int32_t* ids,
                                        uint8_t* skip, float* ghat, float* tau_out, const DecideScratch& sc,
                                        cudaStream_t s);

// Launch with programmatic stream serialization (PDL): the kernel may start
// while its predecessor on the stream finishes and must execute
// griddepcontrol.wait before reading the predecessor's results.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Stage-timing event: an external event-record node while the stream is
// being captured (so graph replays record it), a plain record otherwise.
inline cudaError_t record_stage(cudaEvent_t ev, cudaStream_t s) {
    cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
    cudaError_t e = cudaStreamIsCapturing(s, &st);
    if (e != cudaSuccess) return e;
    return st == cudaStreamCaptureStatusActive ? cudaEventRecordWithFlags(ev, s, cudaEventRecordExternal)
                                               : cudaEventRecord(ev, s);
}

// Raise a kernel's dynamic shared-memory limit on the current device to at
// least `bytes`, never lowering it: layers of different shapes (and the
// no-allocation entry point) share the kernels, so a limit set for one must
// not drop below what another, created or launched earlier or on another
// host thread, still needs. Serialised by a process-wide mutex.
cudaError_t raise_smem_limit(const void* kernel, int bytes);
template <typename K>
inline cudaError_t raise_smem_limit(K* kernel, int bytes) {
    return raise_smem_limit(reinterpret_cast<const void*>(kernel), bytes);
}

// Prefer the largest shared-memory carveout (all kernels share one L1/shared split).
template <typename K>
inline cudaError_t prefer_shared(K kernel) {
    return cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                                (int)cudaSharedmemCarveoutMaxShared);
}

// ---- launchers (ace_expert_gemv.cu) ----
// ev (nullable): events recorded before gate/up, before down, before combine, after combine.
cudaError_t gemv_init(const ace_layer* L);
cudaError_t launch_experts_gemv(const ace_layer* L, const void* x, void* out, int T, cudaStream_t s, cudaEvent_t* ev);

constexpr int kNumStages = 7;

// ---- tensor-core expert path (ace_expert_tc.cu) ----
bool tc_supported(const ace_layer* L);
int tc_token_tile(const ace_layer* L, int T, ace_skip_ctl ctl);
bool tc_use_pair(const ace_layer* L, int T, ace_skip_ctl ctl);
cudaError_t tc_init(ace_layer* L);
// Packs W_gate / W_up / W_down into the tiled, pre-swizzled layouts of w_gu and w_down.
cudaError_t tc_pack_weights(ace_layer* L, const void* w_gate, const void* w_up, const void* w_down, cudaStream_t s);
// ev (nullable): recorded after gather, after gate/up, after down, after combine.
// next (nullable, T > 256 only): the following layer of a stack; the combine
// then also writes that layer's RMSNorm of `out` into next->ws.h.
cudaError_t launch_experts_tc(const ace_layer* L, const void* x, void* out, int T, ace_skip_ctl ctl, cudaStream_t s,
                              cudaEvent_t* ev, const ace_layer* next = nullptr);
// Router logits on the tensor cores (T > kTcSmallT): z = (h W_r^T + b) / temp.
// With router_splits(L, T) > 1 it writes raw partial sums [splits, T, N] into
// ws.act_bf16 and the top-k kernel forms the logits.
cudaError_t launch_router_tc(const ace_layer* L, int T, cudaStream_t s);
int router_splits(const ace_layer* L, int T);

}  // namespace ace

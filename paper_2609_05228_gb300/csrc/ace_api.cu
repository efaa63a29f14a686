// ace_api.cu — the C ABI of libace.so (include/ace.h): argument checks,
// layer-owned weights and workspace, and the launch sequence of the forward.
#include <math.h>
#include <stdio.h>
#include <string.h>

#include <map>
#include <mutex>
#include <string>
#include <vector>

#include "ace_internal.h"

namespace {

thread_local std::string g_last_error;

ace_status fail(ace_status st, const std::string& msg) {
    g_last_error = msg;
    return st;
}

ace_status cuda_fail(cudaError_t e, const char* where) {
    std::string m = std::string(where) + ": " + cudaGetErrorName(e) + " (" + cudaGetErrorString(e) + ")";
    return fail(ACE_ERR_CUDA, m);
}

#define ACE_CUDA(call, where)                              \
    do {                                                   \
        cudaError_t e_ = (call);                           \
        if (e_ != cudaSuccess) return cuda_fail(e_, where); \
    } while (0)

template <typename P>
cudaError_t dalloc(P** p, size_t bytes) {
    void* q = nullptr;
    cudaError_t e = cudaMalloc(&q, bytes < 16 ? 16 : bytes);
    *p = static_cast<P*>(q);
    return e;
}

void free_layer(ace_layer* L) {
    if (!L) return;
    void* ptrs[] = {L->router_w, L->router_b, L->w_gate, L->w_up, L->w_gu, L->w_down, L->gamma, L->a_gsp,
                    L->a_rcr, L->ws.h, L->ws.logits, L->ws.ids, L->ws.gates, L->ws.cval, L->ws.keys, L->ws.skip,
                    L->ws.ghat, L->ws.tau, L->ws.chunk_counts, L->ws.offsets, L->ws.dlist, L->ws.perm,
                    L->ws.slot_pos, L->ws.meta, L->ws.act, L->ws.yslot, L->ws.h_perm, L->ws.act_bf16, L->ws.tt_off, L->ws.tt_tab, L->ws.dec_done, L->ws.tile_cnt, L->ws.sel_hist, L->ws.sel_cand, L->ws.err, L->ws.x_stage, L->ws.out_stage};
    for (void* p : ptrs)
        if (p) cudaFree(p);
    for (cudaEvent_t e : L->ev)
        if (e) cudaEventDestroy(e);
    if (L->hg.exec) cudaGraphExecDestroy(L->hg.exec);
    if (L->hg.own) cudaStreamDestroy(L->hg.own);
    if (L->hg.err_host) cudaFreeHost(L->hg.err_host);
    delete L;
}

// Device-accessible address of page-locked host memory (nullptr if `p` is
// not page-locked and mapped).
void* mapped_host_byte(const void* p) {
    cudaPointerAttributes a{};
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    return a.type == cudaMemoryTypeHost ? a.devicePointer : nullptr;
}

// Device address of a page-locked host buffer of `bytes` bytes, or NULL when
// it is pageable or not mapped as one range (its last byte must map to the
// same offset as its first).
void* mapped_host(const void* p, size_t bytes = 1) {
    void* m = mapped_host_byte(p);
    if (!m || bytes <= 1) return m;
    void* e = mapped_host_byte(static_cast<const char*>(p) + bytes - 1);
    return e == static_cast<char*>(m) + bytes - 1 ? m : nullptr;
}

// Host <-> device copies for the host-buffer calls. Transfers of a few MB are
// latency-bound on the copy engines (about 17 GB/s for 256 KB against about
// 55 GB/s for SMs reading mapped host memory); larger ones run at the link
// rate either way, so they stay on the copy engines.
constexpr size_t kSmCopyMax = 4u << 20;
constexpr int kMaxErrWords = 16;

__global__ void k_copy16(const uint4* __restrict__ src, uint4* __restrict__ dst, long long n) {
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x)
        dst[i] = src[i];
}

struct ErrWords {
    const int* src[kMaxErrWords];
    int n;
};

__global__ void k_err_words(ErrWords w, int* __restrict__ dst) {
    if ((int)threadIdx.x < w.n) dst[threadIdx.x] = *w.src[threadIdx.x];
}

ace_status copy_async(void* dst, const void* src, void* dst_mapped, const void* src_mapped, size_t bytes,
                      cudaMemcpyKind kind, int num_sms, cudaStream_t s) {
    const void* ks = kind == cudaMemcpyHostToDevice ? src_mapped : src;
    void* kd = kind == cudaMemcpyHostToDevice ? dst : dst_mapped;
    if (ks && kd && bytes <= kSmCopyMax && bytes % 16 == 0 && ((uintptr_t)ks | (uintptr_t)kd) % 16 == 0) {
        const long long n = (long long)(bytes / 16);
        const long long want = (n + 255) / 256;
        const int blocks = (int)(want < 4LL * num_sms ? want : 4LL * num_sms);
        k_copy16<<<blocks > 0 ? blocks : 1, 256, 0, s>>>(static_cast<const uint4*>(ks), static_cast<uint4*>(kd), n);
        ACE_CUDA(cudaGetLastError(), "copy kernel");
    } else {
        ACE_CUDA(cudaMemcpyAsync(dst, src, bytes, kind, s), "copy");
    }
    return ACE_OK;
}

// Runs copy-in, `body(stream)` (the forward from dev_in to dev_out), copy-out
// and copies of the device error words `errs` into g.err_host, through a
// CUDA graph captured on the first call and replayed while the stream, the
// host buffers, T, the skip control and the profiling switch stay the same;
// then synchronises. The host buffers are looked up on every call: the graph
// is replayed only while both are still page-locked and mapped at the device
// addresses it was captured with (a buffer freed and its address reused, or
// registered again, is captured anew). Pageable host buffers cannot be
// captured and are enqueued directly. Calls on the legacy default stream use a blocking
// stream owned by g (ordered with the default stream).
template <typename Body>
ace_status run_host_graph(AceHostGraph& g, cudaStream_t user, const void* xh, void* oh, void* dev_in,
                          const void* dev_out, size_t bytes, const int* const* errs, int n_err, int num_sms, int T,
                          ace_skip_ctl ctl, bool profiling, Body body) {
    cudaStream_t s = user;
    if (!s) {
        if (!g.own) ACE_CUDA(cudaStreamCreate(&g.own), "create stream");
        s = g.own;
    }
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    ACE_CUDA(cudaStreamIsCapturing(s, &cs), "query capture");
    if (cs != cudaStreamCaptureStatusNone) return fail(ACE_ERR_INVALID_ARG, "host-buffer calls synchronise and cannot be captured");
    if (g.n_err < n_err) {
        if (g.exec) {
            cudaGraphExecDestroy(g.exec);
            g.exec = nullptr;
        }
        if (g.err_host) cudaFreeHost(g.err_host);
        g.err_host = nullptr;
        g.n_err = 0;
        ACE_CUDA(cudaMallocHost(&g.err_host, n_err * sizeof(int)), "allocate pinned error words");
        g.n_err = n_err;
    }
    const void* xh_m = mapped_host(xh, bytes);
    void* oh_m = mapped_host(oh, bytes);
    const bool same = g.exec && xh_m && oh_m && g.stream == s && g.x_host == xh && g.out_host == oh &&
                      g.x_mapped == xh_m && g.out_mapped == oh_m && g.T == T && g.ctl.mode == ctl.mode &&
                      g.ctl.value == ctl.value && g.ctl.fusion == ctl.fusion && g.profiling == profiling;
    if (!same) {
        if (g.exec) {
            cudaGraphExecDestroy(g.exec);
            g.exec = nullptr;
        }
        void* err_m = mapped_host(g.err_host, n_err * sizeof(int));
        auto enqueue = [&](cudaStream_t st) -> ace_status {
            ace_status r = copy_async(dev_in, xh, nullptr, xh_m, bytes, cudaMemcpyHostToDevice, num_sms, st);
            if (r != ACE_OK) return r;
            r = body(st);
            if (r != ACE_OK) return r;
            r = copy_async(oh, dev_out, oh_m, nullptr, bytes, cudaMemcpyDeviceToHost, num_sms, st);
            if (r != ACE_OK) return r;
            if (err_m && n_err <= kMaxErrWords) {
                ErrWords w{};
                for (int i = 0; i < n_err; ++i) w.src[i] = errs[i];
                w.n = n_err;
                k_err_words<<<1, 32, 0, st>>>(w, static_cast<int*>(err_m));
                ACE_CUDA(cudaGetLastError(), "error-word kernel");
            } else {
                for (int i = 0; i < n_err; ++i)
                    ACE_CUDA(cudaMemcpyAsync(g.err_host + i, errs[i], sizeof(int), cudaMemcpyDeviceToHost, st),
                             "copy error word");
            }
            return ACE_OK;
        };
        if (!xh_m || !oh_m) {
            ace_status st = enqueue(s);
            if (st != ACE_OK) return st;
            ACE_CUDA(cudaStreamSynchronize(s), "forward_host: synchronize");
            return ACE_OK;
        }
        ACE_CUDA(cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal), "begin capture");
        ace_status st = enqueue(s);
        cudaGraph_t graph = nullptr;
        const cudaError_t ce = cudaStreamEndCapture(s, &graph);
        if (st != ACE_OK) {
            if (graph) cudaGraphDestroy(graph);
            return st;
        }
        if (ce != cudaSuccess) return cuda_fail(ce, "end capture");
        const cudaError_t ie = cudaGraphInstantiate(&g.exec, graph, 0);
        cudaGraphDestroy(graph);
        if (ie != cudaSuccess) {
            g.exec = nullptr;
            return cuda_fail(ie, "instantiate graph");
        }
        g.stream = s;
        g.x_host = xh;
        g.out_host = oh;
        g.x_mapped = xh_m;
        g.out_mapped = oh_m;
        g.T = T;
        g.ctl = ctl;
        g.profiling = profiling;
    }
    ACE_CUDA(cudaGraphLaunch(g.exec, s), "graph launch");
    ACE_CUDA(cudaStreamSynchronize(s), "forward_host: synchronize");
    return ACE_OK;
}

bool tables_ok(const float* t, int n) {
    for (int i = 0; i < n; ++i)
        if (!(t[i] >= 0.0f) || !isfinite(t[i])) return false;
    return true;
}

ace_status report_error_word(ace_layer* L, int err) {
    if (err) {
        ACE_CUDA(cudaMemset(L->ws.err, 0, sizeof(int)), "clear device error word");
        if (err & ace::kErrTimeout) return fail(ACE_ERR_TIMEOUT, "a bounded device wait ran out");
        if (err & ace::kErrNumeric) return fail(ACE_ERR_NUMERIC, "non-finite router logits were seen");
        if (err & ace::kErrBounds) return fail(ACE_ERR_CUDA, "a device index check failed (debug build)");
    }
    return ACE_OK;
}

// Debug build: the canary words past every array of the layer (a kernel
// that wrote past an array's end shows here; the first one found is named).
ace_status check_canaries(ace_layer* L) {
    unsigned char buf[ace::kCanaryBytes];
    for (const ace::Canary& c : L->canaries) {
        ACE_CUDA(cudaMemcpy(buf, c.at, sizeof(buf), cudaMemcpyDeviceToHost), "read canary");
        for (size_t i = 0; i < sizeof(buf); ++i)
            if (buf[i] != ace::kCanaryByte)
                return fail(ACE_ERR_CUDA, std::string("device memory past the end of ") + c.name + " was overwritten");
    }
    return ACE_OK;
}

ace_status check_device_word(ace_layer* L) {
    int err = 0;
    ACE_CUDA(cudaMemcpy(&err, L->ws.err, sizeof(int), cudaMemcpyDeviceToHost), "read device error word");
    ace_status st = report_error_word(L, err);
    if (st != ACE_OK) return st;
    return check_canaries(L);
}

ace_status check_ctl(ace_skip_ctl ctl) {
    if (ctl.mode == ACE_SKIP_THRESHOLD) {
        if (!(ctl.value >= 0.0f)) return fail(ACE_ERR_INVALID_ARG, "threshold tau must be >= 0 (not NaN)");
    } else if (ctl.mode == ACE_SKIP_RATIO) {
        if (!(ctl.value >= 0.0f && ctl.value <= 1.0f))
            return fail(ACE_ERR_INVALID_ARG, "skip ratio q must be in [0, 1]");
    } else {
        return fail(ACE_ERR_INVALID_ARG, "unknown skip mode");
    }
    if (ctl.fusion < ACE_FUSION_MAX || ctl.fusion > ACE_FUSION_SCORE)
        return fail(ACE_ERR_INVALID_ARG, "unknown fusion rule");
    return ACE_OK;
}

}  // namespace

namespace ace {
void set_last_error(const char* msg) { g_last_error = msg; }

cudaError_t raise_smem_limit(const void* kernel, int bytes) {
    static std::mutex mu;
    static std::map<std::pair<int, const void*>, int> limits;   // (device, kernel) -> limit set
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    int& cur = limits[{dev, kernel}];
    if (bytes <= cur) return cudaSuccess;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess) cur = bytes;
    return e;
}
}  // namespace ace

extern "C" {

const char* ace_status_string(ace_status s) {
    switch (s) {
        case ACE_OK: return "ACE_OK";
        case ACE_ERR_INVALID_ARG: return "ACE_ERR_INVALID_ARG";
        case ACE_ERR_UNSUPPORTED: return "ACE_ERR_UNSUPPORTED";
        case ACE_ERR_OOM: return "ACE_ERR_OOM";
        case ACE_ERR_CUDA: return "ACE_ERR_CUDA";
        case ACE_ERR_TIMEOUT: return "ACE_ERR_TIMEOUT";
        case ACE_ERR_NUMERIC: return "ACE_ERR_NUMERIC";
        case ACE_ERR_STATE: return "ACE_ERR_STATE";
    }
    return "ACE_ERR_UNKNOWN";
}

const char* ace_last_error_message(void) { return g_last_error.c_str(); }

ace_status ace_layer_create(const ace_layer_desc* desc_in, const void* router_w, const float* router_b,
                            const void* w_gate, const void* w_up, const void* w_down, const void* rms_gamma,
                            const float* a_gsp, const float* a_rcr, void* stream, ace_layer** out_layer) {
    if (!desc_in || !out_layer) return fail(ACE_ERR_INVALID_ARG, "desc and out_layer must be non-NULL");
    *out_layer = nullptr;
    ace_layer_desc D = *desc_in;
    if (D.eps <= 0.f) D.eps = 1e-6f;
    if (D.rms_eps <= 0.f) D.rms_eps = 1e-6f;
    if (D.router_temp <= 0.f) D.router_temp = 1.0f;
    if (D.min_active < 1) D.min_active = 1;
    if (D.hidden <= 0 || D.n_experts <= 0 || D.top_k <= 0 || D.ffn <= 0 || D.max_tokens <= 0)
        return fail(ACE_ERR_INVALID_ARG, "hidden, n_experts, top_k, ffn and max_tokens must be positive");
    if (D.top_k > D.n_experts) return fail(ACE_ERR_INVALID_ARG, "top_k > n_experts");
    if (D.min_active > D.top_k) return fail(ACE_ERR_INVALID_ARG, "min_active > top_k");
    if (D.dtype != ACE_BF16 && D.dtype != ACE_F32) return fail(ACE_ERR_INVALID_ARG, "unknown dtype");
    if (D.n_experts > ace::kMaxExperts) return fail(ACE_ERR_UNSUPPORTED, "n_experts > 1024");
    if (D.top_k > ace::kMaxTopK) return fail(ACE_ERR_UNSUPPORTED, "top_k > 16");
    const int mult = D.dtype == ACE_BF16 ? 64 : 4;
    if (D.hidden % mult || D.ffn % mult)
        return fail(ACE_ERR_UNSUPPORTED, D.dtype == ACE_BF16 ? "hidden and ffn must be multiples of 64"
                                                             : "hidden and ffn must be multiples of 4");
    if ((long long)D.max_tokens * D.top_k > (1LL << 30)) return fail(ACE_ERR_UNSUPPORTED, "max_tokens too large");
    // RMSNorm keeps a token row in registers: 16 x 16-byte vectors per lane
    if (D.hidden > (D.dtype == ACE_BF16 ? 4096 : 2048))
        return fail(ACE_ERR_UNSUPPORTED, "hidden must be <= 4096 (bf16) or <= 2048 (f32)");
    if (!router_w || !w_gate || !w_up || !w_down || !rms_gamma || !a_gsp || !a_rcr)
        return fail(ACE_ERR_INVALID_ARG, "weight, gamma and table pointers must be non-NULL");
    if (D.has_router_bias && !router_b) return fail(ACE_ERR_INVALID_ARG, "has_router_bias set but router_b is NULL");
    if (!tables_ok(a_gsp, D.n_experts) || !tables_ok(a_rcr, D.n_experts))
        return fail(ACE_ERR_INVALID_ARG, "GSP/RCR tables must be finite and >= 0");

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    ace_layer* L = new ace_layer();
    L->desc = D;
    L->elem = D.dtype == ACE_BF16 ? 2 : 4;
    cudaGetDevice(&L->device);
    cudaDeviceGetAttribute(&L->num_sms, cudaDevAttrMultiProcessorCount, L->device);
    if (L->num_sms <= 0) L->num_sms = 1;

    const size_t d = D.hidden, n = D.n_experts, k = D.top_k, m = D.ffn, E = L->elem;
    // Buffers read by tensor maps are padded so that every TMA box (up to
    // 256 rows) lies inside the tensor.
    const size_t T = D.max_tokens < 256 ? 256 : D.max_tokens;
    const size_t slots = (size_t)D.max_tokens * k < 256 ? 256 : (size_t)D.max_tokens * k;
    const size_t n_pad = (n + 255) / 256 * 256;
    const int n_chunks = (int)((T + ace::kChunk - 1) / ace::kChunk);
    ace::Workspace& W = L->ws;
    cudaError_t e = cudaSuccess;
#ifdef ACE_DEBUG_CHECKS
    // canary words past the end of every array (checked by the synchronising calls)
#define ACE_CANARY(ptr, bytes)                                                                    \
    do {                                                                                          \
        const size_t nb_ = (bytes) < 16 ? 16 : (bytes);                                          \
        unsigned char* at_ = reinterpret_cast<unsigned char*>(ptr) + nb_;                         \
        e = cudaMemset(at_, ace::kCanaryByte, ace::kCanaryBytes);                                \
        if (e != cudaSuccess) {                                                                   \
            free_layer(L);                                                                        \
            return cuda_fail(e, "canary fill");                                                   \
        }                                                                                         \
        L->canaries.push_back(ace::Canary{#ptr, at_});                                            \
    } while (0)
    constexpr size_t kPad = ace::kCanaryBytes;
#else
#define ACE_CANARY(ptr, bytes) \
    do {                       \
    } while (0)
    constexpr size_t kPad = 0;
#endif
#define ALLOC(ptr, bytes)                                                   \
    do {                                                                    \
        e = dalloc(&(ptr), ((bytes) < 16 ? 16 : (bytes)) + kPad);           \
        if (e != cudaSuccess) {                                             \
            free_layer(L);                                                  \
            cudaGetLastError();                                             \
            return fail(ACE_ERR_OOM, std::string("cudaMalloc failed for ") + #ptr); \
        }                                                                   \
        ACE_CANARY(ptr, bytes);                                             \
    } while (0)
    L->tc = ace::tc_supported(L);
    ALLOC(L->router_w, n_pad * d * E);
    ALLOC(L->router_b, n * sizeof(float));
    if (L->tc) {
        ALLOC(L->w_gu, n * 2 * m * d * E);
    } else {
        ALLOC(L->w_gate, n * m * d * E);
        ALLOC(L->w_up, n * m * d * E);
    }
    ALLOC(L->w_down, n * d * m * E);
    ALLOC(L->gamma, d * E);
    ALLOC(L->a_gsp, n * sizeof(float));
    ALLOC(L->a_rcr, n * sizeof(float));
    ALLOC(W.h, T * d * E);
    ALLOC(W.logits, T * n * sizeof(float));
    ALLOC(W.ids, slots * sizeof(int32_t));
    ALLOC(W.gates, slots * sizeof(float));
    ALLOC(W.cval, slots * sizeof(float));
    ALLOC(W.keys, slots * sizeof(uint32_t));
    ALLOC(W.skip, slots);
    ALLOC(W.ghat, slots * sizeof(float));
    ALLOC(W.tau, sizeof(float));
    ALLOC(W.chunk_counts, (size_t)n_chunks * n * sizeof(int32_t));
    ALLOC(W.offsets, (n + 1) * sizeof(int32_t));
    ALLOC(W.dlist, n * sizeof(int32_t));
    ALLOC(W.perm, slots * sizeof(int32_t));
    ALLOC(W.slot_pos, slots * sizeof(int32_t));
    ALLOC(W.meta, ace::kMetaCount * sizeof(int32_t));
    ALLOC(W.tile_cnt, (T / 8 + 1) * sizeof(int32_t));
    ALLOC(W.sel_hist, (4096 + 1024) * sizeof(int32_t));
    ALLOC(W.sel_cand, slots * sizeof(uint32_t));
    if (L->tc) {
        ALLOC(W.h_perm, slots * d * E);
        ALLOC(W.act_bf16, slots * m * E);
        ALLOC(W.tt_off, (n + 1) * sizeof(int32_t));
        L->tt_cap = (int)(n + slots / 16 + 1);
        ALLOC(W.tt_tab, (size_t)L->tt_cap * sizeof(int4));
        ALLOC(W.dec_done, (n + slots / 16 + 1) * sizeof(int32_t));
    } else {
        ALLOC(W.act, slots * m * sizeof(float));
    }
    // fp32 per-slot expert outputs: every batch on the CUDA-core path, batches
    // of up to 256 tokens on the tensor path (larger ones write bf16 rows over h_perm)
    const size_t yslot_rows = L->tc ? (size_t)(D.max_tokens < 256 ? D.max_tokens : 256) * k : slots;
    ALLOC(W.yslot, yslot_rows * d * sizeof(float));
    ALLOC(W.err, sizeof(int));
    ALLOC(W.x_stage, T * d * E);
    ALLOC(W.out_stage, T * d * E);
#undef ALLOC
#undef ACE_CANARY
#define CK(call, where)                       \
    do {                                      \
        e = (call);                           \
        if (e != cudaSuccess) {               \
            free_layer(L);                    \
            return cuda_fail(e, where);       \
        }                                     \
    } while (0)
    CK(cudaMemsetAsync(L->router_w, 0, n_pad * d * E, s), "zero router_w padding");
    CK(cudaMemcpyAsync(L->router_w, router_w, n * d * E, cudaMemcpyDeviceToDevice, s), "copy router_w");
    if (D.has_router_bias)
        CK(cudaMemcpyAsync(L->router_b, router_b, n * sizeof(float), cudaMemcpyDeviceToDevice, s), "copy router_b");
    else
        CK(cudaMemsetAsync(L->router_b, 0, n * sizeof(float), s), "zero router_b");
    if (L->tc) {
        CK(ace::tc_pack_weights(L, w_gate, w_up, w_down, s), "pack expert weights");
    } else {
        CK(cudaMemcpyAsync(L->w_gate, w_gate, n * m * d * E, cudaMemcpyDeviceToDevice, s), "copy w_gate");
        CK(cudaMemcpyAsync(L->w_up, w_up, n * m * d * E, cudaMemcpyDeviceToDevice, s), "copy w_up");
        CK(cudaMemcpyAsync(L->w_down, w_down, n * d * m * E, cudaMemcpyDeviceToDevice, s), "copy w_down");
    }
    CK(cudaMemcpyAsync(L->gamma, rms_gamma, d * E, cudaMemcpyDeviceToDevice, s), "copy gamma");
    CK(cudaMemcpyAsync(L->a_gsp, a_gsp, n * sizeof(float), cudaMemcpyHostToDevice, s), "copy a_gsp");
    CK(cudaMemcpyAsync(L->a_rcr, a_rcr, n * sizeof(float), cudaMemcpyHostToDevice, s), "copy a_rcr");
    CK(cudaMemsetAsync(W.meta, 0, ace::kMetaCount * sizeof(int32_t), s), "zero meta");
    CK(cudaMemsetAsync(W.tile_cnt, 0, (T / 8 + 1) * sizeof(int32_t), s), "zero tickets");
    CK(cudaMemsetAsync(W.sel_hist, 0, (4096 + 1024) * sizeof(int32_t), s), "zero select histograms");
    CK(cudaMemsetAsync(W.err, 0, sizeof(int), s), "zero error word");
    CK(cudaMemsetAsync(W.offsets, 0, (n + 1) * sizeof(int32_t), s), "zero offsets");
    CK(ace::route_init(L), "route kernel attributes");
    CK(ace::gemv_init(L), "gemv kernel attributes");
    if (L->tc) CK(ace::tc_init(L), "tensor-core expert setup");
    CK(cudaStreamSynchronize(s), "create: synchronize");
#undef CK
    *out_layer = L;
    return ACE_OK;
}

void ace_layer_destroy(ace_layer* layer) {
    if (!layer) return;
    cudaDeviceSynchronize();
    free_layer(layer);
}

ace_status ace_layer_get_desc(const ace_layer* layer, ace_layer_desc* desc) {
    if (!layer || !desc) return fail(ACE_ERR_INVALID_ARG, "NULL argument");
    *desc = layer->desc;
    return ACE_OK;
}

ace_status ace_route_logits(ace_layer* L, const float* logits, int T, ace_skip_ctl ctl, void* stream) {
    if (!L) return fail(ACE_ERR_INVALID_ARG, "layer is NULL");
    if (T < 0 || T > L->desc.max_tokens) return fail(ACE_ERR_INVALID_ARG, "T out of range [0, max_tokens]");
    if (T > 0 && !logits) return fail(ACE_ERR_INVALID_ARG, "logits is NULL");
    ace_status st = check_ctl(ctl);
    if (st != ACE_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    L->last_T = T;
    L->last_ctl = ctl;
    L->last_stream = s;
    L->last_has_logits = false;
    L->last_launches = 0;
    if (T == 0) return ACE_OK;
    ACE_CUDA(ace::launch_route(L, logits, T, ctl, s), "route launch");
    L->last_launches = ace::route_launch_count(L, T, ctl);
    return ACE_OK;
}

}  // extern "C"

namespace {

// One layer's forward. In a stack (T > 256 only): h_ready = the previous
// layer's combine has already written RMSNorm(x) into L->ws.h, so the
// RMSNorm launch is left out; next = the following layer, whose RMSNorm of
// `out` this layer's combine writes into next->ws.h.
ace_status forward_impl(ace_layer* L, const void* x, void* out, int T, ace_skip_ctl ctl, cudaStream_t s,
                        const ace_layer* next, bool h_ready) {
    L->last_T = T;
    L->last_ctl = ctl;
    L->last_stream = s;
    L->last_has_logits = T > 0;
    L->last_launches = 0;
    if (T == 0) return ACE_OK;
    cudaEvent_t* ev = L->profiling ? L->ev : nullptr;
    const bool small = ace::small_path(T);
    if (small) next = nullptr, h_ready = false;
    if (ev) ACE_CUDA(ace::record_stage(ev[0], s), "event record");
    if (!small && !h_ready) ACE_CUDA(ace::launch_rmsnorm(L, x, T, s), "rmsnorm launch");
    if (ev) ACE_CUDA(ace::record_stage(ev[1], s), "event record");
    if (small) {
        // router and routing in one launch (stage "router" holds both)
        ACE_CUDA(ace::launch_route_fused(L, x, L->ws.logits, T, ctl, s), "route launch");
        if (ev) ACE_CUDA(ace::record_stage(ev[2], s), "event record");
    } else {
        if (L->tc)
            ACE_CUDA(ace::launch_router_tc(L, T, s), "router launch");
        else
            ACE_CUDA(ace::launch_router(L, x, T, false, s), "router launch");
        if (ev) ACE_CUDA(ace::record_stage(ev[2], s), "event record");
        // split-K router: the top-k kernel sums the partials into ws.logits
        ACE_CUDA(ace::launch_route(L, L->ws.logits, T, ctl, s, L->tc ? ace::router_splits(L, T) : 1), "route launch");
    }
    if (ev) ACE_CUDA(ace::record_stage(ev[3], s), "event record");
    if (L->tc) {
        ACE_CUDA(ace::launch_experts_tc(L, x, out, T, ctl, s, ev ? ev + 4 : nullptr, next), "expert launch");
    } else {
        if (ev) ACE_CUDA(ace::record_stage(ev[4], s), "event record");   // no gather stage
        ACE_CUDA(ace::launch_experts_gemv(L, x, out, T, s, ev ? ev + 4 : nullptr), "expert launch");
    }
    L->n_stages = ev ? ace::kNumStages : 0;
    L->last_launches = (small ? 1 : (h_ready ? 1 : 2) + ace::route_launch_count(L, T, ctl)) +
                       (L->tc ? (small ? 2 : (ace::tc_use_pair(L, T, ctl) ? 4 : 3)) : 3);
    return ACE_OK;
}

}  // namespace

extern "C" {

ace_status ace_moe_forward(ace_layer* L, const void* x, void* out, int T, ace_skip_ctl ctl, void* stream) {
    if (!L) return fail(ACE_ERR_INVALID_ARG, "layer is NULL");
    if (T < 0 || T > L->desc.max_tokens) return fail(ACE_ERR_INVALID_ARG, "T out of range [0, max_tokens]");
    if (T > 0 && (!x || !out)) return fail(ACE_ERR_INVALID_ARG, "x and out must be non-NULL");
    if (T > 0 && x == out) return fail(ACE_ERR_INVALID_ARG, "out must not alias x");
    ace_status st = check_ctl(ctl);
    if (st != ACE_OK) return st;
    return forward_impl(L, x, out, T, ctl, static_cast<cudaStream_t>(stream), nullptr, false);
}

ace_status ace_stack_create(ace_layer* const* layers, int n_layers, ace_stack** out_stack) {
    if (!out_stack) return fail(ACE_ERR_INVALID_ARG, "out_stack is NULL");
    *out_stack = nullptr;
    if (!layers || n_layers < 1) return fail(ACE_ERR_INVALID_ARG, "need at least one layer");
    int max_tokens = 0, d = 0;
    for (int l = 0; l < n_layers; ++l) {
        const ace_layer* L = layers[l];
        if (!L) return fail(ACE_ERR_INVALID_ARG, "a layer is NULL");
        for (int j = 0; j < l; ++j)
            if (layers[j] == L) return fail(ACE_ERR_INVALID_ARG, "a layer appears twice in the stack");
        if (!L->tc) return fail(ACE_ERR_UNSUPPORTED, "stacks take bf16 layers on the tensor-core path");
        if (!L->desc.add_residual) return fail(ACE_ERR_INVALID_ARG, "stack layers must be created with add_residual");
        if (l == 0) {
            d = L->desc.hidden;
            max_tokens = L->desc.max_tokens;
        } else {
            if (L->desc.hidden != d) return fail(ACE_ERR_INVALID_ARG, "stack layers must share the hidden size");
            if (L->device != layers[0]->device) return fail(ACE_ERR_INVALID_ARG, "stack layers must share a device");
            max_tokens = L->desc.max_tokens < max_tokens ? L->desc.max_tokens : max_tokens;
        }
    }
    ace_stack* st = new ace_stack();
    st->layers.assign(layers, layers + n_layers);
    st->max_tokens = max_tokens;
    st->hidden = d;
    const size_t bytes = (size_t)max_tokens * d * 2;
    int prev = 0;
    cudaGetDevice(&prev);
    cudaSetDevice(layers[0]->device);
    for (int i = 0; i < 2 && n_layers > 1; ++i) {
        if (cudaMalloc(&st->buf[i], bytes ? bytes : 16) != cudaSuccess) {
            for (int j = 0; j < i; ++j) cudaFree(st->buf[j]);
            cudaSetDevice(prev);
            delete st;
            return fail(ACE_ERR_OOM, "stack buffer allocation failed");
        }
    }
    cudaSetDevice(prev);
    *out_stack = st;
    return ACE_OK;
}

void ace_stack_destroy(ace_stack* st) {
    if (!st) return;
    cudaDeviceSynchronize();
    for (void* b : st->buf)
        if (b) cudaFree(b);
    if (st->hg.exec) cudaGraphExecDestroy(st->hg.exec);
    if (st->hg.own) cudaStreamDestroy(st->hg.own);
    if (st->hg.err_host) cudaFreeHost(st->hg.err_host);
    delete st;
}

ace_status ace_stack_forward_host(ace_stack* st, const void* x_host, void* out_host, int T, ace_skip_ctl ctl,
                                  void* stream) {
    if (!st) return fail(ACE_ERR_INVALID_ARG, "stack is NULL");
    if (T < 0 || T > st->max_tokens) return fail(ACE_ERR_INVALID_ARG, "T out of range [0, max_tokens]");
    if (T > 0 && (!x_host || !out_host)) return fail(ACE_ERR_INVALID_ARG, "x_host and out_host must be non-NULL");
    ace_status rc = check_ctl(ctl);
    if (rc != ACE_OK) return rc;
    if (T == 0) return ACE_OK;
    ace_layer* first = st->layers.front();
    ace_layer* last = st->layers.back();
    const size_t bytes = (size_t)T * st->hidden * 2;
    bool profiling = false;
    for (ace_layer* L : st->layers) profiling = profiling || L->profiling;
    const int n = (int)st->layers.size();
    std::vector<const int*> errs(n);
    for (int l = 0; l < n; ++l) errs[l] = st->layers[l]->ws.err;
    rc = run_host_graph(st->hg, static_cast<cudaStream_t>(stream), x_host, out_host, first->ws.x_stage,
                        last->ws.out_stage, bytes, errs.data(), n, first->num_sms, T, ctl, profiling,
                        [&](cudaStream_t s) -> ace_status {
                            return ace_stack_forward(st, first->ws.x_stage, last->ws.out_stage, T, ctl, s);
                        });
    if (rc != ACE_OK) return rc;
    for (int l = 0; l < n; ++l) {
        rc = report_error_word(st->layers[l], st->hg.err_host[l]);
        if (rc != ACE_OK) return rc;
    }
    return ACE_OK;
}

ace_status ace_stack_forward(ace_stack* st, const void* x, void* out, int T, ace_skip_ctl ctl, void* stream) {
    if (!st) return fail(ACE_ERR_INVALID_ARG, "stack is NULL");
    if (T < 0 || T > st->max_tokens) return fail(ACE_ERR_INVALID_ARG, "T out of range [0, max_tokens]");
    if (T > 0 && (!x || !out)) return fail(ACE_ERR_INVALID_ARG, "x and out must be non-NULL");
    if (T > 0 && x == out) return fail(ACE_ERR_INVALID_ARG, "out must not alias x");
    ace_status rc = check_ctl(ctl);
    if (rc != ACE_OK) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int n = (int)st->layers.size();
    for (int l = 0; l < n; ++l) {
        const void* in = l == 0 ? x : st->buf[(l - 1) & 1];
        void* o = l == n - 1 ? out : st->buf[l & 1];
        const ace_layer* next = l + 1 < n ? st->layers[l + 1] : nullptr;
        rc = forward_impl(st->layers[l], in, o, T, ctl, s, next, l > 0);
        if (rc != ACE_OK) return rc;
    }
    return ACE_OK;
}

ace_status ace_moe_forward_host(ace_layer* L, const void* x_host, void* out_host, int T, ace_skip_ctl ctl,
                                void* stream) {
    if (!L) return fail(ACE_ERR_INVALID_ARG, "layer is NULL");
    if (T < 0 || T > L->desc.max_tokens) return fail(ACE_ERR_INVALID_ARG, "T out of range [0, max_tokens]");
    if (T > 0 && (!x_host || !out_host)) return fail(ACE_ERR_INVALID_ARG, "x_host and out_host must be non-NULL");
    ace_status st = check_ctl(ctl);
    if (st != ACE_OK) return st;
    if (T == 0) return ace_moe_forward(L, L->ws.x_stage, L->ws.out_stage, 0, ctl, stream);
    const size_t bytes = (size_t)T * L->desc.hidden * L->elem;
    const int* errs[1] = {L->ws.err};
    st = run_host_graph(L->hg, static_cast<cudaStream_t>(stream), x_host, out_host, L->ws.x_stage, L->ws.out_stage,
                        bytes, errs, 1, L->num_sms, T, ctl, L->profiling, [&](cudaStream_t s) -> ace_status {
                            return forward_impl(L, L->ws.x_stage, L->ws.out_stage, T, ctl, s, nullptr, false);
                        });
    if (st != ACE_OK) return st;
    return report_error_word(L, L->hg.err_host[0]);
}

ace_status ace_layer_sync(ace_layer* L) {
    if (!L) return fail(ACE_ERR_INVALID_ARG, "layer is NULL");
    ACE_CUDA(cudaStreamSynchronize(L->last_stream), "synchronize");
    return check_device_word(L);
}

ace_status ace_last_skip_mask(ace_layer* L, uint8_t* skip, int32_t* ids, float* gates_hat, float* tau,
                              int32_t* retained) {
    if (!L) return fail(ACE_ERR_INVALID_ARG, "layer is NULL");
    if (L->last_T < 0) return fail(ACE_ERR_STATE, "no forward or route call yet");
    ACE_CUDA(cudaStreamSynchronize(L->last_stream), "synchronize");
    ace_status st = check_device_word(L);
    if (st != ACE_OK) return st;
    const size_t slots = (size_t)L->last_T * L->desc.top_k;
    if (L->last_T == 0) {
        if (tau) *tau = L->last_ctl.mode == ACE_SKIP_THRESHOLD ? L->last_ctl.value : 0.f;
        if (retained) *retained = 0;
        return ACE_OK;
    }
    if (skip) ACE_CUDA(cudaMemcpy(skip, L->ws.skip, slots, cudaMemcpyDeviceToHost), "copy skip");
    if (ids) ACE_CUDA(cudaMemcpy(ids, L->ws.ids, slots * 4, cudaMemcpyDeviceToHost), "copy ids");
    if (gates_hat) ACE_CUDA(cudaMemcpy(gates_hat, L->ws.ghat, slots * 4, cudaMemcpyDeviceToHost), "copy ghat");
    if (tau) ACE_CUDA(cudaMemcpy(tau, L->ws.tau, 4, cudaMemcpyDeviceToHost), "copy tau");
    if (retained)
        ACE_CUDA(cudaMemcpy(retained, L->ws.meta + ace::kMetaRetained, 4, cudaMemcpyDeviceToHost), "copy R");
    return ACE_OK;
}

ace_status ace_last_router_logits(ace_layer* L, float* logits) {
    if (!L || !logits) return fail(ACE_ERR_INVALID_ARG, "NULL argument");
    if (L->last_T < 0 || !L->last_has_logits) return fail(ACE_ERR_STATE, "no forward with router logits yet");
    ACE_CUDA(cudaStreamSynchronize(L->last_stream), "synchronize");
    ACE_CUDA(cudaMemcpy(logits, L->ws.logits, (size_t)L->last_T * L->desc.n_experts * 4, cudaMemcpyDeviceToHost),
             "copy logits");
    return ACE_OK;
}

ace_status ace_last_permutation(ace_layer* L, int32_t* offsets, int32_t* perm) {
    if (!L) return fail(ACE_ERR_INVALID_ARG, "layer is NULL");
    if (L->last_T < 0) return fail(ACE_ERR_STATE, "no forward or route call yet");
    ACE_CUDA(cudaStreamSynchronize(L->last_stream), "synchronize");
    const int n = L->desc.n_experts;
    if (L->last_T == 0) {
        if (offsets) memset(offsets, 0, (n + 1) * sizeof(int32_t));
        return ACE_OK;
    }
    std::vector<int32_t> off(n + 1);
    ACE_CUDA(cudaMemcpy(off.data(), L->ws.offsets, (n + 1) * 4, cudaMemcpyDeviceToHost), "copy offsets");
    if (offsets) memcpy(offsets, off.data(), (n + 1) * 4);
    if (perm && off[n] > 0)
        ACE_CUDA(cudaMemcpy(perm, L->ws.perm, (size_t)off[n] * 4, cudaMemcpyDeviceToHost), "copy perm");
    return ACE_OK;
}

ace_status ace_layer_set_profiling(ace_layer* L, int enable) {
    if (!L) return fail(ACE_ERR_INVALID_ARG, "layer is NULL");
    if (enable && !L->ev[0]) {
        for (int i = 0; i <= ace::kNumStages; ++i) ACE_CUDA(cudaEventCreate(&L->ev[i]), "event create");
    }
    L->profiling = enable != 0;
    L->n_stages = 0;
    return ACE_OK;
}

ace_status ace_last_stage_times(ace_layer* L, float* ms, int n_max, int* n_out) {
    if (!L) return fail(ACE_ERR_INVALID_ARG, "layer is NULL");
    if (!L->profiling || L->n_stages == 0) return fail(ACE_ERR_STATE, "no profiled forward yet");
    ACE_CUDA(cudaStreamSynchronize(L->last_stream), "synchronize");
    const int n = L->n_stages < n_max ? L->n_stages : n_max;
    for (int i = 0; i < n; ++i) ACE_CUDA(cudaEventElapsedTime(&ms[i], L->ev[i], L->ev[i + 1]), "elapsed time");
    if (n_out) *n_out = L->n_stages;
    return ACE_OK;
}

ace_status ace_last_launch_count(const ace_layer* L, int* n_kernels) {
    if (!L || !n_kernels) return fail(ACE_ERR_INVALID_ARG, "NULL argument");
    *n_kernels = L->last_launches;
    return ACE_OK;
}

ace_status ace_debug_set_wait_budget(ace_layer* L, long long cycles) {
    if (!L) return fail(ACE_ERR_INVALID_ARG, "layer is NULL");
    if (cycles < 0) return fail(ACE_ERR_INVALID_ARG, "cycles must be >= 0");
    L->dbg_ready_spin = cycles;
    return ACE_OK;
}

int ace_debug_checks_enabled(void) {
#ifdef ACE_DEBUG_CHECKS
    return 1;
#else
    return 0;
#endif
}

ace_status ace_debug_poke_canary(ace_layer* L, int index) {
    if (!L) return fail(ACE_ERR_INVALID_ARG, "layer is NULL");
    if (L->canaries.empty()) return fail(ACE_ERR_UNSUPPORTED, "canary words exist in the debug build only");
    if (index < 0 || index >= (int)L->canaries.size()) return fail(ACE_ERR_INVALID_ARG, "canary index out of range");
    ACE_CUDA(cudaDeviceSynchronize(), "synchronize");
    ACE_CUDA(cudaMemset(L->canaries[index].at + 7, 0x5A, 1), "overwrite canary byte");
    return ACE_OK;
}

ace_status ace_debug_exp32(const float* x, float* y, int n, void* stream) {
    if (n < 0 || (n > 0 && (!x || !y))) return fail(ACE_ERR_INVALID_ARG, "bad arguments");
    if (n == 0) return ACE_OK;
    ACE_CUDA(ace::launch_debug_exp(x, y, n, static_cast<cudaStream_t>(stream)), "exp launch");
    return ACE_OK;
}

}  // extern "C"

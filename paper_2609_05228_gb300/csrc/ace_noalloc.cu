// ace_noalloc.cu — ace_route_decide_noalloc: the routing decision with all
// scratch memory in a fixed device array of this library, for callers that
// cannot allocate device memory.
#include <mutex>
#include <string>

#include "ace_internal.h"

namespace {

// Limits of the entry point (the scratch below is sized for them).
constexpr int kNaMaxTokens = 256;
constexpr int kNaMaxSlots = 4096;     // T * k
constexpr int kNaMaxExperts = 1024;
constexpr int kNaMaxDevices = 64;

// Byte offsets of the scratch regions (each 256-byte aligned).
constexpr size_t align256(size_t x) { return (x + 255) / 256 * 256; }
constexpr size_t kOffGates = 0;
constexpr size_t kOffCval = kOffGates + align256(kNaMaxSlots * 4);
constexpr size_t kOffKeys = kOffCval + align256(kNaMaxSlots * 4);
constexpr size_t kOffPerm = kOffKeys + align256(kNaMaxSlots * 4);
constexpr size_t kOffSlotPos = kOffPerm + align256(kNaMaxSlots * 4);
constexpr size_t kOffOffsets = kOffSlotPos + align256(kNaMaxSlots * 4);
constexpr size_t kOffDlist = kOffOffsets + align256((kNaMaxExperts + 1) * 4);
constexpr size_t kOffCounters = kOffDlist + align256(kNaMaxExperts * 4);
// counters region: meta [kMetaCount] + tile tickets [kNaMaxTokens/8 + 1] + error word
constexpr size_t kCounterInts = ace::kMetaCount + kNaMaxTokens / 8 + 1 + 1;
constexpr size_t kScratchBytes = kOffCounters + align256(kCounterInts * 4);   // about 100 KB

// The scratch. Every GPU that loads this library holds one copy until the
// process exits. Host code must not use this name as a device address; it
// gets the address with cudaGetSymbolAddress (below).
static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

std::mutex g_mu;
void* g_addr[kNaMaxDevices] = {};     // device address of g_noalloc_scratch, per device

ace_status na_fail(ace_status st, const std::string& m) {
    ace::set_last_error(m.c_str());
    return st;
}

// First call on a device (with that device current): look up the scratch's
// device address with cudaGetSymbolAddress. Later calls reuse it.
ace_status setup_device(int dev, void** out) {
    std::lock_guard<std::mutex> lock(g_mu);
    if (dev < 0 || dev >= kNaMaxDevices) return na_fail(ACE_ERR_UNSUPPORTED, "device index out of range");
    if (!g_addr[dev]) {
        void* p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p)
            return na_fail(ACE_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
        g_addr[dev] = p;
    }
    *out = g_addr[dev];
    return ACE_OK;
}

}  // namespace

extern "C" ace_status ace_route_decide_noalloc(const float* logits, int T, int n_experts, int top_k,
                                               const float* a_gsp, const float* a_rcr, float eps, int min_active,
                                               ace_skip_ctl ctl, int32_t* ids, uint8_t* skip, float* gates_hat,
                                               float* tau, void* stream) {
    if (!logits || !a_gsp || !a_rcr || !ids || !skip || !gates_hat || !tau)
        return na_fail(ACE_ERR_INVALID_ARG, "ace_route_decide_noalloc: NULL pointer");
    if (T < 1 || T > kNaMaxTokens)
        return na_fail(ACE_ERR_INVALID_ARG, "ace_route_decide_noalloc: T must be in [1, 256]");
    if (n_experts < 1 || n_experts > kNaMaxExperts)
        return na_fail(ACE_ERR_INVALID_ARG, "ace_route_decide_noalloc: n_experts must be in [1, 1024]");
    if (top_k < 1 || top_k > ace::kMaxTopK || top_k > n_experts)
        return na_fail(ACE_ERR_INVALID_ARG, "ace_route_decide_noalloc: top_k must be in [1, min(16, n_experts)]");
    if ((long long)T * top_k > kNaMaxSlots)
        return na_fail(ACE_ERR_INVALID_ARG, "ace_route_decide_noalloc: T * top_k must be <= 4096");
    if (min_active < 1) min_active = 1;
    if (min_active > top_k) return na_fail(ACE_ERR_INVALID_ARG, "ace_route_decide_noalloc: min_active > top_k");
    if (!(eps > 0.0f)) eps = 1e-6f;
    if (ctl.mode == ACE_SKIP_THRESHOLD) {
        if (!(ctl.value >= 0.0f)) return na_fail(ACE_ERR_INVALID_ARG, "ace_route_decide_noalloc: tau must be >= 0");
    } else if (ctl.mode == ACE_SKIP_RATIO) {
        if (!(ctl.value >= 0.0f && ctl.value <= 1.0f))
            return na_fail(ACE_ERR_INVALID_ARG, "ace_route_decide_noalloc: q must be in [0, 1]");
    } else {
        return na_fail(ACE_ERR_INVALID_ARG, "ace_route_decide_noalloc: unknown skip mode");
    }
    if (ctl.fusion < ACE_FUSION_MAX || ctl.fusion > ACE_FUSION_SCORE)
        return na_fail(ACE_ERR_INVALID_ARG, "ace_route_decide_noalloc: unknown fusion rule");
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return na_fail(ACE_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
    void* base = nullptr;
    ace_status st = setup_device(dev, &base);
    if (st != ACE_OK) return st;
    unsigned char* b = static_cast<unsigned char*>(base);
    ace::DecideScratch sc;
    sc.gates = reinterpret_cast<float*>(b + kOffGates);
    sc.cval = reinterpret_cast<float*>(b + kOffCval);
    sc.keys = reinterpret_cast<uint32_t*>(b + kOffKeys);
    sc.perm = reinterpret_cast<int32_t*>(b + kOffPerm);
    sc.slot_pos = reinterpret_cast<int32_t*>(b + kOffSlotPos);
    sc.offsets = reinterpret_cast<int32_t*>(b + kOffOffsets);
    sc.dlist = reinterpret_cast<int32_t*>(b + kOffDlist);
    sc.meta = reinterpret_cast<int32_t*>(b + kOffCounters);
    sc.tile_cnt = sc.meta + ace::kMetaCount;
    sc.err = sc.tile_cnt + kNaMaxTokens / 8 + 1;
    // shared-memory limit of the decision kernel for the largest accepted shape
    // (only ever raised; a no-op after the first call on the device)
    e = ace::route_decide_attr((int)ace::route_decide_smem(kNaMaxTokens, kNaMaxSlots / kNaMaxTokens, kNaMaxExperts));
    if (e != cudaSuccess) return na_fail(ACE_ERR_CUDA, std::string("kernel attribute: ") + cudaGetErrorString(e));
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // the kernel's tickets must start at zero; the previous call's values remain otherwise
    e = cudaMemsetAsync(sc.meta, 0, kCounterInts * 4, s);
    if (e != cudaSuccess) return na_fail(ACE_ERR_CUDA, std::string("clear counters: ") + cudaGetErrorString(e));
    e = ace::launch_route_decide_scratch(logits, T, n_experts, top_k, a_gsp, a_rcr, eps, min_active, ctl, ids, skip,
                                         gates_hat, tau, sc, s);
    if (e != cudaSuccess) return na_fail(ACE_ERR_CUDA, std::string("launch: ") + cudaGetErrorString(e));
    return ACE_OK;
}


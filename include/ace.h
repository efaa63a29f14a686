/*
 * ace.h — C ABI of libace.so: the ACE MoE-layer forward with token-adaptive
 * expert skipping, on one GB300 GPU (sm_103a).
 *
 * Method: ACE, "Adaptive Calibration-Free Expert Skipping for MoE-based LLMs".
 *   - router top-k and gates:            §3.1 (routed set {(e_i, g_i)}), Algorithm 1
 *   - per-slot skip decision:            §3.1-3.2 Eqs. gsp_contribution, gsp_probability,
 *                                        rcr_contribution, rcr_probability, ace_contribution,
 *                                        ace_candidate_intersection; Algorithm 4
 *   - target skip ratio -> threshold:    App. B.1 (budget-to-threshold mapping)
 *   - expert FFN:                        Eq. swiglu_expert
 *   - sparse output:                     Eq. ace_sparse_output
 *
 * Conventions common to every call
 *   - Pointers are plain device or host pointers as stated per argument. No
 *     call takes ownership of a caller pointer.
 *   - Weight layouts follow nn.Linear ([out_features, in_features]), row
 *     major: the paper's row-vector W_gate in R^{d x m} is w_gate[e] transposed.
 *   - `stream` is a cudaStream_t (a CUstream) passed as void*; NULL is the
 *     legacy default stream. All device work of a call is ordered on it.
 *   - Every call returns an ace_status; on failure ace_last_error_message()
 *     (thread-local) describes it. No call aborts the process.
 *   - Errors found by kernels (non-finite router logits, a bounded device wait
 *     that ran out) are recorded in a per-layer device word and reported by the
 *     next call that synchronises (ace_last_skip_mask, ace_layer_sync).
 *   - One forward may be in flight per layer at a time; calls on different
 *     layers are independent.
 */
#ifndef ACE_H
#define ACE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum ace_status {
    ACE_OK = 0,
    ACE_ERR_INVALID_ARG = 1,   /* bad pointer, size or mode */
    ACE_ERR_UNSUPPORTED = 2,   /* shape outside what the kernels support */
    ACE_ERR_OOM = 3,           /* device allocation failed at create time */
    ACE_ERR_CUDA = 4,          /* a CUDA runtime call failed */
    ACE_ERR_TIMEOUT = 5,       /* a bounded device wait ran out */
    ACE_ERR_NUMERIC = 6,       /* non-finite router logits were seen */
    ACE_ERR_STATE = 7          /* call out of order (e.g. no forward yet) */
} ace_status;

typedef enum ace_dtype { ACE_BF16 = 0, ACE_F32 = 1 } ace_dtype;

typedef enum ace_skip_mode {
    ACE_SKIP_THRESHOLD = 0,    /* value = tau (Algorithm 4 input tau_q) */
    ACE_SKIP_RATIO = 1         /* value = q in [0,1]; tau derived per batch (App. B.1) */
} ace_skip_mode;

typedef struct ace_layer_desc {
    int hidden;          /* d */
    int n_experts;       /* N, 1..1024 */
    int top_k;           /* k, 1..min(N, 16) */
    int ffn;             /* m, expert FFN width */
    int max_tokens;      /* largest T a forward may pass; sizes the workspace */
    int dtype;           /* ace_dtype of x, out, weights and gamma */
    float eps;           /* the paper's epsilon (Eqs. gsp_probability, rcr_probability,
                            Algorithm 4 gate renormalisation); 1e-6 if <= 0 */
    float rms_eps;       /* RMSNorm epsilon; 1e-6 if <= 0 */
    float router_temp;   /* logits are divided by it; 1 if <= 0 */
    int min_active;      /* m_min of Algorithm 4 (1 = only the top-1 safeguard) */
    int has_router_bias; /* router_b is read when non-zero */
    int add_residual;    /* non-zero: out = x + y (the decoder-block residual around
                            the MoE layer), added in fp32 before rounding to dtype */
} ace_layer_desc;

/*
 * Skip rule: the per-slot score c that is compared with tau (a slot of rank
 * > 0 is a skip candidate when c < tau). p_gsp and p_rcr are the two views
 * of Eqs. gsp_probability and rcr_probability, g the routing gate.
 */
typedef enum ace_fusion {
    ACE_FUSION_MAX = 0,    /* c = max(p_gsp, p_rcr): ACE, skip only when both views
                              are low (Eqs. ace_contribution, ace_candidate_intersection) */
    ACE_FUSION_MIN = 1,    /* c = min(p_gsp, p_rcr): skip when either view is low
                              (§4.3, Tab. fusion_ablation "Min") */
    ACE_FUSION_MEAN = 2,   /* c = (p_gsp + p_rcr) * 0.5 (Tab. fusion_ablation "Mean") */
    ACE_FUSION_GSP = 3,    /* c = p_gsp, the GSP view alone (§4.3, Tab. ablation) */
    ACE_FUSION_RCR = 4,    /* c = p_rcr, the RCR view alone (Tab. ablation) */
    ACE_FUSION_SCORE = 5   /* c = g, router-score skipping (§4.1 Baselines, "Score");
                              the tables are not read */
} ace_fusion;

typedef struct ace_skip_ctl {
    int mode;            /* ace_skip_mode */
    float value;         /* tau (>= 0, may be +inf) or q (in [0,1]) */
    int fusion;          /* ace_fusion; 0 (zero-initialised) is the ACE rule */
} ace_skip_ctl;

typedef struct ace_layer ace_layer;   /* opaque */

/*
 * ace_layer_create — build one MoE layer on the current CUDA device.
 *   router_w  [N, d]      device, dtype        router weight rows w_e (§3.2 logit z_e = x.w_e + b_e)
 *   router_b  [N]         device, float32      router bias b_e; read only if has_router_bias
 *   w_gate    [N, m, d]   device, dtype        per-expert W_gate^T
 *   w_up      [N, m, d]   device, dtype        per-expert W_up^T
 *   w_down    [N, d, m]   device, dtype        per-expert W_down^T
 *   rms_gamma [d]         device, dtype        RMSNorm scale gamma (Gamma = Diag(gamma), §3.1)
 *   a_gsp     [N]         host,   float32      GSP table A^GSP (Algorithm 2), finite, >= 0
 *   a_rcr     [N]         host,   float32      RCR table A^RCR (Algorithm 3), finite, >= 0
 * The weights are copied and repacked into layer-owned device memory; the
 * caller may free its buffers once the call returns (it synchronises
 * `stream`). The workspace for max_tokens is allocated here; the forward
 * allocates nothing.
 * Errors: INVALID_ARG for NULL pointers, non-positive sizes, k > N, tables
 * that are negative or non-finite; UNSUPPORTED for d or m not a multiple of
 * 64 (bf16) or 4 (f32), hidden above 4096 (bf16) or 2048 (f32), N > 1024,
 * k > 16; OOM; CUDA.
 */
ace_status ace_layer_create(const ace_layer_desc* desc,
                            const void* router_w, const float* router_b,
                            const void* w_gate, const void* w_up, const void* w_down,
                            const void* rms_gamma,
                            const float* a_gsp, const float* a_rcr,
                            void* stream, ace_layer** out_layer);

/* Frees everything the layer owns. NULL is a no-op. Synchronises the device. */
void ace_layer_destroy(ace_layer* layer);

/*
 * ace_moe_forward — y_t = sum_{i in I_t} g^_i f_{e_i}(x_t) for t < T
 * (Eq. ace_sparse_output), with RMSNorm, router, top-k, the skip decision of
 * Algorithm 4, compaction of the retained slots and the SwiGLU experts all on
 * the GPU. out = y, or x + y when the layer was created with add_residual.
 * The combine sums a token's slot outputs in rank order (fp32 slot rows for
 * T <= 256, bf16 slot rows above), so repeated calls give the same bits.
 *   x    [T, d]  device, dtype     layer input (pre-RMSNorm hidden states)
 *   out  [T, d]  device, dtype     layer output; must not alias x
 *   T    0..max_tokens             T = 0 is a no-op
 * Stream-ordered and asynchronous; allocates nothing; the sequence of
 * launches depends only on (T, ctl.mode), so it can be captured in a CUDA graph.
 * Errors: INVALID_ARG (NULL, T out of range, ratio outside [0,1], negative
 * or NaN tau, unknown fusion), CUDA.
 */
ace_status ace_moe_forward(ace_layer* layer, const void* x, void* out, int T,
                           ace_skip_ctl ctl, void* stream);

/*
 * Stacks of layers (a decoder block's MoE layers in sequence):
 *   x_{l+1} = x_l + MoE_l(x_l),  out = x_L
 * ace_stack_create takes n_layers distinct layers, each created with
 * add_residual, bf16 and on the tensor-core path (d a multiple of 256, m a
 * multiple of 128), sharing d and the device; the stack holds pointers to
 * them (they must outlive it) and two [max_tokens, d] buffers for the
 * intermediate outputs, max_tokens being the smallest of the layers'.
 * ace_stack_forward runs the layers on `stream` with one skip control for
 * all. For T > 256 each layer's combine also computes the next layer's
 * RMSNorm from the rounded output it writes, so the next layer starts at its
 * router (one kernel and one read of the [T, d] activations fewer per layer);
 * the result is bit-identical to chaining ace_moe_forward calls. After the
 * call, each layer's ace_last_* functions describe its own part.
 * Errors: INVALID_ARG (NULL, duplicates, mismatched layers, T out of range,
 * aliasing, bad control), UNSUPPORTED (a layer not on the tensor-core
 * path), OOM, CUDA.
 */
typedef struct ace_stack ace_stack;   /* opaque */
ace_status ace_stack_create(ace_layer* const* layers, int n_layers, ace_stack** out_stack);
ace_status ace_stack_forward(ace_stack* stack, const void* x, void* out, int T, ace_skip_ctl ctl, void* stream);
/* The same from HOST buffers x_host, out_host [T, d] bf16: one copy in, the
 * stack, one copy out; synchronises `stream` and reports the layers' device
 * error words. */
ace_status ace_stack_forward_host(ace_stack* stack, const void* x_host, void* out_host, int T, ace_skip_ctl ctl,
                                  void* stream);
/* Frees the stack's buffers (not the layers). NULL is a no-op. Synchronises the device. */
void ace_stack_destroy(ace_stack* stack);

/*
 * ace_moe_forward_host — the same forward from HOST buffers: copies x to a
 * layer-owned device buffer, runs ace_moe_forward, copies the result back
 * and synchronises `stream` before returning.
 *   x_host   [T, d] host, dtype
 *   out_host [T, d] host, dtype
 * With page-locked (pinned) host buffers the copy-in, forward and copy-out
 * are captured once as a CUDA graph and replayed while the stream, the host
 * pointers, T and ctl stay the same (one launch per call). Calls on the
 * legacy default stream (NULL) run on a blocking stream of the layer, which
 * is ordered with it. The call cannot be made while `stream` is being
 * captured (INVALID_ARG).
 */
ace_status ace_moe_forward_host(ace_layer* layer, const void* x_host, void* out_host, int T,
                                ace_skip_ctl ctl, void* stream);

/*
 * ace_route_logits — run only the decision steps (top-k + gates, the
 * Algorithm 4 skip decision, App. B.1 threshold in ratio mode, and the
 * compaction) on caller-supplied float32 router logits, as ace_moe_forward
 * does after its router. Results are read with ace_last_skip_mask and
 * ace_last_permutation.
 *   logits [T, N] device, float32
 */
ace_status ace_route_logits(ace_layer* layer, const float* logits, int T, ace_skip_ctl ctl,
                            void* stream);

/*
 * ace_last_skip_mask — results of the last forward / route call, copied to
 * host buffers the caller owns. Synchronises the stream of that call. Any
 * output pointer may be NULL.
 *   skip      [T, k] uint8    1 = slot skipped; slot i is rank i (logit-descending)
 *   ids       [T, k] int32    routed expert e_i
 *   gates_hat [T, k] float32  renormalised gate g^_i (0 where skipped)
 *   tau       [1]   float32   threshold used (derived per batch in ratio mode)
 *   retained  [1]   int32     R, the number of retained slots
 * Errors: STATE before any forward; NUMERIC / TIMEOUT from the device word.
 */
ace_status ace_last_skip_mask(ace_layer* layer, uint8_t* skip, int32_t* ids, float* gates_hat,
                              float* tau, int32_t* retained);

/* Router logits z [T, N] float32 (host) of the last ace_moe_forward. */
ace_status ace_last_router_logits(ace_layer* layer, float* logits);

/*
 * Retained slots grouped by expert, of the last call (host buffers):
 *   offsets [N+1] int32  exclusive scan of per-expert retained counts
 *   perm    [R]   int32  slot ids t*k+i, sorted by (expert, token)
 */
ace_status ace_last_permutation(ace_layer* layer, int32_t* offsets, int32_t* perm);

/* Waits for the layer's last stream and reports any device-side error word. */
ace_status ace_layer_sync(ace_layer* layer);

/*
 * ace_debug_exp32 — the float32 exp used for the gates (x <= 0), applied
 * element-wise on the device: y[i] = exp(x[i]). Exposed so its bits can be
 * checked against an independent implementation.
 *   x, y [n] device float32
 */
ace_status ace_debug_exp32(const float* x, float* y, int n, void* stream);

/*
 * ace_debug_set_wait_budget — test hook for the bounded device waits (the
 * paper has no counterpart). With cycles > 0, the decode expert kernel
 * (batches of at most 256 tokens on the tensor-core path) waits for a token
 * tile's gate/up results with a target that is never reached and gives up
 * after `cycles` SM clock cycles: it sets the layer's error word, lets the
 * copies it has issued land, frees its tensor memory and returns, and the
 * next synchronising call reports ACE_ERR_TIMEOUT. The kernel's other waits
 * keep their normal bound (about 2 s), so such a forward takes a few seconds
 * and its output is not valid. cycles = 0 restores normal operation. Only
 * forwards launched (or graphs captured) while it is set are affected.
 */
ace_status ace_debug_set_wait_budget(ace_layer* layer, long long cycles);

/*
 * Debug build (the paper has no counterpart). libace_debug.so is the same
 * library compiled with ACE_DEBUG_CHECKS:
 *   - the routing, compaction, gather and combine kernels check every index
 *     they compute (expert ids, permutation rows, tile-table entries, slot
 *     rows) before using it; a failed check sets the layer's error word and
 *     the access is skipped, and the next synchronising call (ace_layer_sync,
 *     ace_last_*) returns ACE_ERR_CUDA;
 *   - every device array of a layer is allocated with 256 extra bytes of a
 *     known pattern (canary words), which the synchronising calls compare;
 *     a difference returns ACE_ERR_CUDA naming the array.
 * It is a stand-in for a memory checker on the hand-indexed kernels; the
 * release library compiles the checks away.
 *
 * ace_debug_checks_enabled returns 1 for the debug build, else 0.
 * ace_debug_poke_canary (test hook) overwrites one byte of the canary words
 * of the layer's array number `index` (allocation order), as a kernel that
 * wrote past that array would; ACE_ERR_UNSUPPORTED in the release build,
 * ACE_ERR_INVALID_ARG for an index out of range. It synchronises the device.
 */
int ace_debug_checks_enabled(void);
ace_status ace_debug_poke_canary(ace_layer* layer, int index);

/*
 * Stage timing (instrumentation; the paper has no counterpart). When enabled,
 * each ace_moe_forward records CUDA events on its stream around its stages:
 *   0 RMSNorm (T > 256), 1 router logits (T <= 256: the whole fused
 *   routing), 2 top-k + decision + threshold + compaction (T > 256),
 *   3 token-row gather, 4 expert gate/up, 5 expert down, 6 combine.
 * ace_last_stage_times synchronises the last stream and writes up to n_max
 * stage durations in milliseconds (host float32) of the last forward; it
 * returns the stage count in *n_out. A forward captured into a CUDA graph
 * with timing enabled records external event nodes, so every replay of the
 * graph updates the times. Stage 3 (gather) is empty for the fp32 layer.
 */
ace_status ace_layer_set_profiling(ace_layer* layer, int enable);
ace_status ace_last_stage_times(ace_layer* layer, float* ms, int n_max, int* n_out);

/* Number of kernels the last forward / route call launched (instrumentation). */
ace_status ace_last_launch_count(const ace_layer* layer, int* n_kernels);

/*
 * ace_route_decide_noalloc — the routing decision of ace_route_logits
 * (top-k, gates, Algorithm 4 skip decision, per-batch threshold in ratio
 * mode) without a layer and without allocating any device memory. The paper
 * has no counterpart; this is a deployment variant.
 *
 * For callers that cannot allocate device memory: a serving runtime that owns
 * every byte of the GPU through its own pool and forbids cudaMalloc after
 * start-up, code that runs while another component holds the allocator, or a
 * plugin host that hands in pre-allocated buffers only. The caller supplies
 * inputs and outputs; the intermediate values (gates, scores, candidate
 * keys, the compaction and the kernel's tickets) live in one fixed device
 * array inside this library (about 100 KB, 256-byte aligned). Every GPU that
 * loads the library holds that array until the process exits.
 *   logits    [T, N] device float32     router logits
 *   a_gsp     [N]    device float32     GSP table (finite, >= 0)
 *   a_rcr     [N]    device float32     RCR table (finite, >= 0)
 *   eps       the paper's epsilon (1e-6 if <= 0); min_active = m_min (>= 1)
 *   ids       [T, k] device int32 out   routed expert of slot i (rank order)
 *   skip      [T, k] device uint8 out   1 = skipped
 *   gates_hat [T, k] device float32 out renormalised gate, 0 where skipped
 *   tau       [1]    device float32 out threshold used
 * Limits: 1 <= T <= 256, 1 <= N <= 1024, 1 <= k <= min(16, N), T*k <= 4096;
 * larger sizes return ACE_ERR_INVALID_ARG with a message and launch nothing.
 * The results are bit-identical to ace_route_logits on the same inputs.
 * The first call on a device (with that device current) looks up the array's
 * device address; make that first call before any stream capture. All calls
 * on a device share that device's one array, and it keeps the last call's
 * contents (the kernel's counters are cleared at the start of every call):
 * calls on one device that overlap on the GPU (on different streams, or from
 * different host threads) race. Calls on different devices use different
 * copies of the array and do not. The decision kernel's shared-memory limit
 * is only ever raised, by this call and by ace_layer_create alike, so a
 * layer created on another host thread cannot make this launch fail.
 * Asynchronous on `stream`; errors found by the kernel (NaN logits) are not
 * reported by this entry point.
 */
ace_status ace_route_decide_noalloc(const float* logits, int T, int n_experts, int top_k,
                                    const float* a_gsp, const float* a_rcr, float eps, int min_active,
                                    ace_skip_ctl ctl, int32_t* ids, uint8_t* skip, float* gates_hat,
                                    float* tau, void* stream);

/*
 * ace_offline_tables_device — the offline GSP and RCR tables (Algorithms 2
 * and 3) computed on the GPU from bf16 weights already in device memory, in
 * the layouts ace_layer_create takes. Needs no layer.
 *   GSP: a_up = ||U||_F ||G W_down||_F, a_gate = ||G||_F ||U W_down||_F with
 *        G = Gamma W_gate, U = Gamma W_up; a~ = sqrt(a_up a_gate);
 *        A^GSP = a~ / (mean a~ + eps)  (Eqs. gsp_up_path, gsp_gate_path,
 *        gsp_geometric_mean, gsp_layer_normalization). The two d x d x m
 *        products per expert run on the tensor cores with bf16 operands
 *        exactly as stored and fp32 accumulation; Gamma is applied in fp64
 *        to the row sums of squares.
 *   RCR: centred router rows, prototype q_e = w~_e / (RMS(w~_e) + eps),
 *        a~ = ||f_e(q_e)||_2 / (||q_e||_2 + eps), A^RCR = a~ / (mean a~ + eps)
 *        (Eqs. rcr_centered_router, rcr_direction_prototype,
 *        rcr_raw_amplification, rcr_layer_normalization); q_e is scaled by
 *        gamma first when rcr_apply_gamma != 0. fp32 FMA on the CUDA cores.
 *   d, N, m        hidden size (multiple of 256, <= 16384), experts (1..1024),
 *                  FFN width (multiple of 64)
 *   gamma [d], router_w [N, d], w_gate / w_up [N, m, d], w_down [N, d, m]
 *                  device, bf16
 *   eps            the paper's epsilon (>= 0)
 *   tile_budget    device bytes for the repacked weight tiles (3 d m 2 bytes
 *                  per expert; experts are processed in chunks that fit, at
 *                  least one at a time); 0 = 1.5 GiB
 *   gsp_out, rcr_out [N] host float32, written on success
 * Allocates its device scratch (the tiles plus O(N d) bytes) for the call
 * and frees it before returning; synchronises `stream`. Sums are taken in a
 * fixed order, so the result is the same bits on every run and for every
 * tile_budget.
 * Errors: INVALID_ARG (NULL, non-positive size, eps < 0), UNSUPPORTED (shape),
 * OOM, CUDA, TIMEOUT (a bounded device wait ran out).
 */
ace_status ace_offline_tables_device(int d, int N, int m, const void* gamma, const void* router_w,
                                     const void* w_gate, const void* w_up, const void* w_down, double eps,
                                     int rcr_apply_gamma, size_t tile_budget, float* gsp_out, float* rcr_out,
                                     void* stream);

/* Fills *desc with the layer's descriptor (after defaults were applied). */
ace_status ace_layer_get_desc(const ace_layer* layer, ace_layer_desc* desc);

const char* ace_status_string(ace_status status);
const char* ace_last_error_message(void);

#ifdef __cplusplus
}
#endif

#endif /* ACE_H */

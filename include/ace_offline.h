/* ace_offline.h — offline GSP / RCR expert tables (host CPU, no CUDA).
 *
 * libace_offline.so computes the two per-expert tables the ACE layer takes at
 * ace_layer_create(), once per layer, from the frozen weights alone:
 *   GSP (Algorithm 2; Eqs. gsp_up_path, gsp_gate_path, gsp_geometric_mean,
 *   gsp_layer_normalization): with G = Gamma W_gate and U = Gamma W_up,
 *     a_up = ||U||_F ||G W_down||_F,  a_gate = ||G||_F ||U W_down||_F,
 *     a~_e = sqrt(a_up a_gate),  A^GSP(e) = a~_e / (mean_j a~_j + eps).
 *     ||G W||_F^2 is taken as <G^T G, W W^T>_F (m x m Gram matrices).
 *   RCR (Algorithm 3; Eqs. rcr_centered_router, rcr_direction_prototype,
 *   rcr_raw_amplification, rcr_layer_normalization): centred router rows
 *     w~_e, prototype q_e = w~_e / (RMS(w~_e) + eps) (rho = 1),
 *     a~_e = ||f_e(q_e)||_2 / (||q_e||_2 + eps),  A^RCR(e) = a~_e / (mean a~ + eps),
 *     f_e(q) = (SiLU(q W_gate) * (q W_up)) W_down; with rcr_apply_gamma != 0
 *     q is scaled by gamma first.
 * All arithmetic is fp64; the outputs are rounded to fp32. The result does not
 * depend on the number of threads (each expert is summed in a fixed order by
 * one thread).
 */
#ifndef ACE_OFFLINE_H
#define ACE_OFFLINE_H

#include "ace.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Tables for one layer.
 *   d, N, m      hidden size, experts, expert FFN width (all > 0)
 *   dtype        ACE_BF16 (inputs are bf16 bit patterns, uint16) or ACE_F32
 *   gamma        [d] host, RMSNorm gain
 *   router_w     [N, d] host
 *   w_gate, w_up [N, m, d] host (nn.Linear layout)
 *   w_down       [N, d, m] host
 *   eps          the paper's epsilon
 *   n_threads    worker threads (<= 0: the hardware concurrency)
 *   gsp_out, rcr_out  [N] host fp32, written on success
 * Returns ACE_OK, or ACE_ERR_INVALID_ARG for a NULL pointer or a
 * non-positive size (nothing is written then). Host memory only; the caller
 * owns every buffer. */
ace_status ace_offline_tables(int d, int N, int m, ace_dtype dtype, const void* gamma, const void* router_w,
                              const void* w_gate, const void* w_up, const void* w_down, double eps,
                              int rcr_apply_gamma, int n_threads, float* gsp_out, float* rcr_out);

#ifdef __cplusplus
}
#endif

#endif /* ACE_OFFLINE_H */

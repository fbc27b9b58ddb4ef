/*
 * slimwise_moe.h -- C ABI of the GB300 (sm_103a) pruned-pool batched-decode
 * MoE layer.
 *
 * The layer is the decode-phase MoE block of SlimWise (arXiv 2609.34117):
 * decode runs over a retained expert set K' of m' experts out of m, selected
 * by masking the router (Sec. 3.1, Eq. 2); the top-k (k unchanged by pruning,
 * Sec. 2.3) gates are renormalised over the k selected experts alone
 * (Sec. 3.1); each step streams only the weights of the union of experts
 * selected across the batch (Sec. 2.1, Eq. 1).  For every token t:
 *
 *   z[t,e]   = x_t . Wr[e]                          e in K'
 *   S_t      = top-k of z[t, K'] (logit desc, id asc on ties)
 *   g[t,j]   = exp(z_j - z_1) / sum_{j' in S_t} exp(z_j' - z_1)
 *   y_e(x)   = W_down[e] (SiLU(W_gate[e] x) * (W_up[e] x))
 *   out[t]   = sum_{j=0..k-1} g[t,j] y_{S_t[j]}(x_t)
 *
 * Conventions shared by every entry point
 *   - All array arguments are DEVICE pointers owned by the caller; the
 *     library never allocates, frees or retains them after returning.
 *   - Work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *     stream) and the call returns without synchronising.  Calls that share a
 *     workspace must be ordered (same stream, or synchronised): the workspace
 *     holds the routing state and the intermediate activations of one call.
 *   - Errors are returned as a slimwise_status value; nothing is enqueued
 *     when a host-side check fails.  A device-side wait that timed out is
 *     reported by slimwise_moe_device_status().
 *   - Layouts are row-major; bf16 is IEEE bfloat16 stored in 16 bits.
 *   - Every pointer must be 16-byte aligned.
 *   - Supported shapes: H % 128 == 0, I % 64 == 0, 1 <= E <= 1024,
 *     1 <= top_k <= min(32, m'), B >= 0 (B == 0 is a no-op).
 */
#ifndef SLIMWISE_MOE_H_
#define SLIMWISE_MOE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum slimwise_status {
  SLIMWISE_OK = 0,
  SLIMWISE_ERR_INVALID_ARG = 1,       /* null pointer, k / m' / B out of range */
  SLIMWISE_ERR_UNSUPPORTED_SHAPE = 2, /* H, I, E or alignment not supported     */
  SLIMWISE_ERR_WORKSPACE = 3,         /* workspace smaller than required        */
  SLIMWISE_ERR_CUDA = 4,              /* a CUDA runtime call or launch failed   */
  SLIMWISE_ERR_DEVICE = 5             /* a kernel reported a timeout / bad input */
} slimwise_status;

/* Device-side error bits reported by slimwise_moe_device_status(). */
#define SLIMWISE_DEVERR_PIPELINE_TIMEOUT 0x1   /* an mbarrier wait gave up        */
#define SLIMWISE_DEVERR_DEPENDENCY_TIMEOUT 0x2 /* a down item's wait for its gate/up tiles gave up */
#define SLIMWISE_DEVERR_DUPLICATE_RETAINED 0x4 /* retained_idx has a repeated id  */
#define SLIMWISE_DEVERR_BAD_RETAINED 0x8       /* retained_idx has an id outside [0,E) */
#define SLIMWISE_DEVERR_BAD_TOPK 0x10          /* a given top-k id outside [0,E)  */
#define SLIMWISE_DEVERR_TMEM_PAIR 0x20         /* the two CTAs of an FFN pair hold different tensor memory */

/* Problem shape.  Supported: 0 <= B <= 2^20; H a multiple of 128 in
 * [128, 32768]; I a multiple of 64 in [64, 65536]; 1 <= E <= 1024.  Others
 * return SLIMWISE_ERR_UNSUPPORTED_SHAPE (B out of range: INVALID_ARG). */
typedef struct slimwise_moe_shape {
  int32_t num_tokens;  /* B: decode batch (tokens)           */
  int32_t hidden;      /* H: model width                     */
  int32_t num_experts; /* E: routed experts in the full pool */
  int32_t inter;       /* I: expert intermediate width       */
} slimwise_moe_shape;

/* Human-readable name of a status code (static storage). */
const char *slimwise_status_string(int status);

/*
 * Bytes of device workspace a call with this shape and top_k needs
 * (routing state, grouped activations, expert outputs, counters).
 * Returns SLIMWISE_OK and writes *bytes, or an error for an unsupported
 * shape.  The workspace needs no initialisation and may be reused by
 * consecutive calls on one stream.
 */
int slimwise_moe_workspace_size(const slimwise_moe_shape *shape, int32_t top_k,
                                size_t *bytes);

/*
 * The decode MoE layer over the retained pool K' (Sec. 3.1, Eq. 2).
 *
 *   hidden       bf16 [B, H]     token hidden states
 *   router_w     fp32 [E, H]     router weight of the full pool
 *   retained_idx int32 [m']      ids of K', unique, in [0, E), any order
 *                                (duplicates or out-of-range ids set a
 *                                device error bit; results are then undefined)
 *   n_retained   m', top_k <= m' <= E
 *   w_gate_up    bf16 [E, 2I, H] rows [0, I) = gate, rows [I, 2I) = up
 *   w_down       bf16 [E, H, I]
 *   top_k        k, 1 <= k <= min(32, m')
 *   out          bf16 [B, H]     gate-weighted sum of the k expert outputs
 *   stream       cudaStream_t
 *   workspace    >= slimwise_moe_workspace_size() bytes, 256-byte aligned
 *
 * Only the weights of experts selected by at least one token are read.
 */
int slimwise_moe_decode(const void *hidden, const float *router_w,
                        const int32_t *retained_idx, int32_t n_retained,
                        const void *w_gate_up, const void *w_down,
                        int32_t top_k, void *out, void *stream,
                        const slimwise_moe_shape *shape, void *workspace,
                        size_t workspace_bytes);

/*
 * Full-pool variant: K' = all E experts (the unpruned layer that prefill runs,
 * Sec. 3.1 "masking applied to neither phase").  Arguments as above.
 */
int slimwise_moe_decode_full(const void *hidden, const float *router_w,
                             const void *w_gate_up, const void *w_down,
                             int32_t top_k, void *out, void *stream,
                             const slimwise_moe_shape *shape, void *workspace,
                             size_t workspace_bytes);

/*
 * Launch options for slimwise_moe_decode_ex (all fields may be zero).
 *   ffn_begin / ffn_end  cudaEvent_t recorded on `stream` immediately before
 *                        the expert-FFN kernel and after the combine kernel
 *                        that follows it (NULL: none); used to time the two
 *                        alone.
 *   disable_pdl          1: launch the layer's four kernels with plain stream
 *                        ordering instead of programmatic dependent launch.
 *   grid_ctas            >0: persistent expert-FFN grid size (default: the
 *                        device's SM count).
 *   wait_limit_ns        >0: limit, in ns, of every bounded wait of the
 *                        expert-FFN kernel (default 1 s).  A wait that runs
 *                        out sets SLIMWISE_DEVERR_PIPELINE_TIMEOUT or
 *                        SLIMWISE_DEVERR_DEPENDENCY_TIMEOUT; its CTA then
 *                        drains its copies and MMAs, frees its tensor memory
 *                        and exits, and the output is incomplete.
 *   test_starve_first_down  tests only: 1 makes the first routed down item
 *                        wait for one more gate/up tile than exists, so that
 *                        wait runs out after wait_limit_ns (the timeout path).
 *   ffn_items            form of the expert-FFN work items: 0 or -1 the
 *                        default, 128-row items (256-row ones at token chunks
 *                        of 64-80 rows); 1 CTA-pair items (two 128-row weight
 *                        tiles on the two CTAs of a cluster, one M = 256
 *                        tcgen05 MMA over both) wherever the layer allows
 *                        them (no shared expert, H a multiple of 256, I of
 *                        128).  The outputs agree within the layer's float
 *                        tolerance in every form; pair items measured slower
 *                        on the Qwen-class layer.
 */
typedef struct slimwise_decode_opts {
  void *ffn_begin;
  void *ffn_end;
  int32_t disable_pdl;
  int32_t grid_ctas;
  int64_t wait_limit_ns;
  int32_t test_starve_first_down;
  int32_t ffn_items;
} slimwise_decode_opts;

/* slimwise_moe_decode with launch options; retained_idx NULL = full pool. */
int slimwise_moe_decode_ex(const void *hidden, const float *router_w,
                           const int32_t *retained_idx, int32_t n_retained,
                           const void *w_gate_up, const void *w_down,
                           int32_t top_k, void *out, void *stream,
                           const slimwise_moe_shape *shape, void *workspace,
                           size_t workspace_bytes,
                           const slimwise_decode_opts *opts);

/*
 * Routing only (Sec. 3.1: Eq. 2 mask, top-k, renormalised gates) followed by
 * the grouping of slots by expert, with the results copied out (device
 * buffers; any output may be NULL to skip it):
 *   topk_idx   int32 [B, k]  selected expert ids, selection order
 *   topk_gate  fp32  [B, k]  renormalised gates
 *   counts     int32 [E]     slots routed to each expert
 *   offsets    int32 [E+1]   exclusive prefix sum of counts
 *   union_ids  int32 [E]     selected experts ascending, then -1 padding
 *   union_size int32 [1]     number of distinct selected experts (Eq. 1)
 *   perm       int32 [B*k]   flat slot t*k+j at grouped position p,
 *                            ordered by (expert asc, token asc)
 *   pos        int32 [B*k]   inverse of perm
 * retained_idx NULL = full pool.
 */
int slimwise_moe_route(const void *hidden, const float *router_w,
                       const int32_t *retained_idx, int32_t n_retained,
                       int32_t top_k, void *stream,
                       const slimwise_moe_shape *shape, void *workspace,
                       size_t workspace_bytes, int32_t *topk_idx,
                       float *topk_gate, int32_t *counts, int32_t *offsets,
                       int32_t *union_ids, int32_t *union_size, int32_t *perm,
                       int32_t *pos);

/*
 * Grouping of caller-given selections (the permutation stage alone), e.g. to
 * measure union sizes for uniformly random selections against Eq. 1.
 *   topk_idx  int32 [B, k] device; each row must hold k distinct ids in [0,E)
 * Outputs as in slimwise_moe_route (any may be NULL).  Uses the workspace of
 * shape {B, shape->hidden, E, shape->inter}.
 */
int slimwise_moe_group(const int32_t *topk_idx, int32_t top_k, void *stream,
                       const slimwise_moe_shape *shape, void *workspace,
                       size_t workspace_bytes, int32_t *counts,
                       int32_t *offsets, int32_t *union_ids,
                       int32_t *union_size, int32_t *perm, int32_t *pos);

/*
 * The decode layer with a shared expert (Sec. 3.3): an always-on SwiGLU
 * expert of intermediate width Is under a per-token sigmoid gate, added after
 * the k routed experts.  Qwen3.6's distilled decoder keeps its original
 * shared expert and a second one of the same width under the same gate, i.e.
 * one shared expert of twice the width, which is what this call takes.
 *
 *   out[t] = sum_j g[t,j] E_{idx[t,j]}(x_t) + s_t * SE(x_t)
 *   s_t    = 1 / (1 + exp(-w_shared_gate . x_t)) (fp32; the dot product in
 *            the same summation order as the router logits)
 *
 *   w_shared_gate    fp32 [H]        gate row, 16-byte aligned
 *   w_shared_gate_up bf16 [2Is, H]   rows [0, Is) = gate, [Is, 2Is) = up
 *   w_shared_down    bf16 [H, Is]
 *   inter_shared     Is, a multiple of 64 in [64, 65536]
 *   workspace        >= slimwise_moe_shared_workspace_size() bytes
 * Other arguments as slimwise_moe_decode; retained_idx NULL = full pool.
 * Errors as slimwise_moe_decode; a bad Is or a misaligned shared pointer
 * returns SLIMWISE_ERR_UNSUPPORTED_SHAPE, a NULL one SLIMWISE_ERR_INVALID_ARG.
 */
int slimwise_moe_shared_workspace_size(const slimwise_moe_shape *shape, int32_t top_k,
                                       int32_t inter_shared, size_t *bytes);
int slimwise_moe_decode_shared(const void *hidden, const float *router_w,
                               const int32_t *retained_idx, int32_t n_retained,
                               const void *w_gate_up, const void *w_down,
                               int32_t top_k, const float *w_shared_gate,
                               const void *w_shared_gate_up,
                               const void *w_shared_down, int32_t inter_shared,
                               void *out, void *stream,
                               const slimwise_moe_shape *shape, void *workspace,
                               size_t workspace_bytes);

/* slimwise_moe_decode_shared with the launch options of slimwise_moe_decode_ex. */
int slimwise_moe_decode_shared_ex(const void *hidden, const float *router_w,
                                  const int32_t *retained_idx, int32_t n_retained,
                                  const void *w_gate_up, const void *w_down,
                                  int32_t top_k, const float *w_shared_gate,
                                  const void *w_shared_gate_up,
                                  const void *w_shared_down, int32_t inter_shared,
                                  void *out, void *stream,
                                  const slimwise_moe_shape *shape, void *workspace,
                                  size_t workspace_bytes,
                                  const slimwise_decode_opts *opts);

/*
 * Expert-importance statistics of one calibration batch (Sec. 2.3: routing
 * mass, Expert Activation Norm, REAP; collected with the full pool, App. A).
 * Runs the full-pool layer (its output goes to `out`, bf16 [B, H]) and, for
 * each expert e and each token t that selected it, with gate g and expert
 * output y (before gating), adds to the caller's fp64 [E, 4] device buffer:
 *   stats[e][0] += 1,  stats[e][1] += g,  stats[e][2] += ||y||_2,
 *   stats[e][3] += g * ||y||_2
 * Tokens are taken in order for each expert.  The buffer is caller-owned and
 * accumulates across calls (zero it before the first batch).  Other
 * arguments as slimwise_moe_decode_full; stats must be 8-byte aligned.
 */
int slimwise_moe_expert_stats(const void *hidden, const float *router_w,
                              const void *w_gate_up, const void *w_down,
                              int32_t top_k, double *stats, void *out,
                              void *stream, const slimwise_moe_shape *shape,
                              void *workspace, size_t workspace_bytes);

enum {
  SLIMWISE_CRITERION_MASS = 0, /* score = routing mass stats[e][1]               */
  SLIMWISE_CRITERION_EAN = 1,  /* score = activation norm sum stats[e][2]        */
  SLIMWISE_CRITERION_REAP = 2  /* score = stats[e][3] / stats[e][0] (0 unrouted) */
};

/*
 * Retained set K' from the statistics (Sec. 3.1: rank the layer's experts by
 * an importance criterion, keep the top m'): the n_retained experts of
 * highest score, ties to the lowest id, written ascending to retained_idx
 * (device int32 [n_retained]) -- ready for slimwise_moe_decode or for building
 * the compact checkpoint.  stats: device fp64 [num_experts, 4].  One kernel
 * launch on `stream`; num_experts <= 1024.
 */
int slimwise_moe_select_retained(const double *stats, int32_t num_experts,
                                 int32_t n_retained, int32_t criterion,
                                 int32_t *retained_idx, void *stream);

/*
 * Compact (pruned) checkpoint of one layer (Sec. 3.1: the router mask of
 * Eq. 2 over the full pool and a checkpoint that holds only the retained
 * experts K' are two forms of the same layer; a PD-disaggregated decode
 * instance keeps only the second).  Writes, for the n_retained experts of
 * retained_idx in ascending original id (so that top-k ties in the compact
 * numbering still go to the lowest original id):
 *   w_gate_up_c  bf16 [m', 2I, H]   rows of w_gate_up [E, 2I, H]
 *   w_down_c     bf16 [m', H, I]    rows of w_down [E, H, I]
 *   router_w_c   fp32 [m', H]       rows of router_w [E, H]
 *   ids_c        int32 [m']         original id of compact expert j
 * The compact layer is then run with slimwise_moe_decode_full on shape
 * {B, H, m', I}; its outputs equal the masked pool's bit for bit, and its
 * selections map back through ids_c.
 *   retained_idx  device int32 [n_retained], distinct ids in [0, E), any
 *                 order; 1 <= n_retained <= E.
 *   shape         hidden, num_experts (E) and inter of the full layer
 *                 (num_tokens is not used).
 * All pointers are device pointers owned by the caller, 16-byte aligned
 * (ids_c and retained_idx 4-byte); outputs must not overlap the inputs.  Two
 * kernel launches on `stream`, no host synchronisation.  A repeated or
 * out-of-range id is reported on the device, not by the return code: every
 * entry of ids_c is then -1 and nothing else is written.
 */
int slimwise_moe_compact_layer(const void *w_gate_up, const void *w_down,
                               const float *router_w, const int32_t *retained_idx,
                               int32_t n_retained, const slimwise_moe_shape *shape,
                               void *w_gate_up_c, void *w_down_c, float *router_w_c,
                               int32_t *ids_c, void *stream);

/*
 * slimwise_moe_decode for callers that cannot allocate device memory (an
 * engine that reserved all of its memory up front, a plugin handed only its
 * inputs and outputs): the same layer, with the scratch memory taken from a
 * fixed 16 MiB device array inside this library instead of a caller-given
 * workspace.  The paper has no counterpart; it is a deployment convenience.
 *
 *   Arguments as slimwise_moe_decode, minus workspace / workspace_bytes;
 *   retained_idx NULL = full pool.
 *   Limit: slimwise_moe_workspace_size(shape, top_k) must be <= 16 MiB
 *   (Qwen-class H=2048, E=128, I=768, top-8: B <= 151); larger problems
 *   return SLIMWISE_ERR_WORKSPACE without launching anything.
 *   The array's device address is looked up on the first call made on each
 *   device; make that first call before any stream capture.  A call that
 *   returns SLIMWISE_ERR_CUDA drops the cached address, so after a context
 *   reset (cudaDeviceReset) the next call looks it up again.
 *   All calls share the array: calls whose kernels may overlap on the GPU
 *   (unordered streams) race.  No call allocates or frees memory.
 *   Device-side errors are read with slimwise_moe_noalloc_device_status().
 */
int slimwise_moe_decode_noalloc(const void *hidden, const float *router_w,
                                const int32_t *retained_idx, int32_t n_retained,
                                const void *w_gate_up, const void *w_down,
                                int32_t top_k, void *out, void *stream,
                                const slimwise_moe_shape *shape);

/*
 * The device error bits (SLIMWISE_DEVERR_*) that the last
 * slimwise_moe_decode_noalloc call on the current device left in the
 * library's fixed array, written to *flags after synchronising `stream`.
 * Returns SLIMWISE_OK if none are set, SLIMWISE_ERR_DEVICE otherwise
 * (SLIMWISE_ERR_INVALID_ARG for a NULL flags, SLIMWISE_ERR_CUDA if the read
 * fails).  Like the entry point itself it allocates nothing; the paper has no
 * counterpart.
 */
int slimwise_moe_noalloc_device_status(void *stream, int32_t *flags);

/*
 * Reads (and synchronises `stream` for) the device error bits the last call
 * on this workspace left (SLIMWISE_DEVERR_*), writing them to *flags.
 * Returns SLIMWISE_OK if none are set, SLIMWISE_ERR_DEVICE otherwise.
 */
int slimwise_moe_device_status(const void *workspace, void *stream,
                               int32_t *flags);

#ifdef __cplusplus
}
#endif

#endif /* SLIMWISE_MOE_H_ */

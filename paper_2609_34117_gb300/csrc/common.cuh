// common.cuh -- shared definitions of the sm_103a decode-MoE kernels:
// workspace layout, kernel parameter blocks, and thin inline-PTX wrappers for
// mbarrier, TMA (cp.async.bulk.tensor), tcgen05 (MMA / TMEM) and
// programmatic dependent launch.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "slimwise_moe.h"

namespace slimwise {

// ---------------------------------------------------------------------------
// Tiling constants of the expert-FFN kernel.
// ---------------------------------------------------------------------------
constexpr int kBlockK = 64;          // K elements per pipeline stage (128 B of bf16)
constexpr int kTileRows = 128;       // MMA M: weight rows per work item
constexpr int kGateRows = 64;        // gate rows (and as many up rows) per gate/up item
constexpr int kMaxTokTile = 256;     // MMA N limit: tokens of one expert per item
constexpr int kTokBox = 16;          // token rows per MMA N step
constexpr int kTokBoxSizes = 16;     // token-row TMA boxes of kTokBox * (m + 1) rows, m < 16
constexpr int kATileBytes = kTileRows * kBlockK * 2;   // 16 KiB
constexpr int kMaxExperts = 1024;
constexpr int kMaxTopK = 32;
constexpr int kCombineTile = 128;    // h values per down item (= kTileRows)

// Tokens of one expert handled by one work item (the FFN kernel's largest
// MMA N): a multiple of 16 from 16 to 256; one TMA box of 16 n rows carries
// an item's n16 = n groups of token rows.  Each pipeline stage holds a chunk
// of token rows, so a smaller chunk leaves room for more weight tiles in
// flight.  The chunk covers the mean load of a retained expert (B*k/m'
// selections) plus three standard deviations of a binomial load, and never
// more than twice the mean, rather than the largest possible load (B).  An
// expert with more tokens than a chunk becomes several entries; their items
// are handed out together, so the repeated weight reads come from L2.
__host__ __device__ inline int pow2_at_least(int v) {
  int p = 1;
  while (p < v) p <<= 1;
  return p;
}
__host__ __device__ inline int round16(int v) { return (v + kTokBox - 1) / kTokBox * kTokBox; }
__host__ __device__ inline int token_chunk_for(int B, int k, int m_ret) {
  int most = round16(B);  // an expert is selected at most once per token
  if (most < kTokBox) most = kTokBox;
  if (most > kMaxTokTile) most = kMaxTokTile;
  const float mean = (float)B * (float)k / (float)m_ret;
  const float spread = mean + 3.0f * sqrtf(mean);
  int c = round16((int)ceilf(spread < 2.0f * mean ? spread : 2.0f * mean));
  if (c < kTokBox) c = kTokBox;
  return c < most ? c : most;
}
// Index m of the token box (kTokBox * (m + 1) rows) that covers n16 16-row groups.
__host__ __device__ inline int token_box_for(int n16) { return n16 - 1; }
constexpr int kMinTokChunk = 16;     // smallest token_chunk_for(): bounds the entry count
// Tokens per routing cluster.  One wave of routing CTAs (two per SM) holds
// 38 clusters: above 152 tokens clusters of 4 need two waves, so every pool
// takes 8 tokens per cluster there; above 304 tokens 16, staged as bf16.
inline int route_tokens_per_cluster(int B, int m_ret) {
  (void)m_ret;
  if (B <= 32) return 1;
  if (B <= 64) return 2;
  if (B <= 152) return 4;
  return B <= 304 ? 8 : 16;
}

// Control words at the head of the workspace (int32 each).
enum CtrlWord {
  kCtrlUnionSize = 0,
  kCtrlNumEntries = 1,
  kCtrlItems1 = 2,      // routed gate/up work items
  kCtrlTotalItems = 3,  // all work items (shared and routed, gate/up and down)
  kCtrlWorkCounter = 4, // dynamic scheduler counter
  kCtrlErr = 5,         // SLIMWISE_DEVERR_* bits of the current call
  kCtrlTraceStep = 6,   // step counter of the optional trace ring
  kCtrlWords = 16
};

// Optional timeline trace (compile with -DSLIMWISE_TRACE): %globaltimer
// stamps of each kernel's first CTA, in a ring of kTraceSteps steps that
// follows the control words.  Without the flag nothing is written.
constexpr int kTraceSteps = 16;
enum TraceSlot {
  kTrRouteStart = 0, kTrRouteEnd, kTrGroupStart, kTrGroupEnd,
  kTrFfnStart, kTrFfnFirstData, kTrFfnEnd, kTrSlots = 8
};

// Byte offsets of every workspace region (all 1024-byte aligned).
struct WsLayout {
  size_t ctrl, topk_idx, topk_gate, counts, offsets, union_ids, entries,
      entry_done, perm, pos, xp, act, y, shared_gate, xt, act_s, y_s, total;
  int32_t max_entries;
};

__host__ __device__ inline size_t align_up(size_t v, size_t a) {
  return (v + a - 1) / a * a;
}

// Work entries the workspace has room for: one per selected expert plus one
// per further chunk (the chunk size depends on m', so bounded by the smallest
// chunk), plus the shared expert's chunks of the batch.
__host__ __device__ inline int max_entries_for(int B, int E, int k, int Is) {
  const long long slots = (long long)B * k;
  return E + (int)((slots + kMinTokChunk - 1) / kMinTokChunk) +
         (Is > 0 ? (B + kMinTokChunk - 1) / kMinTokChunk : 0);
}

// Is: intermediate width of the shared expert (0: none).
inline WsLayout make_layout(int B, int H, int E, int I, int k, int Is = 0) {
  WsLayout L;
  size_t o = 0;
  const size_t slots = (size_t)B * k;
  auto take = [&](size_t bytes) {
    size_t r = o;
    o = align_up(o + (bytes ? bytes : 1), 1024);
    return r;
  };
  L.max_entries = max_entries_for(B, E, k, Is);
  L.ctrl = take(kCtrlWords * 4 + kTraceSteps * kTrSlots * 8);
  L.topk_idx = take(slots * 4);
  L.topk_gate = take(slots * 4);
  L.counts = take((size_t)E * 4);
  L.offsets = take((size_t)(E + 1) * 4);
  L.union_ids = take((size_t)E * 4);
  L.entries = take((size_t)L.max_entries * 16);
  L.entry_done = take((size_t)L.max_entries * 4);
  L.perm = take(slots * 4);
  L.pos = take(slots * 4);
  L.xp = take(slots * H * 2);
  L.act = take(slots * I * 2);
  L.y = take(slots * H * 2);
  if (Is > 0) {
    L.shared_gate = take((size_t)B * 4);
    L.xt = take((size_t)B * H * 2);
    L.act_s = take((size_t)B * Is * 2);
    L.y_s = take((size_t)B * H * 2);
  } else {  // no shared expert: no space (these regions are never accessed)
    L.shared_gate = L.xt = L.act_s = L.y_s = o;
  }
  L.total = o;
  return L;
}

// Device view of the workspace.
struct Ws {
  int32_t *ctrl;
  int32_t *topk_idx;
  float *topk_gate;
  int32_t *counts;
  int32_t *offsets;
  int32_t *union_ids;
  int4 *entries;       // {expert, slot_base, n_tokens, 0}
  int32_t *entry_done; // gate/up items finished per entry
  int32_t *perm;
  int32_t *pos;
  __nv_bfloat16 *xp;   // [B*k, H] hidden rows in grouped order
  __nv_bfloat16 *act;  // [B*k, I] SwiGLU activations in grouped order
  __nv_bfloat16 *y;    // [B*k, H] expert outputs in grouped order
  float *shared_gate;  // [B] sigmoid gate of the shared expert
  __nv_bfloat16 *xt;   // [B, H] hidden rows, token order (shared-expert input)
  __nv_bfloat16 *act_s;  // [B, Is] shared-expert activations, token order
  __nv_bfloat16 *y_s;  // [B, H] shared-expert outputs, token order
};

inline Ws make_ws(void *base, const WsLayout &L) {
  char *b = (char *)base;
  Ws w;
  w.ctrl = (int32_t *)(b + L.ctrl);
  w.topk_idx = (int32_t *)(b + L.topk_idx);
  w.topk_gate = (float *)(b + L.topk_gate);
  w.counts = (int32_t *)(b + L.counts);
  w.offsets = (int32_t *)(b + L.offsets);
  w.union_ids = (int32_t *)(b + L.union_ids);
  w.entries = (int4 *)(b + L.entries);
  w.entry_done = (int32_t *)(b + L.entry_done);
  w.perm = (int32_t *)(b + L.perm);
  w.pos = (int32_t *)(b + L.pos);
  w.xp = (__nv_bfloat16 *)(b + L.xp);
  w.act = (__nv_bfloat16 *)(b + L.act);
  w.y = (__nv_bfloat16 *)(b + L.y);
  w.shared_gate = (float *)(b + L.shared_gate);
  w.xt = (__nv_bfloat16 *)(b + L.xt);
  w.act_s = (__nv_bfloat16 *)(b + L.act_s);
  w.y_s = (__nv_bfloat16 *)(b + L.y_s);
  return w;
}

struct Dims {
  int B, H, E, I, k;
  int m_ret;      // retained experts (E for the full pool)
  int tok_chunk;  // max tokens of one expert per work item (multiple of 16, 16..256)
  int Is;         // shared-expert intermediate width (0: no shared expert)
  int S;          // shared-expert work entries: ceil(B / tok_chunk), 0 without one
  int wide;       // 1: a routed work item covers two adjacent 128-row weight tiles
  int pair;       // 1: the same two tiles, one per CTA of a 2-CTA cluster (M = 256 MMA)
};

// Work items per entry: routed gate/up tiles (64 gate + 64 up rows each, or
// twice that for wide items) and down tiles (128 rows of W_down, or 256).
__host__ __device__ inline int item_tiles(const Dims &d) { return (d.wide || d.pair) ? 2 : 1; }
__host__ __device__ inline int gate_up_tiles(const Dims &d) {
  return d.I / (kGateRows * item_tiles(d));
}
__host__ __device__ inline int down_tiles(const Dims &d) {
  return d.H / (kTileRows * item_tiles(d));
}
// Wide items need whole 256-row tiles of both weights and no shared expert
// (its items keep 128 rows, and a stage holds one kind of A tile).  Two
// weight tiles then share each stage's token rows, which halves the token
// rows read per weight byte, but a stage grows by 16 KB and an expert has
// half as many items.  Measured on the Qwen-class layer, they pay at token
// chunks of 64-80 rows with pools of 64 or more experts (the skewed 40-layer
// stack 8 % faster, uniform B = 256 with m' = 64 faster); with larger chunks
// too few stages fit, and with smaller pools too few items remain to balance
// the SMs (B = 128 with m' = 32 was 15 % slower).
constexpr int kWideMinChunk = 64;
constexpr int kWideMaxChunk = 80;
constexpr int kWideMinPool = 64;
// Pair items: a work item's two 128-row weight tiles go to the two CTAs of a
// cluster, which run one M = 256 MMA (tcgen05 cta_group::2) whose N operand,
// the token rows, is split between their shared memories.  Each CTA then
// holds 128 weight rows and half of the token rows per stage: the token rows
// read per weight byte halve, and a stage shrinks, so more of them fit.  On
// the Qwen-class layer they measured slower than 128-row items at every load
// tried (B = 64-512, m' = 32-128: 15-40 %), so a layer uses them only when
// the caller asks (slimwise_decode_opts.ffn_items = 1).

// Kernel launch declarations (defined in their own translation units).
cudaError_t launch_route_topk(const __nv_bfloat16 *hidden, const float *router_w,
                              const int32_t *retained, Dims d, Ws ws, bool pdl,
                              cudaStream_t stream);
// w_shared_gate: fp32 [H] gate row of the shared expert, or NULL (d.Is == 0).
cudaError_t launch_group_gather(const __nv_bfloat16 *hidden, const float *w_shared_gate,
                                Dims d, Ws ws, bool pdl, bool gather, cudaStream_t stream);

struct FfnMaps {
  CUtensorMap w_gu;                 // [E*2I rows, H cols] bf16, box 64 x 64
  CUtensorMap w_down;               // [E*H rows, I cols] bf16, box 64 x 64
  // token rows: box 64 x 16 (m + 1), or 64 x 8 (m + 1) for pair items (each
  // CTA of the pair loads half of an item's rows)
  CUtensorMap xp[kTokBoxSizes];     // [B*k rows, H cols] bf16
  CUtensorMap act[kTokBoxSizes];    // [B*k rows, I cols] bf16
  // shared expert (encoded only when there is one)
  CUtensorMap w_gu_s;               // [2Is rows, H cols] bf16, box 64 x 64
  CUtensorMap w_down_s;             // [H rows, Is cols] bf16, box 64 x 64
  CUtensorMap xt[kTokBoxSizes];     // [B rows, H cols] bf16, hidden in token order
  CUtensorMap act_s[kTokBoxSizes];  // [B rows, Is cols] bf16, token order
};

// timeout_ns: limit of every bounded wait; starve_first_down (tests only):
// the first routed down item waits for a gate/up tile that never exists.
constexpr uint64_t kDefaultWaitLimitNs = 1000000000ull;
// The gate-weighted combine of every (token, 128-column tile), after the
// expert FFN.
cudaError_t launch_combine(Dims d, Ws ws, __nv_bfloat16 *out, bool pdl, cudaStream_t stream);
// retained: the call's retained ids (NULL: the full pool or a compacted one),
// read only to guess which weight tiles to warm in L2.
cudaError_t launch_expert_ffn(const FfnMaps &maps, Dims d, Ws ws,
                              __nv_bfloat16 *out, const int32_t *retained, int grid, bool pdl,
                              cudaStream_t stream, uint64_t timeout_ns = kDefaultWaitLimitNs,
                              int starve_first_down = 0);

// Importance statistics of the last full-pool call in `ws` added to stats
// (fp64 [E, 4]); retained set from statistics (criterion 0 mass, 1 EAN, 2 REAP).
cudaError_t launch_expert_stats(Dims d, Ws ws, double *stats, cudaStream_t stream);
cudaError_t launch_select_retained(const double *stats, int E, int m_prime, int criterion,
                                   int32_t *ids, cudaStream_t stream);

// The compact checkpoint (retained experts' weights and router rows, ascending
// original id); ids_c all -1 on a repeated or out-of-range id.
cudaError_t launch_compact_layer(const void *w_gate_up, const void *w_down, const float *router_w,
                                 const int32_t *retained, int m, int E, int H, int I, int sms,
                                 void *w_gate_up_c, void *w_down_c, float *router_w_c,
                                 int32_t *ids_c, cudaStream_t stream);

#if defined(__CUDACC__)
// ---------------------------------------------------------------------------
// Device helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Trace stamp of the current step (see TraceSlot); a no-op unless built with
// SLIMWISE_TRACE.  `step` is the value of ctrl[kCtrlTraceStep] for this call.
__device__ __forceinline__ void trace_stamp(const Ws &ws, int step, int slot) {
#ifdef SLIMWISE_TRACE
  uint64_t *ring = reinterpret_cast<uint64_t *>(ws.ctrl + kCtrlWords);
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  ring[(step & (kTraceSteps - 1)) * kTrSlots + slot] = t;
#else
  (void)ws; (void)step; (void)slot;
#endif
}

// Programmatic dependent launch.
__device__ __forceinline__ void pdl_wait_primary() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// mbarrier ------------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count)
               : "memory");
}
__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar,
                                                      uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(
                   bar),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: returns false after `timeout_ns` or once *abort is set.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity,
                                                  volatile int *abort,
                                                  uint64_t timeout_ns) {
#pragma unroll 1
  for (int i = 0; i < 256; ++i)
    if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
#pragma unroll 1
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort) return false;
    if (global_timer_ns() - t0 > timeout_ns) return false;
  }
}

// Bounded wait that ignores the abort flag (used to drain after an abort).
__device__ __forceinline__ bool mbar_wait_timeout(uint32_t bar, uint32_t parity,
                                                  uint64_t timeout_ns) {
  const uint64_t t0 = global_timer_ns();
#pragma unroll 1
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (global_timer_ns() - t0 > timeout_ns) return false;
  }
}

// Clusters (CTA pairs of the expert FFN) ------------------------------------
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Address, in the cluster's shared window, of the variable at shared address
// `addr` of this CTA, in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
// Arrive on an mbarrier of another CTA of the cluster (cluster address),
// releasing this thread's earlier memory operations at cluster scope.
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cl_bar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cl_bar)
               : "memory");
}
__device__ __forceinline__ uint32_t ld_shared_cluster(uint32_t cl_addr) {
  uint32_t v;
  asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(cl_addr) : "memory");
  return v;
}
__device__ __forceinline__ void st_shared_cluster(uint32_t cl_addr, int v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(cl_addr), "r"(v) : "memory");
}
// try_wait acquiring at cluster scope: for barriers that another CTA arrives on.
__device__ __forceinline__ bool mbar_try_wait_cluster(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded cluster-scope wait: false after `timeout_ns`, or once *abort is set
// (abort may be NULL: the wait then ignores it).
__device__ __forceinline__ bool mbar_wait_cluster_bounded(uint32_t bar, uint32_t parity,
                                                          volatile int *abort,
                                                          uint64_t timeout_ns) {
#pragma unroll 1
  for (int i = 0; i < 256; ++i)
    if (mbar_try_wait_cluster(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
#pragma unroll 1
  while (true) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    if (abort && *abort) return false;
    if (global_timer_ns() - t0 > timeout_ns) return false;
  }
}
// Every thread of every CTA of the cluster.
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile(
      "barrier.cluster.arrive.release.aligned;\n\t"
      "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// TMA -----------------------------------------------------------------------
__device__ __forceinline__ void tma_prefetch_desc(const void *map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)map) : "memory");
}
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
// 2-D tiled load; x = innermost (element) coordinate, y = row.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void *map,
                                            uint32_t bar, int x, int y,
                                            uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_"
      "tx::bytes.L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"((uint64_t)map), "r"(x), "r"(y), "r"(bar), "l"(policy)
      : "memory");
}
// The same load by the second CTA of a pair: the data lands in this CTA's
// shared memory and completes bytes on the pair leader's mbarrier
// (`cl_bar`, a cluster address).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const void *map,
                                                 uint32_t cl_bar, int x, int y,
                                                 uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::"
      "bytes.L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"((uint64_t)map), "r"(x), "r"(y), "r"(cl_bar), "l"(policy)
      : "memory");
}
// L2 prefetch of one box of a 2-D tensor map (no shared memory, no barrier).
__device__ __forceinline__ void tma_prefetch_2d(const void *map, int x, int y) {
  asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(
                   (uint64_t)map),
               "r"(x), "r"(y)
               : "memory");
}
__device__ __forceinline__ void prefetch_l2(const void *p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_shared() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// tcgen05 -------------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile(
      "tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
          dst_smem),
      "r"(ncols)
      : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::
                   : "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(
                   taddr),
               "r"(ncols)
               : "memory");
}
// The CTA-pair forms (cta_group::2): alloc, relinquish and dealloc are run
// by one warp of each CTA of the pair; every tcgen05 instruction of a kernel
// uses one cta_group.
__device__ __forceinline__ void tmem_alloc_pair(uint32_t dst_smem, uint32_t ncols) {
  asm volatile(
      "tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
      "r"(ncols)
      : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// D[tmem] (+)= A[smem] * B[smem]^T, bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void tc_mma_bf16(uint32_t d_tmem, uint64_t a_desc,
                                            uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(
          d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// M = 256 over the CTA pair (issued by the pair's first CTA): A rows 0-127
// and D lanes 0-127 in that CTA, rows 128-255 in the second; the N operand's
// rows are split in halves, the first half in the first CTA.  The smem
// descriptors address both CTAs' operands at the same offsets.
__device__ __forceinline__ void tc_mma_bf16_pair(uint32_t d_tmem, uint64_t a_desc,
                                                 uint64_t b_desc, uint32_t idesc,
                                                 uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on the mbarrier at shared address `bar` of each CTA in `cta_mask`
// once every previously issued pair MMA of this thread completed.
__device__ __forceinline__ void tc_commit_pair(uint32_t bar, uint16_t cta_mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster."
      "b64 [%0], %1;" ::"r"(bar),
      "h"(cta_mask)
      : "memory");
}
// Arrive on `bar` once every previously issued MMA of this thread completed.
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 "
      "[%0];" ::"r"(bar)
      : "memory");
}
// 32 lanes x 32 bit, 16 consecutive columns per thread.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, "
      "[%16];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]),
        "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]), "=r"(v[9]),
        "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]),
        "=r"(v[15])
      : "r"(taddr)
      : "memory");
}
__device__ __forceinline__ void tmem_ld_wait() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle,
// 8-row core groups 1024 bytes apart (SBO), tile base 1024-byte aligned.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);   // start address
  d |= (uint64_t)1 << 16;                     // LBO (unused for SW128 K-major)
  d |= (uint64_t)(1024 >> 4) << 32;           // SBO
  d |= (uint64_t)1 << 46;                     // descriptor version (sm_100 family)
  d |= (uint64_t)2 << 61;                     // SWIZZLE_128B
  return d;
}

// Instruction descriptor, kind::f16: bf16 x bf16 -> fp32, both K-major.
__device__ __forceinline__ uint32_t idesc_bf16_f32(int M, int N) {
  return (1u << 4)                       // D format: fp32
         | (1u << 7)                     // A format: bf16
         | (1u << 10)                    // B format: bf16
         | ((uint32_t)(N >> 3) << 17)    // N / 8
         | ((uint32_t)(M >> 4) << 24);   // M / 16
}
#endif  // __CUDACC__

}  // namespace slimwise

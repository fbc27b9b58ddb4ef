// expert_ffn.cu -- grouped SwiGLU expert FFN over the selected-expert union,
// and the gate-weighted combine of its outputs (a second, small kernel).
//
// Decode reads the weights of every expert in the union of the batch's
// selections once per step (SlimWise Sec. 2.1, Eq. 1) and each expert sees
// few tokens (Sec. 2.1: about B*k/m per step), so the kernel is a weight
// stream: HBM -> (TMA, 128-byte swizzle) -> shared-memory ring ->
// tcgen05.mma with the weights as the M = 128 operand and the expert's
// tokens as the N operand (16..256, padded to 16) -> TMEM accumulators ->
// epilogue warps.
//
// One persistent CTA per SM (320 threads):
//   warp 0   producer (one thread): takes work items from a global counter,
//            waits for a down item's activations, and issues each stage's
//            copies -- the 128-row weight tile (two 64-row boxes) and the
//            item's token rows (one box, its height the token count rounded
//            up to 16 rows).  Each copy costs the issuing thread about 40 ns
//            (a streaming probe), so a stage takes three copies whatever the
//            number of tokens and the descriptors are chosen once per item;
//            at that count the copy rate no longer bounds the kernel (a
//            second issuing warp for the token box changed nothing).
//   warp 1   MMA issuer (one thread) and TMEM owner; double-buffered
//            accumulators so the epilogue of one item overlaps the next.
//   warps 2-9 two epilogue warpgroups; group g handles the items of
//            accumulator buffer g (every other item).
// Work items, all of gate/up before any of down (so a down item only waits
// for work that has already been handed out):
//   gate/up (entry, i-tile): A = 64 gate rows + the matching 64 up rows of
//            W_gu[e], K = H; epilogue computes act = SiLU(gate) * up (fp32),
//            stores bf16 act in grouped order and counts the tile done.
//   down    (entry, h-tile): A = 128 rows of W_down[e], K = I, B = act of the
//            entry's tokens (after all its gate/up tiles are done); epilogue
//            rounds the fp32 accumulators to bf16 y in grouped order (like
//            act, an intermediate in the activation type: half the bytes
//            for the combine to read, 2-4 us a step faster at B >= 256).
// The combine kernel runs next on the stream (programmatic dependent launch:
// its CTAs become resident beside this grid's last CTAs): one warp per
// (token, 128-column tile) sums g[t,j] y_j in j order and writes bf16.  With
// the whole GPU's warps on it the combine takes a few microseconds after the
// last expert output, where combining inside this kernel left it to the few
// CTAs that finished the last items.
// Every wait is bounded (1 s unless the caller sets another limit): on
// timeout the CTA records an error bit in the workspace, stops taking work,
// drains its own copies and MMAs, frees TMEM and exits.  The 128 threads of an
// epilogue group take each wait's outcome together (a barrier reduction), so
// a wait that completes just as another thread gives up cannot split the
// group between its named barrier and the exit.
#include "common.cuh"

namespace slimwise {

constexpr int kEpiGroups = 2;    // epilogue warpgroups, one per TMEM accumulator
constexpr int kEpiThreads = 128; // threads of one epilogue warpgroup
constexpr int kFfnThreads = 64 + kEpiGroups * kEpiThreads;
constexpr int kItemRing = 4;
constexpr int kXchStride = 17;  // padded row stride (floats) of the exchange buffer
constexpr int kXchBytes = kEpiGroups * kTileRows * kXchStride * 4;

// A pipeline stage: one 64-wide K sub-tile (one 128-byte swizzle atom) of
// the item's weight rows -- 128, or 256 for a wide item -- then tok_chunk
// token rows of the same K range (half of them in each CTA of a pair).
struct FfnSmem {
  int stages;
  int a_bytes;
  int stage_bytes;
  size_t xch_off, bar_off, misc_off, total;
};

__host__ __device__ inline FfnSmem ffn_smem_plan(int tok_chunk, int stages, int wide,
                                                  int pair) {
  FfnSmem p;
  p.stages = stages;
  p.a_bytes = kATileBytes * (wide ? 2 : 1);
  p.stage_bytes = p.a_bytes + (pair ? tok_chunk / 2 : tok_chunk) * kBlockK * 2;
  p.xch_off = (size_t)stages * p.stage_bytes;
  p.bar_off = p.xch_off + kXchBytes;
  // full[S], empty[S], acc_full[2], acc_empty[2], item_full[R], item_empty[R],
  // drain, and for a pair mailbox_full[R], mailbox_empty[R]
  p.misc_off = p.bar_off + 8 * (2 * stages + 4 + 2 * kItemRing + 1 + (pair ? 2 * kItemRing : 0));
  // item ring, tmem base, abort, consumed stages, and for a pair the mailbox[R]
  p.total = p.misc_off + 4 * (kItemRing + 3 + (pair ? kItemRing : 0)) + 1024;
  return p;
}

// TMEM accumulators: one per 128 weight rows of an item, N = tok_chunk
// columns each, in two buffers (the epilogue of one item overlaps the MMAs
// of the next): at most 512 columns, so wide items need tok_chunk <= 128.
__host__ __device__ inline int ffn_acc_cols(const Dims &d) { return (d.wide ? 2 : 1) * d.tok_chunk; }

struct Item {
  int down;      // 0: gate/up, 1: down
  int shared;    // 1: the shared expert (token order), 0: a routed expert
  int entry;
  int tile;
  int expert;
  int slot_base;
  int n;         // tokens
  int n16;       // tokens rounded up to 16, / 16
};

// Work-item ranges of one launch, in the order they are handed out:
//   [shared gate/up: S*t1s][routed gate/up: r1][shared down: S*t2][routed down]
// Every gate/up item precedes every down item; the shared expert's items go
// first in each phase (they depend on no routing and have the widest entries).
struct ItemPlan {
  int r1;           // routed gate/up items
  int t1, t1s, t2;  // tiles per entry: routed gate/up, shared gate/up, down
  int S;            // shared-expert entries (0: none); routed entries follow them
};

template <bool kShared>
__device__ __forceinline__ Item decode_item(int item, const ItemPlan &ip, const Ws &ws) {
  Item it;
  it.shared = 0;
  if constexpr (!kShared) {
    if (item < ip.r1) {
      it.down = 0;
      it.entry = item / ip.t1;
      it.tile = item - it.entry * ip.t1;
    } else {
      const int j = item - ip.r1;
      it.down = 1;
      it.entry = j / ip.t2;
      it.tile = j - it.entry * ip.t2;
    }
  } else {
    const int s1 = ip.S * ip.t1s;
    const int g = s1 + ip.r1;
    const int s2 = ip.S * ip.t2;
    int j, t;
    if (item < s1) {
      it.down = 0; it.shared = 1; j = item; t = ip.t1s;
    } else if (item < g) {
      it.down = 0; j = item - s1; t = ip.t1;
    } else if (item < g + s2) {
      it.down = 1; it.shared = 1; j = item - g; t = ip.t2;
    } else {
      it.down = 1; j = item - g - s2; t = ip.t2;
    }
    const int e = j / t;
    it.tile = j - e * t;
    it.entry = it.shared ? e : ip.S + e;
  }
  const int4 en = __ldcg(&ws.entries[it.entry]);
  it.expert = en.x;
  it.slot_base = en.y;
  it.n = en.z;
  it.n16 = (en.z + 15) >> 4;
  return it;
}

// out[t, h] = sum_j g[t,j] y[pos(t,j), h] in j order (then the shared
// expert's term) for the 128 h of one tile, by one warp: lane l covers
// h = 4l..4l+3 with one 16-byte load per selection (a y tile row is 512
// contiguous bytes), up to 8 loads in flight per lane; lanes j < k hold
// selection j's grouped position and gate.
template <bool kShared>
__device__ __forceinline__ void combine_token(const Ws &ws, const Dims &d,
                                              __nv_bfloat16 *__restrict__ out, int t, int tile,
                                              int lane, int p, float gj, float sg) {
  const __nv_bfloat16 *ytile = ws.y + tile * kCombineTile + 4 * lane;
  float4 acc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
  for (int j0 = 0; j0 < d.k; j0 += 8) {
    uint2 v[8];
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
      const int pj = __shfl_sync(0xFFFFFFFFu, p, (j0 + jj) & 31);
      if (j0 + jj < d.k)
        v[jj] = __ldcg(reinterpret_cast<const uint2 *>(ytile + (size_t)pj * d.H));
    }
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
      const float w = __shfl_sync(0xFFFFFFFFu, gj, (j0 + jj) & 31);
      if (j0 + jj < d.k) {
        acc.x = fmaf(w, __uint_as_float(v[jj].x << 16), acc.x);
        acc.y = fmaf(w, __uint_as_float(v[jj].x & 0xFFFF0000u), acc.y);
        acc.z = fmaf(w, __uint_as_float(v[jj].y << 16), acc.z);
        acc.w = fmaf(w, __uint_as_float(v[jj].y & 0xFFFF0000u), acc.w);
      }
    }
  }
  if constexpr (kShared) {
    // the shared expert's term, after the k routed ones (Sec. 3.3)
    const uint2 vs = __ldcg(reinterpret_cast<const uint2 *>(
        ws.y_s + (size_t)t * d.H + tile * kCombineTile + 4 * lane));
    acc.x = fmaf(sg, __uint_as_float(vs.x << 16), acc.x);
    acc.y = fmaf(sg, __uint_as_float(vs.x & 0xFFFF0000u), acc.y);
    acc.z = fmaf(sg, __uint_as_float(vs.y << 16), acc.z);
    acc.w = fmaf(sg, __uint_as_float(vs.y & 0xFFFF0000u), acc.w);
  }
  const __nv_bfloat162 lo = __floats2bfloat162_rn(acc.x, acc.y);
  const __nv_bfloat162 hi = __floats2bfloat162_rn(acc.z, acc.w);
  *reinterpret_cast<uint2 *>(out + (size_t)t * d.H + tile * kCombineTile + 4 * lane) =
      make_uint2(*reinterpret_cast<const uint32_t *>(&lo),
                 *reinterpret_cast<const uint32_t *>(&hi));
}

// Named barrier of epilogue group g (ids 1.., id 0 is __syncthreads).
__device__ __forceinline__ void epi_bar(int g) {
  asm volatile("bar.sync %0, %1;" ::"r"(1 + g), "n"(kEpiThreads) : "memory");
}

// The same barrier, returning whether `v` holds on every thread of group g.
__device__ __forceinline__ bool epi_all(int g, bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 q, %1, 0;\n\t"
      "bar.red.and.pred p, %2, %3, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)v), "r"(1 + g), "n"(kEpiThreads)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ int ld_acquire(const int *p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void raise_abort(volatile int *abort, Ws &ws, int bit) {
  *abort = 1;
  atomicOr(&ws.ctrl[kCtrlErr], bit);
}

// At most 128 registers a thread (320 threads: 40 K of the SM's 64 K), so
// that a CTA of the dependent combine kernel (256 threads, 72 registers)
// can become resident beside this one.
//
// kPair: the grid is made of 2-CTA clusters.  A routed work item covers two
// adjacent 128-row weight tiles (as a wide item does); CTA r of the pair
// loads tile r and token rows [r N/2, (r + 1) N/2) of the item's N, and the
// pair's first CTA issues one M = 256 MMA per K step over both CTAs' shared
// memory.  Only that CTA's producer takes items from the global counter; it
// hands each one to the second CTA through a mailbox in the second CTA's
// shared memory, so both CTAs work through the same items in the same order.
// The second CTA's copies complete bytes on the first CTA's stage barriers;
// the MMA commits arrive on the stage and accumulator barriers of both CTAs;
// each CTA's epilogue reads its own TMEM lanes (its 128 weight rows) and
// releases the accumulator to the first CTA's MMA issuer.
template <bool kShared, bool kWide, bool kPair>
__global__ void __maxnreg__(128)
    expert_ffn_kernel(const __grid_constant__ FfnMaps maps, Dims d, Ws ws,
                      __nv_bfloat16 *__restrict__ out,
                      const int32_t *__restrict__ retained, int stages,
                      int tmem_cols, int static_first, int early_dependents,
                      uint64_t timeout_ns,
                      int starve_first_down) {
  static_assert(!(kPair && (kShared || kWide)), "pair items are routed 128-row tiles");
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const FfnSmem plan = ffn_smem_plan(d.tok_chunk, stages, d.wide, kPair ? 1 : 0);
  const uint32_t smem_base = smem_u32(smem);
  float *xch = reinterpret_cast<float *>(smem + plan.xch_off);
  const uint32_t bar0 = smem_base + (uint32_t)plan.bar_off;
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (stages + s); };
  auto accf_bar = [&](int b) { return bar0 + 8u * (2 * stages + b); };
  auto acce_bar = [&](int b) { return bar0 + 8u * (2 * stages + 2 + b); };
  auto itf_bar = [&](int r) { return bar0 + 8u * (2 * stages + 4 + r); };
  auto ite_bar = [&](int r) { return bar0 + 8u * (2 * stages + 4 + kItemRing + r); };
  const uint32_t drain_bar = bar0 + 8u * (2 * stages + 4 + 2 * kItemRing);
  // pair mailbox: full barriers live in the second CTA, empty ones in the first
  auto mbf_bar = [&](int r) { return bar0 + 8u * (2 * stages + 5 + 2 * kItemRing + r); };
  auto mbe_bar = [&](int r) { return bar0 + 8u * (2 * stages + 5 + 3 * kItemRing + r); };
  int *misc = reinterpret_cast<int *>(smem + plan.misc_off);
  volatile int *ring = misc;                         // [kItemRing]
  volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(misc + kItemRing);
  volatile int *abort = misc + kItemRing + 1;
  volatile int *consumed = misc + kItemRing + 2;     // stages the MMA finished with
  volatile int *mbox = misc + kItemRing + 3;         // [kItemRing], pair only

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t crank = kPair ? cluster_ctarank() : 0u;  // CTA of the pair
  const bool lead = crank == 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accf_bar(b), 1);
      // a pair's accumulator is released by one thread of each CTA's group
      mbar_init(acce_bar(b), kPair ? 2 : kEpiThreads);
    }
    for (int r = 0; r < kItemRing; ++r) {
      mbar_init(itf_bar(r), 1);
      mbar_init(ite_bar(r), 1 + kEpiGroups * kEpiThreads);
      if constexpr (kPair) {
        mbar_init(mbf_bar(r), 1);
        mbar_init(mbe_bar(r), 1);
      }
    }
    mbar_init(drain_bar, 1);
    *abort = 0;
    *consumed = 0;
    mbar_fence_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&maps.w_gu);
    tma_prefetch_desc(&maps.w_down);
    for (int m = 0; m < kTokBoxSizes && kTokBox * (m + 1) <= d.tok_chunk; ++m) {
      tma_prefetch_desc(&maps.xp[m]);
      tma_prefetch_desc(&maps.act[m]);
      if constexpr (kShared) {
        tma_prefetch_desc(&maps.xt[m]);
        tma_prefetch_desc(&maps.act_s[m]);
      }
    }
    if constexpr (kShared) {
      tma_prefetch_desc(&maps.w_gu_s);
      tma_prefetch_desc(&maps.w_down_s);
    }
  }
  if (warp == 1) {
    if constexpr (kPair) {
      tmem_alloc_pair(smem_u32((const void *)tmem_slot), (uint32_t)tmem_cols);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(smem_u32((const void *)tmem_slot), (uint32_t)tmem_cols);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  __syncthreads();
  // both CTAs' barriers are initialised before either arrives on the other's
  if constexpr (kPair) cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // the pair MMA writes both CTAs' accumulators at the first CTA's address:
  // the second CTA checks that its allocation is the same, else it takes no
  // work (its partner's waits then run out)
  if constexpr (kPair) {
    if (threadIdx.x == 0 && !lead &&
        ld_shared_cluster(mapa_shared(smem_u32((const void *)tmem_slot), 0u)) != tmem_base)
      raise_abort(abort, ws, SLIMWISE_DEVERR_TMEM_PAIR);
  }

  // While the grouping kernel runs (this grid may already be resident), warm
  // L2 with this CTA's likely first work item: the gate/up tile that item
  // number blockIdx.x (for a pair, the cluster's number) has when each
  // retained expert is selected and takes one entry.  The work list runs in
  // ascending expert order, so entry j is then the j-th retained expert
  // (retained ids listed in ascending order), which holds for nearly every
  // pool once B k >= 2 m'.  The guess uses only this call's inputs, so it is
  // as good for a stack of different layers as for one layer called again
  // (guessing from the previous call's work list cost a 10-layer skewed stack
  // 3.8 %).  A wide item warms only its first 64 gate and 64 up rows: all of
  // them would be 152 MB, more than L2 holds; each CTA of a pair warms its
  // own 64 gate and 64 up rows.  Prefetches only, every index bounded, so a
  // wrong guess costs bandwidth, never correctness.
  const int item0 = kPair ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
  if constexpr (!kShared) {
    if (warp == 0 && lane == 0 && d.B * d.k >= 2 * d.m_ret) {
      const int t1g = gate_up_tiles(d);
      const int rows = kGateRows * item_tiles(d);  // gate rows (and up rows) of an item
      const int entry = item0 / t1g;
      if (entry < d.m_ret) {
        const int e = retained ? __ldcg(retained + entry) : entry;
        if (e >= 0 && e < d.E) {
          const int row0 = e * 2 * d.I + (item0 - entry * t1g) * rows + (int)crank * kGateRows;
          for (int kc = 0; kc < d.H / kBlockK; ++kc) {
            tma_prefetch_2d(&maps.w_gu, kc * kBlockK, row0);
            tma_prefetch_2d(&maps.w_gu, kc * kBlockK, row0 + d.I);
          }
        }
      }
    }
  }

  // Everything below reads the grouping kernel's results.
  pdl_wait_primary();
  // Above 64 tokens the combine kernel that follows may become resident now
  // (it waits for this grid to finish): measured 2-4 us faster per step at
  // B = 128-512, 0.5 us slower at B = 64, where the trigger stays at the end
  // of the work.
  if (early_dependents) pdl_launch_dependents();
#ifdef SLIMWISE_TRACE
  const int tr_step = ws.ctrl[kCtrlTraceStep] - 1;
  if (blockIdx.x == 0 && threadIdx.x == 0) trace_stamp(ws, tr_step, kTrFfnStart);
#endif

  const int total = __ldcg(&ws.ctrl[kCtrlTotalItems]);
  const int t1 = gate_up_tiles(d);
  const int t2 = down_tiles(d);
  ItemPlan ip;
  ip.r1 = __ldcg(&ws.ctrl[kCtrlItems1]);
  ip.t1 = t1;
  ip.t1s = kShared ? d.Is / kGateRows : 0;
  ip.t2 = t2;
  ip.S = kShared ? d.S : 0;
  const int nb_cols = ffn_acc_cols(d);  // TMEM columns per accumulator buffer
  constexpr int wmul = kWide ? 2 : 1;   // 128-row halves of a routed item in this CTA
  // 128-row tiles of a routed item (across the pair): its gate/up items count
  // as many finished tiles towards the entry's down items
  constexpr int tiles_per_item = (kWide || kPair) ? 2 : 1;


  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol_w = l2_policy_evict_first();
      const uint64_t pol_x = l2_policy_evict_last();
      int stage = 0;
      uint32_t phase = 0;
      int slot = 0;
      uint32_t rphase = 0;
      int issued = 0;
      // With every CTA of the grid resident (one per SM), CTA i's first item
      // is item i (for pairs, cluster i's) and later ones come from the
      // counter past the grid: the first item costs no atomic round trip after
      // the dependency wait.
      const int n_first = kPair ? (int)(gridDim.x >> 1) : (int)gridDim.x;
      bool first = static_first != 0;
      for (;;) {
        int item;
        if (!kPair || lead) {
          item = first ? item0
                       : (static_first ? n_first : 0) + atomicAdd(&ws.ctrl[kCtrlWorkCounter], 1);
          first = false;
          if (*abort) item = 0x7FFFFFFF;
          if constexpr (kPair) {
            // hand the item to the second CTA; an item past the end (or the
            // abort sentinel) ends its loop too
            if (!mbar_wait_cluster_bounded(mbe_bar(slot), rphase ^ 1u, nullptr, timeout_ns)) {
              if (!*abort) raise_abort(abort, ws, SLIMWISE_DEVERR_PIPELINE_TIMEOUT);
              break;
            }
            st_shared_cluster(mapa_shared(smem_u32((const void *)(mbox + slot)), 1u), item);
            mbar_arrive_cluster(mapa_shared(mbf_bar(slot), 1u));
          }
        } else {
          // the second CTA of a pair: the item its first CTA took
          if (!mbar_wait_cluster_bounded(mbf_bar(slot), rphase, abort, timeout_ns)) {
            if (!*abort) raise_abort(abort, ws, SLIMWISE_DEVERR_PIPELINE_TIMEOUT);
            break;
          }
          item = mbox[slot];
          mbar_arrive_cluster(mapa_shared(mbe_bar(slot), 0u));
          if (*abort) item = 0x7FFFFFFF;
        }
        if (!mbar_wait_bounded(ite_bar(slot), rphase ^ 1u, abort, timeout_ns)) {
          if (!*abort) raise_abort(abort, ws, SLIMWISE_DEVERR_PIPELINE_TIMEOUT);
          break;
        }
        ring[slot] = item;
        mbar_arrive(itf_bar(slot));
        if (++slot == kItemRing) {
          slot = 0;
          rphase ^= 1u;
        }
        if (item >= total) {
          // no work left for this CTA: the next kernel on the stream may start
          // its launch (it waits for this grid's completion before reading)
          pdl_launch_dependents();
          break;
        }
        const Item it = decode_item<kShared>(item, ip, ws);
        // the item's token rows: one box of the tokens rounded up to 16
        // rows (rows past the entry are loaded but not multiplied); each CTA
        // of a pair loads half of them, from 8 n16 rows further for the second
        const int box_m = token_box_for(it.n16);
        const int tok_row = it.slot_base + (kPair ? (int)crank * it.n16 * (kTokBox / 2) : 0);
        // weight rows: per 128-row half of the item, two 64-row boxes -- the
        // gate rows and the matching up rows, or 128 consecutive down rows;
        // a pair's CTA r loads half r
        const int halves = (kShared && it.shared) ? 1 : wmul;
        const int hstep = it.down ? kTileRows : kGateRows;  // row offset of half 1
        int nk, row0, row1;
        const void *amap;
        const void *bmap;
        if (kShared && it.shared) {
          // the shared expert: its own weights, tokens in batch order
          nk = it.down ? d.Is / kBlockK : d.H / kBlockK;
          amap = it.down ? (const void *)&maps.w_down_s : (const void *)&maps.w_gu_s;
          bmap = it.down ? (const void *)&maps.act_s[box_m] : (const void *)&maps.xt[box_m];
          row0 = it.down ? it.tile * kTileRows : it.tile * kGateRows;
          row1 = it.down ? row0 + kGateRows : row0 + d.Is;
        } else {
          nk = it.down ? d.I / kBlockK : d.H / kBlockK;
          amap = it.down ? (const void *)&maps.w_down : (const void *)&maps.w_gu;
          bmap = it.down ? (const void *)&maps.act[box_m] : (const void *)&maps.xp[box_m];
          const int half0 = kPair ? (int)crank : 0;
          if (it.down) {
            row0 = it.expert * d.H + (it.tile * tiles_per_item + half0) * kTileRows;
            row1 = row0 + kGateRows;
          } else {
            row0 = it.expert * 2 * d.I + (it.tile * tiles_per_item + half0) * kGateRows;
            row1 = row0 + d.I;
          }
        }
        if (it.down) {
          // the entry's activations must be complete: all its gate/up tiles
          const int *done = &ws.entry_done[it.entry];
          int need = (kShared && it.shared) ? ip.t1s : t1 * (kPair ? 2 : 1);
          // test only: the first routed down item waits for one gate/up tile
          // more than exist, so its wait runs out (the timeout path)
          if (starve_first_down && item == ip.S * ip.t1s + ip.r1) ++need;
          bool ok = ld_acquire(done) >= need;
          if (!ok) {
            const uint64_t t0 = global_timer_ns();
            while (!(ok = ld_acquire(done) >= need)) {
              if (*abort) break;
              if (global_timer_ns() - t0 > timeout_ns) {
                raise_abort(abort, ws, SLIMWISE_DEVERR_DEPENDENCY_TIMEOUT);
                break;
              }
              __nanosleep(128);
            }
          }
          if (!ok) break;
          fence_proxy_async_global();
        }
        // bytes the stage barrier expects: for a pair, both CTAs' copies
        const uint32_t stage_tx =
            kPair ? (uint32_t)(2 * kATileBytes + it.n16 * kTokBox * kBlockK * 2)
                  : (uint32_t)(halves * kATileBytes + kTokBox * (box_m + 1) * kBlockK * 2);
        bool ok = true;
        for (int kc = 0; kc < nk; ++kc) {
          if (!mbar_wait_bounded(empty_bar(stage), phase ^ 1u, abort, timeout_ns)) {
            if (!*abort) raise_abort(abort, ws, SLIMWISE_DEVERR_PIPELINE_TIMEOUT);
            ok = false;
            break;
          }
          const int x = kc * kBlockK;
          const uint32_t a = smem_base + (uint32_t)(stage * plan.stage_bytes);
          if (kPair && !lead) {
            const uint32_t lb = mapa_shared(full_bar(stage), 0u);
            tma_load_2d_pair(a, amap, lb, x, row0, pol_w);
            tma_load_2d_pair(a + kATileBytes / 2, amap, lb, x, row1, pol_w);
            tma_load_2d_pair(a + (uint32_t)plan.a_bytes, bmap, lb, x, tok_row, pol_x);
          } else {
            mbar_arrive_expect_tx(full_bar(stage), stage_tx);
            for (int h = 0; h < halves; ++h) {
              const uint32_t ah = a + (uint32_t)(h * kATileBytes);
              tma_load_2d(ah, amap, full_bar(stage), x, row0 + h * hstep, pol_w);
              tma_load_2d(ah + kATileBytes / 2, amap, full_bar(stage), x, row1 + h * hstep,
                          pol_w);
            }
            tma_load_2d(a + (uint32_t)plan.a_bytes, bmap, full_bar(stage), x, tok_row, pol_x);
          }
          ++issued;
          if (++stage == stages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
      }
      if (kPair && !lead) {
        // The second CTA's stages complete on the first CTA's barriers; the
        // first CTA's MMAs read them and their commits arrive here.  Wait
        // (bounded) until every stage still in the ring has been released,
        // so that no copy, read or arrival is left on this CTA's shared
        // memory when it exits.
        const int from = issued > stages ? issued - stages : 0;
        for (int s = from; s < issued; ++s)
          mbar_wait_timeout(empty_bar(s % stages), (uint32_t)((s / stages) & 1), 10000000ull);
      } else if (*abort) {
        // let this CTA's copies in flight land before shared memory goes away
        for (int s = *consumed; s < issued; ++s)
          mbar_wait_timeout(full_bar(s % stages), (uint32_t)((s / stages) & 1), 10000000ull);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && kPair && !lead) {
      // the second CTA of a pair issues no MMA: it only keeps its item ring
      // moving
      int slot = 0;
      uint32_t rphase = 0;
      for (;;) {
        if (!mbar_wait_bounded(itf_bar(slot), rphase, abort, timeout_ns)) {
          if (!*abort) raise_abort(abort, ws, SLIMWISE_DEVERR_PIPELINE_TIMEOUT);
          break;
        }
        const int item = ring[slot];
        mbar_arrive(ite_bar(slot));
        if (++slot == kItemRing) {
          slot = 0;
          rphase ^= 1u;
        }
        if (item >= total) break;
      }
    } else if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int slot = 0;
      uint32_t rphase = 0;
      int n_consumed = 0;
      bool issued_any = false;
      for (int local = 0;; ++local) {
        if (!mbar_wait_bounded(itf_bar(slot), rphase, abort, timeout_ns)) {
          if (!*abort) raise_abort(abort, ws, SLIMWISE_DEVERR_PIPELINE_TIMEOUT);
          break;
        }
        const int item = ring[slot];
        mbar_arrive(ite_bar(slot));
        if (++slot == kItemRing) {
          slot = 0;
          rphase ^= 1u;
        }
        if (item >= total) break;
        const Item it = decode_item<kShared>(item, ip, ws);
        const int b = local & 1;
        const uint32_t use = (uint32_t)(local >> 1);
        const bool freed =
            kPair ? mbar_wait_cluster_bounded(acce_bar(b), (use & 1u) ^ 1u, abort, timeout_ns)
                  : mbar_wait_bounded(acce_bar(b), (use & 1u) ^ 1u, abort, timeout_ns);
        if (!freed) {
          if (!*abort) raise_abort(abort, ws, SLIMWISE_DEVERR_PIPELINE_TIMEOUT);
          break;
        }
        tc_fence_after();
        // half h of the item: A = the stage's weight rows [128 h, 128 h + 128),
        // D = columns [h tok_chunk, ...) of the buffer; B = the token rows.
        // A pair runs one M = 256 MMA: A rows 128-255 and B rows N/2.. are the
        // second CTA's, at the same shared-memory offsets.
        const uint32_t d_tmem = tmem_base + (uint32_t)(b * nb_cols);
        const uint32_t idesc = idesc_bf16_f32(kPair ? 2 * kTileRows : kTileRows, it.n16 * kTokBox);
        const int halves = (kShared && it.shared) ? 1 : wmul;
        const int inner = (kShared && it.shared) ? d.Is : d.I;
        const int nk = it.down ? inner / kBlockK : d.H / kBlockK;
        bool ok = true;
        for (int kc = 0; kc < nk; ++kc) {
          if (!mbar_wait_bounded(full_bar(stage), phase, abort, timeout_ns)) {
            if (!*abort) raise_abort(abort, ws, SLIMWISE_DEVERR_PIPELINE_TIMEOUT);
            ok = false;
            break;
          }
          tc_fence_after();
#ifdef SLIMWISE_TRACE
          if (blockIdx.x == 0 && n_consumed == 0) trace_stamp(ws, tr_step, kTrFfnFirstData);
#endif
          const uint32_t a = smem_base + (uint32_t)(stage * plan.stage_bytes);
          const uint32_t bs = a + (uint32_t)plan.a_bytes;
          if constexpr (kPair) {
#pragma unroll
            for (int kk = 0; kk < kBlockK / 16; ++kk)
              tc_mma_bf16_pair(d_tmem, smem_desc_sw128(a + kk * 32), smem_desc_sw128(bs + kk * 32),
                               idesc, (kc | kk) != 0 ? 1u : 0u);
            tc_commit_pair(empty_bar(stage), (uint16_t)3);
          } else {
            for (int h = 0; h < halves; ++h) {
              const uint32_t as = a + (uint32_t)(h * kATileBytes);
#pragma unroll
              for (int kk = 0; kk < kBlockK / 16; ++kk)
                tc_mma_bf16(d_tmem + (uint32_t)(h * d.tok_chunk), smem_desc_sw128(as + kk * 32),
                            smem_desc_sw128(bs + kk * 32), idesc, (kc | kk) != 0 ? 1u : 0u);
            }
            tc_commit(empty_bar(stage));
          }
          issued_any = true;
          *consumed = ++n_consumed;
          if (++stage == stages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        if constexpr (kPair) tc_commit_pair(accf_bar(b), (uint16_t)3);
        else tc_commit(accf_bar(b));
      }
      if (*abort && issued_any) {
        if constexpr (kPair) tc_commit_pair(drain_bar, (uint16_t)1);
        else tc_commit(drain_bar);
        mbar_wait_timeout(drain_bar, 0, 10000000ull);
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    // Two warpgroups; group g owns TMEM accumulator buffer g, i.e. the items
    // with local index = g (mod 2), so one group's epilogue overlaps the
    // other's and the MMA of the next item.
    const int g = (warp - 2) >> 2;      // epilogue group
    const int q = warp & 3;             // TMEM lane quarter of this warp
    const int row = 32 * q + lane;      // accumulator row = TMEM lane
    const int et = (threadIdx.x - 64) & (kEpiThreads - 1);
    float *xb = xch + g * kTileRows * kXchStride;
    int slot = 0;
    uint32_t rphase = 0;
    for (int local = 0;; ++local) {
      bool got = mbar_wait_bounded(itf_bar(slot), rphase, abort, timeout_ns);
      if (!got && !*abort) raise_abort(abort, ws, SLIMWISE_DEVERR_PIPELINE_TIMEOUT);
      if (!epi_all(g, got)) break;
      const int item = ring[slot];
      mbar_arrive(ite_bar(slot));
      if (++slot == kItemRing) {
        slot = 0;
        rphase ^= 1u;
      }
      if (item >= total) break;
      const int b = local & 1;
      if (b != g) continue;
      const Item it = decode_item<kShared>(item, ip, ws);
      const uint32_t use = (uint32_t)(local >> 1);
      const int halves = (kShared && it.shared) ? 1 : wmul;
      got = mbar_wait_bounded(accf_bar(b), use & 1u, abort, timeout_ns);
      if (!got && !*abort) raise_abort(abort, ws, SLIMWISE_DEVERR_PIPELINE_TIMEOUT);
      if (!epi_all(g, got)) break;
      tc_fence_after();
      const uint32_t taddr = tmem_base + ((uint32_t)(32 * q) << 16) + (uint32_t)(b * nb_cols);
      // 128-row tile of the item that TMEM half hh holds: half hh of a wide
      // item, the CTA's own half of a pair item
      const int tile0 = (kShared && it.shared) ? it.tile
                                               : it.tile * tiles_per_item + (kPair ? (int)crank : 0);
      if (!it.down) {
        // gate rows live in TMEM lanes 0..63, the matching up rows in 64..127
        const int n_loc = et >> 3;          // token column within a 16-chunk
        const int i0 = (et & 7) * 8;        // 8 consecutive intermediate indices
        for (int hh = 0; hh < halves; ++hh) {
          // half hh of a wide item is the 64 gate + 64 up rows of tile 2 t + hh
          const int act_col = (tile0 + hh) * kGateRows + i0;
          for (int c = 0; c < it.n16; ++c) {
            uint32_t v[16];
            tmem_ld16(taddr + (uint32_t)(hh * d.tok_chunk) + c * 16, v);
            tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 16; ++j) xb[row * kXchStride + j] = __uint_as_float(v[j]);
            epi_bar(g);
            const int col = c * 16 + n_loc;
            if (col < it.n) {
              uint32_t packed[4];
#pragma unroll
              for (int ii = 0; ii < 8; ii += 2) {
                float a2[2];
#pragma unroll
                for (int u2 = 0; u2 < 2; ++u2) {
                  const float gv = xb[(i0 + ii + u2) * kXchStride + n_loc];
                  const float uv = xb[(kGateRows + i0 + ii + u2) * kXchStride + n_loc];
                  // SiLU(g) * u = g / (1 + e^-g) * u
                  a2[u2] = gv * __frcp_rn(1.0f + __expf(-gv)) * uv;
                }
                __nv_bfloat162 h2 = __floats2bfloat162_rn(a2[0], a2[1]);
                packed[ii / 2] = *reinterpret_cast<uint32_t *>(&h2);
              }
              // routed: grouped order [B*k, I]; shared: token order [B, Is]
              __nv_bfloat16 *arow = (kShared && it.shared)
                                        ? ws.act_s + (size_t)(it.slot_base + col) * d.Is
                                        : ws.act + (size_t)(it.slot_base + col) * d.I;
              *reinterpret_cast<uint4 *>(arow + act_col) =
                  make_uint4(packed[0], packed[1], packed[2], packed[3]);
            }
            epi_bar(g);  // the exchange buffer is rewritten by the next chunk
          }
        }
        tc_fence_before();
        if constexpr (!kPair) mbar_arrive(acce_bar(b));
        // publish the activations to the TMA (async proxy) readers of any CTA
        fence_proxy_async_global();
        __threadfence();
        epi_bar(g);
        if (et == 0) {
          if constexpr (kPair)
            mbar_arrive_cluster(mapa_shared(acce_bar(b), 0u));
          atomicAdd(&ws.entry_done[it.entry], 1);
        }
      } else {
        __nv_bfloat16 *ybase = (kShared && it.shared) ? ws.y_s : ws.y;  // token / grouped order
        for (int hh = 0; hh < halves; ++hh) {
          const int h = (tile0 + hh) * kTileRows + row;
          for (int c = 0; c < it.n16; ++c) {
            uint32_t v[16];
            tmem_ld16(taddr + (uint32_t)(hh * d.tok_chunk) + c * 16, v);
            tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int col = c * 16 + j;
              if (col < it.n)
                ybase[(size_t)(it.slot_base + col) * d.H + h] = __float2bfloat16_rn(__uint_as_float(v[j]));
            }
          }
        }
        // the expert outputs are all a down item writes: the combine kernel
        // that follows this grid sums them
        tc_fence_before();
        if constexpr (kPair) {
          epi_bar(g);
          if (et == 0) mbar_arrive_cluster(mapa_shared(acce_bar(b), 0u));
        } else {
          mbar_arrive(acce_bar(b));
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  // neither CTA of a pair leaves (or frees TMEM) while the other may still
  // use its shared memory, barriers or TMEM
  if constexpr (kPair) cluster_sync_all();
#ifdef SLIMWISE_TRACE
  if (threadIdx.x == 0) {
    uint64_t t = global_timer_ns();
    atomicMax(reinterpret_cast<unsigned long long *>(ws.ctrl + kCtrlWords) +
                  (tr_step & (kTraceSteps - 1)) * kTrSlots + kTrFfnEnd,
              (unsigned long long)t);
  }
#endif
  if (warp == 1) {
    tc_fence_after();
    if constexpr (kPair) tmem_dealloc_pair(tmem_base, (uint32_t)tmem_cols);
    else tmem_dealloc(tmem_base, (uint32_t)tmem_cols);
  }
}

// The combine of every (token, 128-column tile) after the FFN grid has
// finished: one warp per pair, the same arithmetic and order as the fused
// combine (combine_token).  Launched as the FFN's programmatic dependent, so
// its CTAs become resident beside the FFN's last CTAs and start as soon as
// the FFN's expert outputs are complete.
constexpr int kCombineThreads = 256;

template <bool kShared>
__global__ void __launch_bounds__(kCombineThreads)
    combine_kernel(Dims d, Ws ws, __nv_bfloat16 *__restrict__ out) {
  const int t2 = d.H / kCombineTile;
  const int lane = threadIdx.x & 31;
  const int wpc = kCombineThreads / 32;
  const int pairs = d.B * t2;
  // One pair per warp (the grid covers them all).  Its grouped positions and
  // gates were written by the routing and grouping kernels, which finished
  // before the expert FFN started its work, so they are read before waiting
  // for the FFN; only the expert outputs need the wait.
  const int pr = blockIdx.x * wpc + (threadIdx.x >> 5);
  const int t = pr / t2;
  int p = 0;
  float gj = 0.0f, sg = 0.0f;
  if (pr < pairs) {
    if (lane < d.k) {
      p = __ldcg(&ws.pos[(size_t)t * d.k + lane]);
      gj = __ldcg(&ws.topk_gate[(size_t)t * d.k + lane]);
    }
    if constexpr (kShared) sg = __ldcg(&ws.shared_gate[t]);
  }
  pdl_wait_primary();
  // The next call's routing is not signalled early: its CTAs would compete
  // for SMs with this grid's (and, with 8-token routing clusters, wait for
  // whole GPCs), which cost up to 7 us at B = 288, m' = 32.  It starts when
  // this grid ends.
  if (pr < pairs) combine_token<kShared>(ws, d, out, t, pr - t * t2, lane, p, gj, sg);
}

cudaError_t launch_combine(Dims d, Ws ws, __nv_bfloat16 *out, bool pdl, cudaStream_t stream) {
  const int pairs = d.B * (d.H / kCombineTile);
  const int wpc = kCombineThreads / 32;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((pairs + wpc - 1) / wpc);
  cfg.blockDim = dim3(kCombineThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  if (d.Is > 0) return cudaLaunchKernelEx(&cfg, combine_kernel<true>, d, ws, out);
  return cudaLaunchKernelEx(&cfg, combine_kernel<false>, d, ws, out);
}

int ffn_stages_for(int tok_chunk, int wide, int pair, size_t smem_limit) {
  int s = 12;
  while (s > 2 && ffn_smem_plan(tok_chunk, s, wide, pair).total + 1024 > smem_limit) --s;
  return s;
}

// Clusters of two FFN CTAs that can be resident at once (the pairs' SMs must
// share a GPC), kept per device and shared-memory size.
cudaError_t pair_clusters_resident(const void *kernel, size_t smem, int dev, int *n) {
  thread_local int last_dev = -1;
  thread_local size_t last_smem = 0;
  thread_local int last_n = 0;
  if (dev == last_dev && smem == last_smem) {
    *n = last_n;
    return cudaSuccess;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2);
  cfg.blockDim = dim3(kFfnThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int c = 0;
  cudaError_t err = cudaOccupancyMaxActiveClusters(&c, kernel, &cfg);
  if (err != cudaSuccess) return err;
  if (c < 1) return cudaErrorInvalidConfiguration;
  last_dev = dev;
  last_smem = smem;
  last_n = c;
  *n = c;
  return cudaSuccess;
}

cudaError_t launch_expert_ffn(const FfnMaps &maps, Dims d, Ws ws,
                              __nv_bfloat16 *out, const int32_t *retained, int grid, bool pdl,
                              cudaStream_t stream, uint64_t timeout_ns,
                              int starve_first_down) {
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  int optin = 0, sms = 0;
  err = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (err != cudaSuccess) return err;
  err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (err != cudaSuccess) return err;
  // the token maps exist for boxes of 16 (m + 1) <= tok_chunk rows, and an
  // entry's box covers at most tok_chunk rows: tok_chunk must be a multiple
  // of 16 in [16, 256]
  if (d.tok_chunk < kTokBox || d.tok_chunk > kMaxTokTile || d.tok_chunk % kTokBox != 0)
    return cudaErrorInvalidValue;
  // the dependent combine kernel needs no shared memory: every byte the
  // block may opt into goes to pipeline stages
  const int stages = ffn_stages_for(d.tok_chunk, d.wide, d.pair, (size_t)optin);
  const size_t smem = ffn_smem_plan(d.tok_chunk, stages, d.wide, d.pair).total + 1024;
  if (smem > (size_t)optin) return cudaErrorInvalidConfiguration;
  // wide items only without a shared expert, on whole 256-row tiles, with
  // both accumulators of two buffers in the 512 TMEM columns
  if (d.wide && (d.Is > 0 || d.I % (2 * kGateRows) != 0 || d.H % (2 * kTileRows) != 0 ||
                 d.tok_chunk > 128))
    return cudaErrorInvalidValue;
  // pair items likewise, and never together with wide ones
  if (d.pair && (d.wide || d.Is > 0 || d.I % (2 * kGateRows) != 0 || d.H % (2 * kTileRows) != 0))
    return cudaErrorInvalidValue;
  auto kernel = d.Is > 0   ? expert_ffn_kernel<true, false, false>
                : d.pair ? expert_ffn_kernel<false, false, true>
                : d.wide ? expert_ffn_kernel<false, true, false>
                         : expert_ffn_kernel<false, false, false>;
  err = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (err != cudaSuccess) return err;
  int tmem_cols = 32;
  while (tmem_cols < 2 * ffn_acc_cols(d)) tmem_cols <<= 1;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kFfnThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  int na = 0;
  if (pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  // items are assigned statically to first CTAs only if all of them are
  // resident at once (a down item may wait on another CTA's first item)
  int resident = sms;
  if (d.pair) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = 2;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = 1;
    ++na;
    int clusters = 0;
    err = pair_clusters_resident((const void *)kernel, smem, dev, &clusters);
    if (err != cudaSuccess) return err;
    resident = 2 * clusters;
    // whole pairs, no more than fit at once
    grid &= ~1;
    if (grid > resident) grid = resident;
    if (grid < 2) grid = 2;
    cfg.gridDim = dim3(grid);
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  const int static_first = grid <= resident ? 1 : 0;
  const int early_dependents = d.B > 64 ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, maps, d, ws, out, retained, stages, tmem_cols,
                            static_first, early_dependents, timeout_ns, starve_first_down);
}

}  // namespace slimwise

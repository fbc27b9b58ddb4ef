// route_topk.cu -- router logits over the retained pool, top-k and
// renormalised gates (SlimWise Sec. 3.1, Eq. 2 and the renormalisation that
// follows it).
//
// A thread-block cluster of kClusterCtas CTAs handles TB tokens.  CTA r of
// the cluster evaluates the logits of its slice of the retained experts for
// those tokens and writes each one, through distributed shared memory, into
// the shared memory of the CTA that runs that token's top-k (token tw on CTA
// tw mod 8); after one cluster barrier every top-k reads only its own shared
// memory.  Each CTA thus reads only 1/kClusterCtas of the router rows, and no
// global counter or second kernel is needed to join the slices.
//
// Logits follow the canonical fp32 order: lane l of a warp owns elements
// 128c + 4l + q (q = 0..3) of every 128-wide chunk c, accumulated with fused
// multiply-adds in (c, q) order, then the 32 lane partials are combined by an
// xor butterfly (offsets 16, 8, 4, 2, 1).  Two tokens' sums advance together
// in one packed fma.rn.f32x2 (two independent fp32 fused multiply-adds, each
// rounded as fmaf), which halves the multiply-add instructions of the
// issue-bound logit phase at large batches without changing a bit.  Pruned
// experts are never evaluated: restricting top-k to K' is the Eq. 2 mask
// with tau = -inf, with no separate masking pass.  Top-k is a warp-wide
// arg-max repeated k times on (order-preserving logit bits desc, expert id
// asc): each lane sorts its candidates once, then every round is two warp
// reductions over the lanes' current heads, so ties go to the lowest
// original id whatever the order of K'.
#include <cooperative_groups.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace slimwise {

constexpr int kRouteThreads = 256;
constexpr int kRouteWarps = kRouteThreads / 32;
constexpr int kClusterCtas = 8;
constexpr int kChunkBatch = 8;  // 128-wide chunks whose loads are issued together
constexpr int kPairChunkBatch = 4;  // the same, per row, when a warp takes two rows

// Order-preserving map of an fp32 value to uint32 (-0 folded onto +0).
__device__ __forceinline__ uint32_t logit_order_bits(float z) {
  uint32_t b = __float_as_uint(z);
  if ((b << 1) == 0u) b = 0u;
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float logit_from_order_bits(uint32_t o) {
  uint32_t b = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
  return __uint_as_float(b);
}

// Hidden rows are staged in shared memory either as bf16 (half the space) or
// converted once to fp32 (no per-use conversion).  The product and the
// summation order are the same.  With two or more tokens per cluster the
// tokens are staged in pairs, interleaved element by element: for token pair
// tp, 128-wide chunk c and lane l, the quads ((tp nchunks + c) 2 + half) 32
// + l hold elements h = 128 c + 4 l + 2 half + {0, 1} as (t, h), (t + 1, h),
// (t, h + 1), (t + 1, h + 1), so that one load gives both tokens' values of
// two elements and consecutive lanes read consecutive quads.  A single token
// (TB = 1) is staged as its plain row.
// load_x4: the four consecutive staged elements from element index i.
__device__ __forceinline__ float4 load_x4(const __nv_bfloat16 *xs, size_t i) {
  const uint2 xr = *reinterpret_cast<const uint2 *>(xs + i);
  return make_float4(__uint_as_float(xr.x << 16), __uint_as_float(xr.x & 0xFFFF0000u),
                     __uint_as_float(xr.y << 16), __uint_as_float(xr.y & 0xFFFF0000u));
}
__device__ __forceinline__ float4 load_x4(const float *xs, size_t i) {
  return *reinterpret_cast<const float4 *>(xs + i);
}

// c0 = fma(a0, w, c0) and c1 = fma(a1, w, c1): two independent fused
// multiply-adds in one packed instruction, each rounded once to nearest
// exactly as fmaf, so two tokens' canonical sums advance together.
__device__ __forceinline__ void ffma2_acc(float &c0, float &c1, float a0, float a1, float w) {
  asm("{\n\t.reg .b64 ra, rw, rc;\n\t"
      "mov.b64 ra, {%2, %3};\n\t"
      "mov.b64 rw, {%4, %4};\n\t"
      "mov.b64 rc, {%0, %1};\n\t"
      "fma.rn.f32x2 rc, ra, rw, rc;\n\t"
      "mov.b64 {%0, %1}, rc;\n\t}"
      : "+f"(c0), "+f"(c1)
      : "f"(a0), "f"(a1), "f"(w));
}

// Element index of quad (tp, c, half, lane) of the paired staging.
__device__ __forceinline__ size_t pair_quad(int tp, int nchunks, int c, int half, int lane) {
  return ((((size_t)tp * nchunks + c) * 2 + half) * 32 + lane) * 4;
}

// Chunk c of one router row (lane's four weights w) into every token's sum,
// elements h = 128 c + 4 lane + q in q order.
template <int TB, typename XT>
__device__ __forceinline__ void fma_chunk(const XT *xs, int nchunks, int c, int lane, float4 w,
                                          float (&p)[TB]) {
  if constexpr (TB == 1) {
    const float4 x = load_x4(xs, ((size_t)c * 32 + lane) * 4);
    p[0] = fmaf(x.x, w.x, p[0]);
    p[0] = fmaf(x.y, w.y, p[0]);
    p[0] = fmaf(x.z, w.z, p[0]);
    p[0] = fmaf(x.w, w.w, p[0]);
  } else {
#pragma unroll
    for (int tp = 0; tp < TB / 2; ++tp) {
      const float4 a = load_x4(xs, pair_quad(tp, nchunks, c, 0, lane));
      const float4 b = load_x4(xs, pair_quad(tp, nchunks, c, 1, lane));
      ffma2_acc(p[2 * tp], p[2 * tp + 1], a.x, a.y, w.x);
      ffma2_acc(p[2 * tp], p[2 * tp + 1], a.z, a.w, w.y);
      ffma2_acc(p[2 * tp], p[2 * tp + 1], b.x, b.y, w.z);
      ffma2_acc(p[2 * tp], p[2 * tp + 1], b.z, b.w, w.w);
    }
  }
}

// Two router rows at once: each staged hidden vector feeds both rows' sums.
template <int TB, typename XT>
__device__ __forceinline__ void fma_chunk2(const XT *xs, int nchunks, int c, int lane, float4 w0,
                                           float4 w1, float (&p0)[TB], float (&p1)[TB]) {
  if constexpr (TB == 1) {
    const float4 x = load_x4(xs, ((size_t)c * 32 + lane) * 4);
    p0[0] = fmaf(x.x, w0.x, p0[0]);
    p0[0] = fmaf(x.y, w0.y, p0[0]);
    p0[0] = fmaf(x.z, w0.z, p0[0]);
    p0[0] = fmaf(x.w, w0.w, p0[0]);
    p1[0] = fmaf(x.x, w1.x, p1[0]);
    p1[0] = fmaf(x.y, w1.y, p1[0]);
    p1[0] = fmaf(x.z, w1.z, p1[0]);
    p1[0] = fmaf(x.w, w1.w, p1[0]);
  } else {
#pragma unroll
    for (int tp = 0; tp < TB / 2; ++tp) {
      const float4 a = load_x4(xs, pair_quad(tp, nchunks, c, 0, lane));
      const float4 b = load_x4(xs, pair_quad(tp, nchunks, c, 1, lane));
      ffma2_acc(p0[2 * tp], p0[2 * tp + 1], a.x, a.y, w0.x);
      ffma2_acc(p0[2 * tp], p0[2 * tp + 1], a.z, a.w, w0.y);
      ffma2_acc(p0[2 * tp], p0[2 * tp + 1], b.x, b.y, w0.z);
      ffma2_acc(p0[2 * tp], p0[2 * tp + 1], b.z, b.w, w0.w);
      ffma2_acc(p1[2 * tp], p1[2 * tp + 1], a.x, a.y, w1.x);
      ffma2_acc(p1[2 * tp], p1[2 * tp + 1], a.z, a.w, w1.y);
      ffma2_acc(p1[2 * tp], p1[2 * tp + 1], b.x, b.y, w1.z);
      ffma2_acc(p1[2 * tp], p1[2 * tp + 1], b.z, b.w, w1.w);
    }
  }
}

// Hidden rows are staged as fp32 (no conversion per use) except at TB = 4
// and TB = 16, which stage bf16: at 16 tokens so that two CTAs fit on an SM,
// at 4 because it measured no slower.
template <int TB>
struct StageType {
  using T = float;
};
template <>
struct StageType<4> {
  using T = __nv_bfloat16;
};
template <>
struct StageType<16> {
  using T = __nv_bfloat16;
};


// Shared memory of one CTA: hidden rows (TB x H elements of StageType, in
// token pairs from TB = 2 on; see load_x4), the logits of
// the tokens whose top-k it runs [ceil(TB/8)][m] fp32 (written by every CTA
// of the cluster), retained ids [m] int32.  Rows of tokens past the batch are
// zero, so every token slot computes (and discards) a logit.
// Round j of the top-k: the winner (order bits whi, complemented id wlo) goes
// to lane j.  With no candidate left (fewer than k distinct ids, already
// reported) a valid id stands in.
__device__ __forceinline__ void take_winner(uint32_t whi, uint32_t wlo, int j, int lane,
                                            const int32_t *ids, const Dims &d, float &my_z,
                                            int &my_e) {
  uint32_t wid = 0xFFFFFFFFu - wlo;
  if (whi == 0u || wid >= (uint32_t)d.E) wid = (uint32_t)ids[0];
  if (lane == j) {
    my_z = logit_from_order_bits(whi);
    my_e = (int)wid;
  }
}

// TB tokens per cluster; NC candidates per lane in the register top-k
// (m' <= 32 NC), or NC = 0 for the general top-k of larger pools.
template <int TB, int NC>
// Two CTAs per SM worth of registers, so one wave of CTAs holds 38 clusters.
__global__ void __launch_bounds__(kRouteThreads, 2)
    route_topk_kernel(const __nv_bfloat16 *__restrict__ hidden,
                      const float *__restrict__ router_w,
                      const int32_t *__restrict__ retained, Dims d, Ws ws) {
  using XT = typename StageType<TB>::T;
  extern __shared__ __align__(16) unsigned char smem[];
  cg::cluster_group cluster = cg::this_cluster();
  const int crank = (int)cluster.block_rank();
  const int H = d.H, m = d.m_ret, k = d.k;
  const int slice = (m + kClusterCtas - 1) / kClusterCtas;
  constexpr int kOwn = (TB + kClusterCtas - 1) / kClusterCtas;  // tokens whose top-k a CTA runs
  XT *xs = reinterpret_cast<XT *>(smem);
  float *zs = reinterpret_cast<float *>(smem + (size_t)TB * H * sizeof(XT));  // [kOwn][m]
  int32_t *ids = reinterpret_cast<int32_t *>(zs + (size_t)kOwn * m);

  // Before waiting for the previous kernel on the stream (this CTA may be
  // resident while it finishes): warm L2 with this CTA's router rows.  These
  // are prefetches only -- no value read here is used, and the ids that
  // address them are read past L1 -- so the results do not depend on whether
  // the previous kernel wrote the router rows or the retained ids.
  {
    const int r_lo = crank * slice, r_hi = min(m, r_lo + slice);
    const int lpr = H / 32;  // 128-byte lines per fp32 router row
    for (int i = threadIdx.x; i < (r_hi - r_lo) * lpr; i += blockDim.x) {
      const int r = r_lo + i / lpr;
      const int e = min(max(retained ? __ldcg(retained + r) : r, 0), d.E - 1);
      prefetch_l2(router_w + (size_t)e * H + (size_t)(i % lpr) * 32);
    }
  }
  // The inputs may come from the previous kernel on the stream.
  pdl_wait_primary();
  // Let the grouping kernel become resident; it waits for this grid to end.
  pdl_launch_dependents();
#ifdef SLIMWISE_TRACE
  const int tr_step = ws.ctrl[kCtrlTraceStep];
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    trace_stamp(ws, tr_step, kTrRouteStart);
    reinterpret_cast<uint64_t *>(ws.ctrl + kCtrlWords)[(tr_step & (kTraceSteps - 1)) * kTrSlots + kTrFfnEnd] = 0;
  }
#endif

  const int cluster_id = blockIdx.x / kClusterCtas;
  const int t0 = cluster_id * TB;
  const int nt = min(TB, d.B - t0);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // Retained ids, clamped into [0, E) so a bad id cannot fault; the grid's
  // last CTA also reports bad and repeated ids and resets the error word of
  // this call.
  for (int r = threadIdx.x; r < m; r += blockDim.x) {
    int e = retained ? retained[r] : r;
    ids[r] = min(max(e, 0), d.E - 1);
  }
  if (blockIdx.x == gridDim.x - 1) {
    __shared__ uint32_t seen[kMaxExperts / 32];
    __shared__ int bad;
    for (int i = threadIdx.x; i < kMaxExperts / 32; i += blockDim.x) seen[i] = 0;
    if (threadIdx.x == 0) bad = 0;
    __syncthreads();
    for (int r = threadIdx.x; r < m; r += blockDim.x) {
      int e = retained ? retained[r] : r;
      if (e < 0 || e >= d.E) {
        atomicOr(&bad, SLIMWISE_DEVERR_BAD_RETAINED);
      } else {
        uint32_t bit = 1u << (e & 31);
        if (atomicOr(&seen[e >> 5], bit) & bit)
          atomicOr(&bad, SLIMWISE_DEVERR_DUPLICATE_RETAINED);
      }
    }
    __syncthreads();
    if (threadIdx.x == 0) ws.ctrl[kCtrlErr] = bad;
  }

  // Hidden rows of the cluster's tokens (16-byte vectors of 8 bf16), zero
  // past the batch.  Each thread issues TB loads before storing any, so the
  // staging costs one memory round trip per TB * 256 vectors.  With token
  // pairs a thread loads the same vector of both tokens of a pair and writes
  // the four interleaved quads it covers (lanes 2 (v mod 16) and 2 (v mod 16)
  // + 1 of chunk v / 16, both halves).
  const int vecs = H / 8;
  const int nchunks = H / 128;
  auto hidden_vec = [&](int t, int v) {
    return t < nt ? reinterpret_cast<const uint4 *>(hidden + (size_t)(t0 + t) * H)[v]
                  : make_uint4(0u, 0u, 0u, 0u);
  };
  if constexpr (TB == 1) {
    for (int v = threadIdx.x; v < vecs; v += kRouteThreads) {
      const uint4 r = hidden_vec(0, v);
      float4 *dst = reinterpret_cast<float4 *>(xs + 8 * v);
      dst[0] = make_float4(__uint_as_float(r.x << 16), __uint_as_float(r.x & 0xFFFF0000u),
                           __uint_as_float(r.y << 16), __uint_as_float(r.y & 0xFFFF0000u));
      dst[1] = make_float4(__uint_as_float(r.z << 16), __uint_as_float(r.z & 0xFFFF0000u),
                           __uint_as_float(r.w << 16), __uint_as_float(r.w & 0xFFFF0000u));
    }
  } else {
    constexpr int kPairsPerPass = TB / 2;  // pair-vectors per thread per pass
    const int items = (TB / 2) * vecs;
    for (int i0 = 0; i0 < items; i0 += kPairsPerPass * kRouteThreads) {
      uint4 r0[kPairsPerPass], r1[kPairsPerPass];
#pragma unroll
      for (int u = 0; u < kPairsPerPass; ++u) {
        const int i = i0 + u * kRouteThreads + (int)threadIdx.x;
        const int tp = i / vecs, v = i - tp * vecs;
        const bool in = i < items;
        r0[u] = in ? hidden_vec(2 * tp, v) : make_uint4(0u, 0u, 0u, 0u);
        r1[u] = in ? hidden_vec(2 * tp + 1, v) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < kPairsPerPass; ++u) {
        const int i = i0 + u * kRouteThreads + (int)threadIdx.x;
        if (i >= items) break;
        const int tp = i / vecs, v = i - tp * vecs;
        const int c = v >> 4, l0 = 2 * (v & 15);
        // words w of a vector hold elements 2w (low half) and 2w + 1 (high)
        const uint32_t a[4] = {r0[u].x, r0[u].y, r0[u].z, r0[u].w};
        const uint32_t b[4] = {r1[u].x, r1[u].y, r1[u].z, r1[u].w};
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          // elements 2w, 2w + 1: lane l0 + w / 2, half w % 2
          const size_t q = pair_quad(tp, nchunks, c, w & 1, l0 + (w >> 1));
          if constexpr (sizeof(XT) == 2) {
            // (t, 2w) | (t + 1, 2w) << 16, then the same for element 2w + 1
            *reinterpret_cast<uint2 *>(xs + q) =
                make_uint2((a[w] & 0xFFFFu) | (b[w] << 16), (a[w] >> 16) | (b[w] & 0xFFFF0000u));
          } else {
            *reinterpret_cast<float4 *>(xs + q) =
                make_float4(__uint_as_float(a[w] << 16), __uint_as_float(b[w] << 16),
                            __uint_as_float(a[w] & 0xFFFF0000u), __uint_as_float(b[w] & 0xFFFF0000u));
          }
        }
      }
    }
  }
  __syncthreads();

  // Logits of this CTA's slice [r_lo, r_hi) of the retained list.  With at
  // least two rows per warp (at 8 tokens per cluster: two rows per slice), a
  // warp takes its rows in pairs (rows r, r + 1), which halves the
  // shared-memory reads of the staged hidden rows; the sums and their order
  // are those of one row at a time.
  const int r_lo = crank * slice, r_hi = min(m, r_lo + slice);
  // At 8 tokens per cluster the staged rows' shared-memory reads bound the
  // logits, so pairs pay from two rows on (1.6 us at B = 256, m' = 64); at
  // 16 tokens (fewer warps busy) they lost 2 us at B = 512, m' = 32.
  const int npair = ((TB == 8 && r_hi - r_lo >= 2) || r_hi - r_lo >= 2 * kRouteWarps)
                        ? (r_hi - r_lo) / 2 : 0;
  for (int pi = warp; pi < npair; pi += kRouteWarps) {
    const int r = r_lo + 2 * pi;
    const float4 *w0 = reinterpret_cast<const float4 *>(router_w + (size_t)ids[r] * H) + lane;
    const float4 *w1 = reinterpret_cast<const float4 *>(router_w + (size_t)ids[r + 1] * H) + lane;
    float p0[TB], p1[TB];
#pragma unroll
    for (int t = 0; t < TB; ++t) p0[t] = p1[t] = 0.0f;
    for (int c0 = 0; c0 < nchunks; c0 += kPairChunkBatch) {
      float4 v0[kPairChunkBatch], v1[kPairChunkBatch];
#pragma unroll
      for (int u = 0; u < kPairChunkBatch; ++u)
        if (c0 + u < nchunks) {
          v0[u] = __ldg(w0 + 32 * (c0 + u));
          v1[u] = __ldg(w1 + 32 * (c0 + u));
        }
#pragma unroll
      for (int u = 0; u < kPairChunkBatch; ++u)
        if (c0 + u < nchunks)
          fma_chunk2<TB>(xs, nchunks, c0 + u, lane, v0[u], v1[u], p0, p1);
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1)
#pragma unroll
      for (int t = 0; t < TB; ++t) {
        p0[t] = p0[t] + __shfl_xor_sync(0xFFFFFFFFu, p0[t], off);
        p1[t] = p1[t] + __shfl_xor_sync(0xFFFFFFFFu, p1[t], off);
      }
    // lane t sends token t's two logits to the CTA that runs its top-k
#pragma unroll
    for (int t = 0; t < TB; ++t)
      if (lane == t && t < nt) {
        float *dst = cluster.map_shared_rank(zs, t % kClusterCtas) + (size_t)(t / kClusterCtas) * m;
        dst[r] = p0[t];
        dst[r + 1] = p1[t];
      }
  }
  for (int r = r_lo + 2 * npair + warp; r < r_hi; r += kRouteWarps) {
    const float4 *wrow = reinterpret_cast<const float4 *>(router_w + (size_t)ids[r] * H) + lane;
    float p[TB];
#pragma unroll
    for (int t = 0; t < TB; ++t) p[t] = 0.0f;
    for (int c0 = 0; c0 < nchunks; c0 += kChunkBatch) {
      float4 v[kChunkBatch];
#pragma unroll
      for (int u = 0; u < kChunkBatch; ++u)
        if (c0 + u < nchunks) v[u] = __ldg(wrow + 32 * (c0 + u));
#pragma unroll
      for (int u = 0; u < kChunkBatch; ++u)
        if (c0 + u < nchunks) fma_chunk<TB>(xs, nchunks, c0 + u, lane, v[u], p);
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1)
#pragma unroll
      for (int t = 0; t < TB; ++t) p[t] = p[t] + __shfl_xor_sync(0xFFFFFFFFu, p[t], off);
#pragma unroll
    for (int t = 0; t < TB; ++t)
      if (lane == t && t < nt)
        cluster.map_shared_rank(zs, t % kClusterCtas)[(size_t)(t / kClusterCtas) * m + r] = p[t];
  }
  // every logit is in the shared memory of the CTA that needs it; after this
  // barrier no CTA touches another's shared memory, so none waits at the end
  cluster.sync();

  // Top-k and gates: token tw of the cluster is handled by warp tw / 8 of the
  // cluster's CTA tw % 8, so the tokens' top-k run side by side.
  const int tw = warp * kClusterCtas + crank;
  if (tw < nt) {
    const int t = t0 + tw;
    float my_z = 0.0f;
    int my_e = 0;
    if constexpr (NC > 0) {
      // this lane's candidates r = lane + 32 i (i < NC) as 64-bit keys
      // (order-preserving logit bits, complemented id; 0 = none), kept sorted
      // descending in registers -- every index below is a compile-time one;
      // all loads are issued before any is used
      float zc[NC];
#pragma unroll
      for (int i = 0; i < NC; ++i) {
        const int r = lane + 32 * i;
        if (r < m) {
          zc[i] = zs[(size_t)warp * m + r];
        }
      }
      unsigned long long key[NC];
#pragma unroll
      for (int i = 0; i < NC; ++i) {
        const int r = lane + 32 * i;
        key[i] = r < m ? ((unsigned long long)logit_order_bits(zc[i]) << 32) |
                             (unsigned long long)(0xFFFFFFFFu - (uint32_t)ids[r])
                       : 0ull;
#pragma unroll
        for (int j = i; j > 0; --j)
          if (key[j] > key[j - 1]) {
            const unsigned long long tmp = key[j];
            key[j] = key[j - 1];
            key[j - 1] = tmp;
          }
      }
      // k rounds: the warp's largest head key wins and its lane pops it
      for (int j = 0; j < k; ++j) {
        const unsigned long long mine = key[0];
        const uint32_t hi = (uint32_t)(mine >> 32), lo = (uint32_t)mine;
        const uint32_t whi = __reduce_max_sync(0xFFFFFFFFu, hi);
        const uint32_t wlo = __reduce_max_sync(0xFFFFFFFFu, hi == whi ? lo : 0u);
        const unsigned long long win = ((unsigned long long)whi << 32) | wlo;
        // pop every copy of the winner (repeated retained ids give equal keys)
        for (int pops = 0; pops < NC && key[0] == win && win != 0ull; ++pops) {
#pragma unroll
          for (int i = 0; i + 1 < NC; ++i) key[i] = key[i + 1];
          key[NC - 1] = 0ull;
        }
        take_winner(whi, wlo, j, lane, ids, d, my_z, my_e);
      }
    } else {
      // large pools: the lane's candidates sorted in a local array
      unsigned long long key[kMaxExperts / 32];
      int nc = 0;
      for (int r0 = lane; r0 < m; r0 += 128) {
        float zc[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int r = r0 + 32 * u;
          if (r < m) {
            zc[u] = zs[(size_t)warp * m + r];
          }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int r = r0 + 32 * u;
          if (r < m) {
            const unsigned long long kv = ((unsigned long long)logit_order_bits(zc[u]) << 32) |
                                          (unsigned long long)(0xFFFFFFFFu - (uint32_t)ids[r]);
            int i = nc++;
            while (i > 0 && key[i - 1] < kv) {
              key[i] = key[i - 1];
              --i;
            }
            key[i] = kv;
          }
        }
      }
      int head = 0;
      for (int j = 0; j < k; ++j) {
        const unsigned long long mine = head < nc ? key[head] : 0ull;
        const uint32_t hi = (uint32_t)(mine >> 32), lo = (uint32_t)mine;
        const uint32_t whi = __reduce_max_sync(0xFFFFFFFFu, hi);
        const uint32_t wlo = __reduce_max_sync(0xFFFFFFFFu, hi == whi ? lo : 0u);
        const unsigned long long win = ((unsigned long long)whi << 32) | wlo;
        while (head < nc && key[head] == win) ++head;
        take_winner(whi, wlo, j, lane, ids, d, my_z, my_e);
      }
    }
    // g_j = exp(z_j - z_1) / sum_j' exp(z_j' - z_1), the sum in j order.
    const float z1 = __shfl_sync(0xFFFFFFFFu, my_z, 0);
    const float w = (lane < k) ? expf(my_z - z1) : 0.0f;
    float denom = 0.0f;
    for (int j = 0; j < k; ++j) denom += __shfl_sync(0xFFFFFFFFu, w, j);
    if (lane < k) {
      ws.topk_idx[(size_t)t * k + lane] = my_e;
      ws.topk_gate[(size_t)t * k + lane] = w / denom;
    }
  }
#ifdef SLIMWISE_TRACE
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    trace_stamp(ws, tr_step, kTrRouteEnd);
    ws.ctrl[kCtrlTraceStep] = tr_step + 1;
  }
#endif
}

// Dynamic shared memory of a routing CTA with TB tokens.
template <int TB>
size_t route_smem_bytes(const Dims &d) {
  return (size_t)TB * d.H * sizeof(typename StageType<TB>::T) +
         (size_t)((TB + kClusterCtas - 1) / kClusterCtas) * d.m_ret * 4 + (size_t)d.m_ret * 4;
}

template <int TB, int NC>
cudaError_t launch_route_tb(const __nv_bfloat16 *hidden, const float *router_w,
                            const int32_t *retained, Dims d, Ws ws, bool pdl,
                            cudaStream_t stream) {
  const size_t smem = route_smem_bytes<TB>(d);
  cudaError_t err = cudaFuncSetAttribute(
      route_topk_kernel<TB, NC>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (err != cudaSuccess) return err;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(((d.B + TB - 1) / TB) * kClusterCtas);
  cfg.blockDim = dim3(kRouteThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kClusterCtas;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, route_topk_kernel<TB, NC>, hidden, router_w, retained, d, ws);
}

template <int TB>
cudaError_t launch_route_nc(const __nv_bfloat16 *hidden, const float *router_w,
                            const int32_t *retained, Dims d, Ws ws, bool pdl,
                            cudaStream_t stream) {
  if (d.m_ret <= 128) return launch_route_tb<TB, 4>(hidden, router_w, retained, d, ws, pdl, stream);
  if (d.m_ret <= 256) return launch_route_tb<TB, 8>(hidden, router_w, retained, d, ws, pdl, stream);
  return launch_route_tb<TB, 0>(hidden, router_w, retained, d, ws, pdl, stream);
}

cudaError_t launch_route_topk(const __nv_bfloat16 *hidden, const float *router_w,
                              const int32_t *retained, Dims d, Ws ws, bool pdl,
                              cudaStream_t stream) {
  int dev = 0, optin = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  err = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (err != cudaSuccess) return err;
  // wide hidden rows: fewer tokens per cluster until they fit in shared memory
  int tb = route_tokens_per_cluster(d.B, d.m_ret);
  auto fits = [&](int t) {
    const size_t need = t == 16 ? route_smem_bytes<16>(d) : t == 8 ? route_smem_bytes<8>(d)
                      : t == 4 ? route_smem_bytes<4>(d) : t == 2 ? route_smem_bytes<2>(d)
                      : route_smem_bytes<1>(d);
    return need <= (size_t)optin;
  };
  while (tb > 1 && !fits(tb)) tb >>= 1;
  switch (tb) {
    case 1: return launch_route_nc<1>(hidden, router_w, retained, d, ws, pdl, stream);
    case 2: return launch_route_nc<2>(hidden, router_w, retained, d, ws, pdl, stream);
    case 4: return launch_route_nc<4>(hidden, router_w, retained, d, ws, pdl, stream);
    case 8: return launch_route_nc<8>(hidden, router_w, retained, d, ws, pdl, stream);
    default: return launch_route_nc<16>(hidden, router_w, retained, d, ws, pdl, stream);
  }
}

}  // namespace slimwise

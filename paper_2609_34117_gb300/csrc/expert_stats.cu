// expert_stats.cu -- expert-importance statistics of a calibration pass and
// the retained set they select (SlimWise Sec. 2.3 and Sec. 3.1).
//
// The statistics are taken from a full-pool layer call: its workspace holds,
// for every (token, selection) slot in grouped order (expert ascending, token
// ascending), the selected expert's output row y (accumulated in fp32, stored
// as bf16) and, through perm, the slot's gate.  For each expert e and each token t routed to it:
//   stats[e][0] += 1             tokens routed to e
//   stats[e][1] += g_te          routing mass
//   stats[e][2] += ||y||_2       expert activation norm (EAN)
//   stats[e][3] += g_te ||y||_2  REAP numerator (score = stats[3] / stats[0])
// One warp per expert walks its rows in order, so every expert's sums are
// taken in token order; they accumulate in fp64 across calibration batches.
#include "common.cuh"

namespace slimwise {

constexpr int kStatsWarps = 8;

__global__ void __launch_bounds__(kStatsWarps * 32)
    expert_stats_kernel(Dims d, Ws ws, double *__restrict__ stats) {
  const int lane = threadIdx.x & 31;
  const int e = blockIdx.x * kStatsWarps + (threadIdx.x >> 5);
  if (e >= d.E) return;
  const int p0 = __ldcg(&ws.offsets[e]), p1 = __ldcg(&ws.offsets[e + 1]);
  double cnt = 0.0, mass = 0.0, ean = 0.0, reap = 0.0;
  for (int p = p0; p < p1; ++p) {
    // ||y||^2: lane l sums its 8-wide columns 256c + 8l .. +7, then an xor
    // butterfly over the lanes
    const uint4 *row = reinterpret_cast<const uint4 *>(ws.y + (size_t)p * d.H);
    float s = 0.0f;
    for (int c = lane; c < d.H / 8; c += 32) {
      const uint4 v = __ldcg(row + c);
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float a = __uint_as_float(w[q] << 16), b = __uint_as_float(w[q] & 0xFFFF0000u);
        s = fmaf(a, a, s);
        s = fmaf(b, b, s);
      }
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, off);
    const double nrm = sqrt((double)s);
    const double g = (double)__ldcg(&ws.topk_gate[__ldcg(&ws.perm[p])]);
    cnt += 1.0;
    mass += g;
    ean += nrm;
    reap += g * nrm;
  }
  if (lane == 0) {
    double *st = stats + (size_t)e * 4;
    st[0] += cnt;
    st[1] += mass;
    st[2] += ean;
    st[3] += reap;
  }
}

cudaError_t launch_expert_stats(Dims d, Ws ws, double *stats, cudaStream_t stream) {
  const int ctas = (d.E + kStatsWarps - 1) / kStatsWarps;
  expert_stats_kernel<<<ctas, kStatsWarps * 32, 0, stream>>>(d, ws, stats);
  return cudaGetLastError();
}

// Retained set: the m' experts of highest score, ties to the lowest id, ids
// ascending.  Scores: 0 routing mass, 1 EAN, 2 REAP (numerator / count, 0 for
// an expert no token chose).  One CTA; each thread ranks its experts against
// all others, then a block scan compacts the kept ids.
__device__ __forceinline__ double expert_score(const double *st, int criterion) {
  if (criterion == 0) return st[1];
  if (criterion == 1) return st[2];
  return st[0] > 0.0 ? st[3] / st[0] : 0.0;
}

__global__ void __launch_bounds__(kMaxExperts)
    select_retained_kernel(const double *__restrict__ stats, int E, int m_prime,
                           int criterion, int32_t *__restrict__ ids) {
  __shared__ double score[kMaxExperts];
  __shared__ int warp_sum[kMaxExperts / 32];
  const int e = threadIdx.x;
  if (e < E) score[e] = expert_score(stats + (size_t)e * 4, criterion);
  __syncthreads();
  int keep = 0;
  if (e < E) {
    const double se = score[e];
    int rank = 0;
    for (int f = 0; f < E; ++f) {
      const double sf = score[f];
      rank += (sf > se || (sf == se && f < e)) ? 1 : 0;
    }
    keep = rank < m_prime ? 1 : 0;
  }
  // exclusive scan of keep over the block: warp inclusive scans, then warp totals
  const int lane = e & 31, w = e >> 5;
  int incl = keep;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int o = __shfl_up_sync(0xFFFFFFFFu, incl, off);
    if (lane >= off) incl += o;
  }
  if (lane == 31) warp_sum[w] = incl;
  __syncthreads();
  if (w == 0) {
    const int nw = blockDim.x / 32;
    int v = lane < nw ? warp_sum[lane] : 0;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int o = __shfl_up_sync(0xFFFFFFFFu, v, off);
      if (lane >= off) v += o;
    }
    if (lane < nw) warp_sum[lane] = v;  // inclusive totals
  }
  __syncthreads();
  const int before = (w > 0 ? warp_sum[w - 1] : 0) + incl - keep;
  if (keep) ids[before] = e;
}

cudaError_t launch_select_retained(const double *stats, int E, int m_prime, int criterion,
                                   int32_t *ids, cudaStream_t stream) {
  const int threads = (E + 31) / 32 * 32;
  select_retained_kernel<<<1, threads, 0, stream>>>(stats, E, m_prime, criterion, ids);
  return cudaGetLastError();
}

}  // namespace slimwise

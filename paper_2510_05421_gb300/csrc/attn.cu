// Block-causal multi-query attention over the KV cache.
//
// The verify pass of Sec. 3.3 evaluates h_{L,t+i-1} for i = 1..k_spec in one
// pass: query row i of a sequence's block sits at position n+i and sees
// cache positions 0..n+i (the block's own K/V rows were written into the
// cache by the QKV epilogue just before).  Draft and AR passes are the
// one-row case, prefill chunks the many-row case.
//
// A CTA covers (position split, KV head, sequence x query group) and reads
// each K/V row of its split once for all queries of the group (the block's
// rows times the query heads sharing the KV head, GQA).  Split boundaries
// are fixed multiples of `split_len`, independent of the number of query
// rows; the last CTA to finish a (sequence, group, head) combines the splits
// in split order.  Within a split, positions are assigned to warps by a fixed
// rule, and positions a row must not see contribute exact zeros, so a row's
// output does not depend on how many rows share the launch.
//
// The bf16 tensor-core kernel (attn_mma_kernel; decode passes and prefill
// chunks) instead splits each row's own positions evenly: see the rule at
// its split set-up.
//
// Decode (<= 16 rows per sequence): attn_dec_kernel streams the split's K/V
// through a shared-memory ring by bulk copies and keeps a query group's
// vectors, scores and accumulators in registers; each warp walks its
// positions four at a time (lane = hd/32 dims), reduces the dot products
// with shuffles and runs an online softmax; the four warps merge through
// shared memory at the end.
// Prefill chunks: attn_smem_kernel stages 64-position K/V blocks in shared
// memory for 16 queries at a time.
#include <algorithm>
#include <cmath>
#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.h"

namespace dvi {

namespace cg = cooperative_groups;

constexpr int kRegQ = 8;      // query vectors per CTA in the decode kernel
constexpr int kRegPos = 4;    // positions per warp step

template <typename T, int N>
__device__ __forceinline__ void load_n(const T* src, float* dst);
template <>
__device__ __forceinline__ void load_n<__nv_bfloat16, 4>(const __nv_bfloat16* src, float* dst) {
  const uint2 u = *reinterpret_cast<const uint2*>(src);
  dst[0] = bf16_lo(u.x); dst[1] = bf16_hi(u.x); dst[2] = bf16_lo(u.y); dst[3] = bf16_hi(u.y);
}
template <>
__device__ __forceinline__ void load_n<__nv_bfloat16, 2>(const __nv_bfloat16* src, float* dst) {
  const uint32_t u = *reinterpret_cast<const uint32_t*>(src);
  dst[0] = bf16_lo(u); dst[1] = bf16_hi(u);
}
template <>
__device__ __forceinline__ void load_n<float, 4>(const float* src, float* dst) {
  const float4 a = *reinterpret_cast<const float4*>(src);
  dst[0] = a.x; dst[1] = a.y; dst[2] = a.z; dst[3] = a.w;
}
template <>
__device__ __forceinline__ void load_n<float, 2>(const float* src, float* dst) {
  const float2 a = *reinterpret_cast<const float2*>(src);
  dst[0] = a.x; dst[1] = a.y;
}
template <>
__device__ __forceinline__ void load_n<__nv_bfloat16, 8>(const __nv_bfloat16* src, float* dst) {
  const uint4 u = *reinterpret_cast<const uint4*>(src);
  dst[0] = bf16_lo(u.x); dst[1] = bf16_hi(u.x); dst[2] = bf16_lo(u.y); dst[3] = bf16_hi(u.y);
  dst[4] = bf16_lo(u.z); dst[5] = bf16_hi(u.z); dst[6] = bf16_lo(u.w); dst[7] = bf16_hi(u.w);
}
template <>
__device__ __forceinline__ void load_n<float, 8>(const float* src, float* dst) {
  const float4 a = *reinterpret_cast<const float4*>(src);
  const float4 b = *reinterpret_cast<const float4*>(src + 4);
  dst[0] = a.x; dst[1] = a.y; dst[2] = a.z; dst[3] = a.w; dst[4] = b.x; dst[5] = b.y; dst[6] = b.z; dst[7] = b.w;
}

// Decode launches (<= 16 rows per sequence, GQA group <= 8): bf16 caches use
// the tensor-core kernel (16 query vectors per CTA), f32 caches the CUDA-core
// kernel (8); prefill chunks the shared-memory kernel (16).
static __host__ __device__ inline bool use_reg_kernel(int rows_per_seq, int G) {
  return rows_per_seq <= 16 && G <= kRegQ;
}
// Query rows per CTA; scratch is sized with the f32 decode grouping, the
// largest number of groups any kernel uses.
static __host__ __device__ inline int rows_per_group(int rows_per_seq, int G, bool bf16) {
  if (!use_reg_kernel(rows_per_seq, G)) return kAttnQ / G;
  return (bf16 ? kAttnQ : kRegQ) / G;
}

// Combine of the splits of one (sequence, group, head): the CTA that finishes
// last merges the partial (m, l, acc) of every split in split order.
// Returns false in every other CTA.
__device__ bool split_combine_arrive(const AttnArgs& a, int slot, int n_active, int* flag) {
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) *flag = (atomicAdd(a.counters + slot, 1) == n_active - 1);
  __syncthreads();
  if (!*flag) return false;
  __threadfence();
  if (threadIdx.x == 0) a.counters[slot] = 0;
  return true;
}

template <typename TO>
__device__ void combine_splits(const AttnArgs& a, const float* all, size_t per, int n_active, int qi, int d,
                               TO* dst) {
  const int hd = a.head_dim;
  float M = -INFINITY;
  for (int s = 0; s < n_active; ++s) M = fmaxf(M, __ldcg(all + s * per + kAttnQ * hd + qi));
  float L = 0.f, O = 0.f;
  for (int s = 0; s < n_active; ++s) {
    const float ms = __ldcg(all + s * per + kAttnQ * hd + qi);
    const float w = (ms == -INFINITY) ? 0.f : expf(ms - M);
    L = fmaf(__ldcg(all + s * per + kAttnQ * hd + kAttnQ + qi), w, L);
    O = fmaf(__ldcg(all + s * per + qi * hd + d), w, O);
  }
  Act<TO>::st(dst, a.o_plane, O / L);
}

// ------------------------------------------------------------------ decode
// K/V of the CTA's positions stream through a ring of kDecStages shared-memory
// stages in 64-position chunks (one 1D bulk copy each for K and V: the rows of
// one (sequence, KV head) are contiguous).  The four warps split the work as
// WQ query pairs x WP position slices (WQ*WP = 4): warp (wq, wp) handles
// queries 2wq, 2wq+1 on positions of slice wp of every chunk, four at a time;
// a lane holds hd/32 dims of its two queries.  Scores are kept in base 2
// (log2 e folded into the query scale) so the softmax uses exp2.
constexpr int kDecStages = 2;
constexpr int kChunkPos = 64;
constexpr int kQPW = 2;                 // query vectors per warp
constexpr float kLog2e = 1.4426950408889634f;

template <typename T, int DPL>
__global__ void __launch_bounds__(128) attn_dec_kernel(const AttnArgs a, int wq_count) {
  constexpr int HD = 32 * DPL;
  constexpr int kRowBytes = HD * sizeof(T);
  constexpr int kStageBytes = kChunkPos * kRowBytes;   // one of K or V
  extern __shared__ __align__(128) uint8_t dsm[];
  __shared__ __align__(8) uint64_t full[kDecStages];
  __shared__ float wm[4][kQPW], wl[4][kQPW];
  __shared__ float wacc[4][kQPW][HD];
  __shared__ int flag;
  uint8_t* ring = dsm;    // [stage][K | V][64][HD]
  griddep_launch();
  griddep_wait();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int WQ = wq_count, WP = 4 / wq_count;
  const int wq = warp % WQ, wp = warp / WQ;
  const int G = a.n_heads / a.n_kv_heads;
  const int RQ = kRegQ / G;
  const int n_qg = (a.rows_per_seq + RQ - 1) / RQ;
  const int split = blockIdx.x, g = blockIdx.y;
  const int sl = blockIdx.z / n_qg, qg = blockIdx.z % n_qg;
  const int seq = a.seq0 + sl;
  const int i0 = qg * RQ;
  const int nrows = min(RQ, a.rows_per_seq - i0);
  const int Q = nrows * G;
  const int base = a.lens[seq] + a.pos_off;
  const int t_cta = min(base + i0 + nrows, a.max_len);
  const int p0 = split * a.split_len;
  if (p0 >= t_cta) return;
  const int p1 = min(p0 + a.split_len, t_cta);
  const int n_active = (t_cta + a.split_len - 1) / a.split_len;
  const int nch = (p1 - p0 + kChunkPos - 1) / kChunkPos;

  const size_t head_off = (static_cast<size_t>(seq) * a.n_kv_heads + g) * a.max_len * HD;
  const T* kb = static_cast<const T*>(a.kc) + head_off;
  const T* vb = static_cast<const T*>(a.vc) + head_off;
  auto issue = [&](int ch) {
    const int st = ch % kDecStages;
    const int pc = p0 + ch * kChunkPos;
    const uint32_t bytes = static_cast<uint32_t>(min(kChunkPos, p1 - pc)) * kRowBytes;
    mbar_arrive_expect_tx(&full[st], 2 * bytes);
    bulk_load(ring + st * 2 * kStageBytes, kb + static_cast<size_t>(pc) * HD, bytes, &full[st]);
    bulk_load(ring + st * 2 * kStageBytes + kStageBytes, vb + static_cast<size_t>(pc) * HD, bytes, &full[st]);
  };
  if (tid == 0) {
    for (int st = 0; st < kDecStages; ++st) mbar_init(&full[st], 1);
    mbar_fence_init();
  }
  __syncthreads();
  if (tid == 0)
    for (int ch = 0; ch < min(kDecStages, nch); ++ch) issue(ch);

  float q[kQPW][DPL], m[kQPW], l[kQPW], acc[kQPW][DPL];
  int lim[kQPW];
#pragma unroll
  for (int u = 0; u < kQPW; ++u) {
    const int qi = wq * kQPW + u;
    lim[u] = -1;
    m[u] = -INFINITY;
    l[u] = 0.f;
#pragma unroll
    for (int e = 0; e < DPL; ++e) {
      q[u][e] = 0.f;
      acc[u][e] = 0.f;
    }
    if (qi < Q) {
      const int ii = qi / G, hh = qi % G;
      const int n = sl * a.rows_per_seq + i0 + ii;
      const float* src = a.q + static_cast<size_t>(n) * a.ld_q + (g * G + hh) * HD + lane * DPL;
#pragma unroll
      for (int e = 0; e < DPL; ++e) q[u][e] = src[e] * (a.scale * kLog2e);
      lim[u] = base + i0 + ii;            // last position row ii may see
    }
  }
  const bool active = wq * kQPW < Q;      // warp-uniform
  const int slice = kChunkPos / WP;

  for (int ch = 0; ch < nch; ++ch) {
    const int st = ch % kDecStages;
    // a wait that runs out only flags the status: every warp must still reach
    // the block barrier below
    mbar_wait(&full[st], (ch / kDecStages) & 1, a.status);
    const T* ks = reinterpret_cast<const T*>(ring + st * 2 * kStageBytes);
    const T* vs = reinterpret_cast<const T*>(ring + st * 2 * kStageBytes + kStageBytes);
    const int pc = p0 + ch * kChunkPos;
    if (active) {
      for (int o0 = wp * slice; o0 < (wp + 1) * slice; o0 += kRegPos) {
        float kr[kRegPos][DPL], vr[kRegPos][DPL];
#pragma unroll
        for (int j = 0; j < kRegPos; ++j) {
          if (pc + o0 + j < p1) {
            load_n<T, DPL>(ks + (o0 + j) * HD + lane * DPL, kr[j]);
            load_n<T, DPL>(vs + (o0 + j) * HD + lane * DPL, vr[j]);
          } else {
#pragma unroll
            for (int e = 0; e < DPL; ++e) { kr[j][e] = 0.f; vr[j][e] = 0.f; }
          }
        }
        float sc[kRegPos][kQPW];
#pragma unroll
        for (int j = 0; j < kRegPos; ++j)
#pragma unroll
          for (int u = 0; u < kQPW; ++u) {
            float t = 0.f;
#pragma unroll
            for (int e = 0; e < DPL; ++e) t = fmaf(q[u][e], kr[j][e], t);
            t = warp_sum(t);
            const int pos = pc + o0 + j;
            sc[j][u] = (pos < p1 && pos <= lim[u]) ? t : -INFINITY;
          }
#pragma unroll
        for (int u = 0; u < kQPW; ++u) {
          float bm = sc[0][u];
#pragma unroll
          for (int j = 1; j < kRegPos; ++j) bm = fmaxf(bm, sc[j][u]);
          if (bm == -INFINITY) continue;      // nothing this row may see here
          const float mn = fmaxf(m[u], bm);
          const float c = (m[u] == -INFINITY) ? 0.f : exp2f(m[u] - mn);
          l[u] *= c;
#pragma unroll
          for (int e = 0; e < DPL; ++e) acc[u][e] *= c;
#pragma unroll
          for (int j = 0; j < kRegPos; ++j) {
            const float pj = exp2f(sc[j][u] - mn);
            l[u] += pj;
#pragma unroll
            for (int e = 0; e < DPL; ++e) acc[u][e] = fmaf(pj, vr[j][e], acc[u][e]);
          }
          m[u] = mn;
        }
      }
    }
    __syncthreads();                      // stage `st` consumed by every warp
    if (tid == 0 && ch + kDecStages < nch) issue(ch + kDecStages);
  }
  // merge the position slices of each query
#pragma unroll
  for (int u = 0; u < kQPW; ++u) {
    if (lane == 0) {
      wm[warp][u] = m[u];
      wl[warp][u] = l[u];
    }
#pragma unroll
    for (int e = 0; e < DPL; ++e) wacc[warp][u][lane * DPL + e] = acc[u][e];
  }
  __syncthreads();
  const int hq_base = g * G;
  const int slot = (sl * n_qg + qg) * a.n_kv_heads + g;
  const size_t per = static_cast<size_t>(kAttnQ) * (HD + 2);
  float* mine = a.part + (static_cast<size_t>(slot) * a.n_splits_max + split) * per;
  for (int idx = tid; idx < Q * HD; idx += 128) {
    const int qi = idx / HD, d = idx % HD;
    const int w0 = qi / kQPW, u = qi % kQPW;           // warps w0 + WQ*p hold query qi
    float M = -INFINITY;
    for (int p = 0; p < WP; ++p) M = fmaxf(M, wm[w0 + WQ * p][u]);
    float Ls = 0.f, O = 0.f;
    for (int p = 0; p < WP; ++p) {
      const float mw = wm[w0 + WQ * p][u];
      const float ww = (mw == -INFINITY) ? 0.f : exp2f(mw - M);
      Ls = fmaf(wl[w0 + WQ * p][u], ww, Ls);
      O = fmaf(wacc[w0 + WQ * p][u][d], ww, O);
    }
    if (n_active == 1) {
      const int ii = qi / G, hh = qi % G;
      const int n = sl * a.rows_per_seq + i0 + ii;
      Act<T>::st(static_cast<T*>(a.o) + static_cast<size_t>(n) * a.ld_o + (hq_base + hh) * HD + d, a.o_plane, O / Ls);
    } else {
      mine[qi * HD + d] = O;
      if (d == 0) {
        mine[kAttnQ * HD + qi] = M;
        mine[kAttnQ * HD + kAttnQ + qi] = Ls;
      }
    }
  }
  if (n_active == 1) return;
  if (!split_combine_arrive(a, slot, n_active, &flag)) return;
  // combine the splits in split order (maxima in base 2)
  const float* all = a.part + static_cast<size_t>(slot) * a.n_splits_max * per;
  __shared__ float cw[kAttnQ];      // 1 / sum of weights, per query
  __shared__ float cM[kAttnQ];
  if (tid < Q) {
    float M = -INFINITY;
    for (int s2 = 0; s2 < n_active; ++s2) M = fmaxf(M, __ldcg(all + s2 * per + kAttnQ * HD + tid));
    float Ls = 0.f;
    for (int s2 = 0; s2 < n_active; ++s2) {
      const float ms = __ldcg(all + s2 * per + kAttnQ * HD + tid);
      Ls = fmaf(__ldcg(all + s2 * per + kAttnQ * HD + kAttnQ + tid), ms == -INFINITY ? 0.f : exp2f(ms - M), Ls);
    }
    cM[tid] = M;
    cw[tid] = 1.f / Ls;
  }
  __syncthreads();
  for (int idx = tid; idx < Q * HD; idx += 128) {
    const int qi = idx / HD, d = idx % HD;
    float O = 0.f;
    for (int s2 = 0; s2 < n_active; ++s2) {
      const float ms = __ldcg(all + s2 * per + kAttnQ * HD + qi);
      O = fmaf(__ldcg(all + s2 * per + qi * HD + d), ms == -INFINITY ? 0.f : exp2f(ms - cM[qi]), O);
    }
    const int ii = qi / G, hh = qi % G;
    const int n = sl * a.rows_per_seq + i0 + ii;
    Act<T>::st(static_cast<T*>(a.o) + static_cast<size_t>(n) * a.ld_o + (hq_base + hh) * HD + d, a.o_plane,
               O * cw[qi]);
  }
}

// ------------------------------------------------------------------ decode, bf16
// Tensor-core decode attention (bf16 cache).  Queries and probabilities enter
// the bf16 MMAs as hi + lo pairs, so only the cache itself is bf16-rounded.
// A CTA covers 16 query rows (the
// block's rows x the GQA heads of one KV head, zero-padded) and its split's
// positions in 64-position chunks, double-buffered by TMA (128-byte swizzle,
// so the fragment loads below are bank-conflict free).  Warp w owns chunk
// positions 16w..16w+15: S = Q K^T with mma.m16n8k16 (Q fragments held in
// registers, K as the column-major operand read straight from the swizzled
// rows), an online softmax over its columns in base 2, then O += P V with the
// accumulator fragments of S reused as the A operand and V fragments loaded
// transposed by ldmatrix.  The four warps merge in shared memory; the splits
// of one (sequence, query group, KV head) form a thread-block cluster and
// each rank combines a slice of the outputs over every rank's (m, l, O)
// through distributed shared memory, in rank order.
constexpr int kMmaQ = 16;

template <int HD>
__global__ void __launch_bounds__(128) attn_mma_kernel(const __grid_constant__ CUtensorMap mk,
                                                       const __grid_constant__ CUtensorMap mv, const AttnArgs a) {
  constexpr int kBoxes = HD / 64;                    // 64-dim TMA boxes per row
  constexpr int kBoxBytes = 64 * 128;                // 64 positions x 128 B
  constexpr int kStage = 2 * kBoxes * kBoxBytes;     // K boxes, then V boxes
  constexpr int kNT = HD / 8;                        // O n-tiles
  extern __shared__ __align__(1024) uint8_t dsm_raw[];
  __shared__ __align__(8) uint64_t full[kDecStages];
  __shared__ float wm[4][kMmaQ], wl[4][kMmaQ];
  __shared__ float cm[kMmaQ], cl[kMmaQ];             // this split's merged max / sum
  __shared__ float ww[4][kMmaQ];                     // per-warp merge weights
  __shared__ float rw[8][kMmaQ], rinv[kMmaQ];        // per-rank combine weights, 1 / sum
  const uint32_t raw = smem_u32(dsm_raw);
  uint8_t* ring = dsm_raw + (((raw + 1023u) & ~1023u) - raw);
  float* wO = reinterpret_cast<float*>(ring);                       // [4][16][HD], after the loop
  float* cO = reinterpret_cast<float*>(ring) + 4 * kMmaQ * HD;      // [16][HD] this split's O
  griddep_launch();
  if (a.dep_wait) {
    if (threadIdx.x == 0) dep_wait(a.dep_wait, a.dep_count, a.status);
    __syncthreads();
  } else {
    griddep_wait();
  }
  cg::cluster_group cluster = cg::this_cluster();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int gq = lane >> 2, tq = lane & 3;           // mma fragment coordinates
  const int G = a.n_heads / a.n_kv_heads;
  const int RQ = kMmaQ / G;
  const int n_qg = (a.rows_per_seq + RQ - 1) / RQ;
  const int S = a.n_splits_max;                      // cluster size
  const int split = blockIdx.x, g = blockIdx.y;
  const int sl = blockIdx.z / n_qg, qg = blockIdx.z % n_qg;
  const int seq = a.seq0 + sl;
  const int i0 = qg * RQ;
  const int nrows = min(RQ, a.rows_per_seq - i0);
  const int Q = nrows * G;
  const int base = a.lens[seq] + a.pos_off;
  // Split `split` of a row at position p covers the 64-position chunks
  // [split*C/S, (split+1)*C/S) of the C = p/64 + 1 chunks that hold positions
  // 0..p: a function of p alone, so a row's result is the same whichever
  // rows share the CTA, and every split gets the same number of chunks (to
  // within one).  The CTA runs the union of its rows' chunk ranges; a chunk
  // outside a row's range is masked for that row and leaves its state exact.
  const int p_min = min(base + i0, a.max_len - 1);
  const int p_max = min(base + i0 + nrows - 1, a.max_len - 1);
  const int c0 = split * (p_min / kChunkPos + 1) / S;
  const int nch = max(0, (split + 1) * (p_max / kChunkPos + 1) / S - c0);
  const int row0 = static_cast<int>(a.kv_row0 + (static_cast<long long>(seq) * a.n_kv_heads + g) * a.max_len);

  auto issue = [&](int ch) {
    const int st = ch % kDecStages;
    const int y = row0 + (c0 + ch) * kChunkPos;
    mbar_arrive_expect_tx(&full[st], kStage);
    for (int b = 0; b < kBoxes; ++b) {
      tma_load_2d(ring + st * kStage + b * kBoxBytes, &mk, b * 64, y, &full[st], 0ull);
      tma_load_2d(ring + st * kStage + (kBoxes + b) * kBoxBytes, &mv, b * 64, y, &full[st], 0ull);
    }
  };
  if (tid == 0) {
    for (int st = 0; st < kDecStages; ++st) mbar_init(&full[st], 1);
    mbar_fence_init();
    tma_prefetch_desc(&mk);
    tma_prefetch_desc(&mv);
  }
  __syncthreads();
  if (tid == 0)
    for (int ch = 0; ch < min(kDecStages, nch); ++ch) issue(ch);

  // Q fragments (rows gq and gq+8), scaled by 1/sqrt(hd) * log2(e), as a
  // bf16 pair hi + lo (two products per K fragment keep 16 bits of q)
  uint32_t qa[HD / 16][4], qb[HD / 16][4];
  int lim0 = -1, lim1 = -1, lo0 = 0, hi0 = 0, lo1 = 0, hi1 = 0;
  {
    const float sc = a.scale * kLog2e;
    const float* qrow[2] = {nullptr, nullptr};
    for (int h = 0; h < 2; ++h) {
      const int qi = gq + 8 * h;
      if (qi < Q) {
        const int ii = qi / G, hh = qi % G;
        const int n = sl * a.rows_per_seq + i0 + ii;
        qrow[h] = a.q + static_cast<size_t>(n) * a.ld_q + (g * G + hh) * HD;
        if (h == 0) lim0 = base + i0 + ii;
        else lim1 = base + i0 + ii;
      }
    }
    // this split's positions of each row: [lo, hi)
    const int C0 = min(max(lim0, 0), a.max_len - 1) / kChunkPos + 1;
    const int C1 = min(max(lim1, 0), a.max_len - 1) / kChunkPos + 1;
    lo0 = split * C0 / S * kChunkPos;
    hi0 = (split + 1) * C0 / S * kChunkPos;
    lo1 = split * C1 / S * kChunkPos;
    hi1 = (split + 1) * C1 / S * kChunkPos;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const float* qr = qrow[r & 1];
        const int col = kk * 16 + (r >> 1) * 8 + 2 * tq;
        qa[kk][r] = 0u;
        qb[kk][r] = 0u;
        if (qr) {
          const float2 v = *reinterpret_cast<const float2*>(qr + col);
          split_bf16x2(v.x * sc, v.y * sc, qa[kk][r], qb[kk][r]);
        }
      }
    }
  }
  float o[kNT][4];
#pragma unroll
  for (int nt = 0; nt < kNT; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) o[nt][e] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;

  for (int ch = 0; ch < nch; ++ch) {
    const int st = ch % kDecStages;
    mbar_wait(&full[st], (ch / kDecStages) & 1, a.status);
    const uint8_t* ks = ring + st * kStage;
    const uint8_t* vs = ks + kBoxes * kBoxBytes;
    const int pc = (c0 + ch) * kChunkPos;
    // S = Q K^T for this warp's 16 positions (two n-tiles of 8)
    float sacc[2][4], slo[2][4];   // q_hi K^T and q_lo K^T: independent MMA chains
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) sacc[nt][e] = slo[nt][e] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
      const int box = (kk * 16) / 64, c = ((kk * 16) % 64) / 8;
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) {
        const int pr = warp * 16 + nt * 8 + gq;                   // row of the chunk
        const uint8_t* rowp = ks + box * kBoxBytes + pr * 128;
        const uint32_t b0 = *reinterpret_cast<const uint32_t*>(rowp + ((c ^ (pr & 7)) << 4) + 4 * tq);
        const uint32_t b1 = *reinterpret_cast<const uint32_t*>(rowp + (((c + 1) ^ (pr & 7)) << 4) + 4 * tq);
        mma_bf16_16816(sacc[nt], qa[kk], b0, b1);
        mma_bf16_16816(slo[nt], qb[kk], b0, b1);
      }
    }
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) sacc[nt][e] += slo[nt][e];
    // mask, online softmax (rows gq and gq+8; columns spread over the 4 lanes tq)
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int pos = pc + warp * 16 + nt * 8 + 2 * tq + e;
        if (!(pos >= lo0 && pos < hi0 && pos <= lim0)) sacc[nt][e] = -INFINITY;
        if (!(pos >= lo1 && pos < hi1 && pos <= lim1)) sacc[nt][2 + e] = -INFINITY;
        mx0 = fmaxf(mx0, sacc[nt][e]);
        mx1 = fmaxf(mx1, sacc[nt][2 + e]);
      }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
    // a row with nothing visible so far keeps its state untouched
    const float c0 = (mn0 == -INFINITY) ? 1.f : (m0 == -INFINITY ? 0.f : exp2f(m0 - mn0));
    const float c1 = (mn1 == -INFINITY) ? 1.f : (m1 == -INFINITY ? 0.f : exp2f(m1 - mn1));
    uint32_t pa[4], pb[4];   // P as a bf16 pair hi + lo
    {
      float pv[2][4];
#pragma unroll
      for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          pv[nt][e] = (sacc[nt][e] == -INFINITY) ? 0.f : exp2f(sacc[nt][e] - mn0);
          pv[nt][2 + e] = (sacc[nt][2 + e] == -INFINITY) ? 0.f : exp2f(sacc[nt][2 + e] - mn1);
        }
      l0 = l0 * c0 + ((pv[0][0] + pv[0][1]) + (pv[1][0] + pv[1][1]));
      l1 = l1 * c1 + ((pv[0][2] + pv[0][3]) + (pv[1][2] + pv[1][3]));
      split_bf16x2(pv[0][0], pv[0][1], pa[0], pb[0]);
      split_bf16x2(pv[0][2], pv[0][3], pa[1], pb[1]);
      split_bf16x2(pv[1][0], pv[1][1], pa[2], pb[2]);
      split_bf16x2(pv[1][2], pv[1][3], pa[3], pb[3]);
    }
    m0 = mn0;
    m1 = mn1;
#pragma unroll
    for (int nt = 0; nt < kNT; ++nt) {
      o[nt][0] *= c0;
      o[nt][1] *= c0;
      o[nt][2] *= c1;
      o[nt][3] *= c1;
    }
    // O += P V: V rows are this warp's 16 positions, read transposed
#pragma unroll
    for (int nt = 0; nt < kNT; nt += 2) {
      const int mi = lane >> 3, rr = lane & 7;
      const int pr = warp * 16 + (mi & 1) * 8 + rr;
      const int db = nt + (mi >> 1);                              // 8-dim block
      const int box = db / 8, c = db % 8;
      const uint32_t addr = smem_u32(vs + box * kBoxBytes + pr * 128 + ((c ^ (pr & 7)) << 4));
      uint32_t r[4];
      ldmatrix_x4_trans(r, addr);
      mma_bf16_16816(o[nt], pa, r[0], r[1]);
      mma_bf16_16816(o[nt], pb, r[0], r[1]);
      mma_bf16_16816(o[nt + 1], pa, r[2], r[3]);
      mma_bf16_16816(o[nt + 1], pb, r[2], r[3]);
    }
    __syncthreads();                      // stage `st` consumed by every warp
    if (tid == 0 && ch + kDecStages < nch) issue(ch + kDecStages);
  }
  // full row sums across the four lanes of a row
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  // merge the four warps into this split's (m, l, O) (the ring is free now);
  // only the Q live query rows are merged
  if (tq == 0) {
    wm[warp][gq] = m0;
    wm[warp][gq + 8] = m1;
    wl[warp][gq] = l0;
    wl[warp][gq + 8] = l1;
  }
#pragma unroll
  for (int nt = 0; nt < kNT; ++nt) {
    const int d = nt * 8 + 2 * tq;
    if (gq < Q) {
      wO[(warp * kMmaQ + gq) * HD + d] = o[nt][0];
      wO[(warp * kMmaQ + gq) * HD + d + 1] = o[nt][1];
    }
    if (gq + 8 < Q) {
      wO[(warp * kMmaQ + gq + 8) * HD + d] = o[nt][2];
      wO[(warp * kMmaQ + gq + 8) * HD + d + 1] = o[nt][3];
    }
  }
  __syncthreads();
  if (tid < Q) {
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) M = fmaxf(M, wm[w][tid]);
    float Ls = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float wt = (wm[w][tid] == -INFINITY) ? 0.f : exp2f(wm[w][tid] - M);
      ww[w][tid] = wt;
      Ls = fmaf(wl[w][tid], wt, Ls);
    }
    cm[tid] = M;
    cl[tid] = Ls;
  }
  __syncthreads();
  for (int idx = tid; idx < Q * HD; idx += 128) {
    const int qi = idx / HD, d = idx % HD;
    float O = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) O = fmaf(wO[(w * kMmaQ + qi) * HD + d], ww[w][qi], O);
    cO[idx] = O;
  }
  // combine the splits of the cluster: per query row, the rank weights
  // 2^(m_r - M) and 1 / sum_r l_r 2^(m_r - M) once; then rank r finishes
  // output elements r*128 + tid, (r + S)*128 + tid, ...
  cluster.sync();
  const float* pO[8];
#pragma unroll
  for (int r = 0; r < 8; ++r) pO[r] = cluster.map_shared_rank(cO, r < S ? r : 0);
  if (tid < Q) {
    float ms[8], ls[8];
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      ms[r] = r < S ? cluster.map_shared_rank(cm, r)[tid] : -INFINITY;
      ls[r] = r < S ? cluster.map_shared_rank(cl, r)[tid] : 0.f;
    }
    float M = ms[0];
#pragma unroll
    for (int r = 1; r < 8; ++r) M = fmaxf(M, ms[r]);
    float Ls = 0.f;
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      const float w = (ms[r] == -INFINITY) ? 0.f : exp2f(ms[r] - M);
      rw[r][tid] = w;
      Ls = fmaf(ls[r], w, Ls);
    }
    rinv[tid] = 1.f / Ls;
  }
  __syncthreads();
  const int hq_base = g * G;
  for (int idx = split * 128 + tid; idx < Q * HD; idx += S * 128) {
    const int qi = idx / HD, d = idx % HD;
    float os[8];
#pragma unroll
    for (int r = 0; r < 8; ++r) os[r] = r < S ? pO[r][idx] : 0.f;
    float O = 0.f;
#pragma unroll
    for (int r = 0; r < 8; ++r)
      if (r < S) O = fmaf(os[r], rw[r][qi], O);
    const int ii = qi / G, hh = qi % G;
    const int n = sl * a.rows_per_seq + i0 + ii;
    Act<__nv_bfloat16>::st(static_cast<__nv_bfloat16*>(a.o) + static_cast<size_t>(n) * a.ld_o + (hq_base + hh) * HD + d,
                           a.o_plane, O * rinv[qi]);
  }
  cluster.sync();   // every rank keeps its shared memory until all have read it
  if (a.dep_signal) {
    __syncthreads();
    if (threadIdx.x == 0) dep_signal(a.dep_signal);
  }
}

// ------------------------------------------------------------------ prefill
template <typename T, typename TO>
__global__ void __launch_bounds__(128, 2) attn_smem_kernel(const AttnArgs a) {
  extern __shared__ float sm[];
  const int hd = a.head_dim;
  float* qs = sm;                                  // [kAttnQ][hd]
  float* ks = qs + kAttnQ * hd;                    // [64][hd+1]
  float* vs = ks + kAttnBlk * (hd + 1);            // [64][hd]
  float* ps = vs + kAttnBlk * hd;                  // [kAttnQ][64]
  float* m_s = ps + kAttnQ * kAttnBlk;             // [kAttnQ]
  float* l_s = m_s + kAttnQ;
  float* al_s = l_s + kAttnQ;
  int* flag = reinterpret_cast<int*>(al_s + kAttnQ);
  griddep_launch();
  griddep_wait();

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = a.n_heads / a.n_kv_heads;
  const int RQ = kAttnQ / G;
  const int n_qg = (a.rows_per_seq + RQ - 1) / RQ;
  const int split = blockIdx.x, g = blockIdx.y;
  const int sl = blockIdx.z / n_qg, qg = blockIdx.z % n_qg;
  const int seq = a.seq0 + sl;
  const int i0 = qg * RQ;
  const int nrows = min(RQ, a.rows_per_seq - i0);
  const int Q = nrows * G;
  const int base = a.lens[seq] + a.pos_off;
  const int t_cta = min(base + i0 + nrows, a.max_len);
  const int p0 = split * a.split_len;
  if (p0 >= t_cta) return;
  const int p1 = min(p0 + a.split_len, t_cta);
  const int n_active = (t_cta + a.split_len - 1) / a.split_len;

  for (int idx = tid; idx < Q * hd; idx += 128) {
    const int qi = idx / hd, d = idx % hd;
    const int ii = qi / G, hh = qi % G;
    const int n = sl * a.rows_per_seq + i0 + ii;
    qs[idx] = a.q[static_cast<size_t>(n) * a.ld_q + (g * G + hh) * hd + d] * a.scale;
  }
  if (tid < kAttnQ) { m_s[tid] = -INFINITY; l_s[tid] = 0.f; }
  const T* kbase = static_cast<const T*>(a.kc) + (static_cast<size_t>(seq) * a.n_kv_heads + g) * a.max_len * hd;
  const T* vbase = static_cast<const T*>(a.vc) + (static_cast<size_t>(seq) * a.n_kv_heads + g) * a.max_len * hd;
  const int qstride = 128 / hd;
  const int d_pv = tid % hd, qpar = tid / hd;
  float o_acc[kAttnQ];
#pragma unroll
  for (int u = 0; u < kAttnQ; ++u) o_acc[u] = 0.f;
  __syncthreads();

  const int c8 = hd / 8;
  for (int b0 = p0; b0 < p1; b0 += kAttnBlk) {
    const int nb = min(kAttnBlk, p1 - b0);
    for (int idx = tid; idx < kAttnBlk * c8; idx += 128) {
      const int r = idx / c8, c = (idx % c8) * 8;
      float kv[8], vv[8];
      if (r < nb) {
        load_n<T, 8>(kbase + static_cast<size_t>(b0 + r) * hd + c, kv);
        load_n<T, 8>(vbase + static_cast<size_t>(b0 + r) * hd + c, vv);
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) { kv[e] = 0.f; vv[e] = 0.f; }
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        ks[r * (hd + 1) + c + e] = kv[e];
        vs[r * hd + c + e] = vv[e];
      }
    }
    __syncthreads();
    {
      const int jj = tid % kAttnBlk, qs0 = tid / kAttnBlk;
      float acc[kAttnQ / 2];
#pragma unroll
      for (int u = 0; u < kAttnQ / 2; ++u) acc[u] = 0.f;
      const float* kr = ks + jj * (hd + 1);
      for (int d = 0; d < hd; ++d) {
        const float kd = kr[d];
#pragma unroll
        for (int u = 0; u < kAttnQ / 2; ++u) {
          const int qi = qs0 + 2 * u;
          if (qi < Q) acc[u] = fmaf(qs[qi * hd + d], kd, acc[u]);
        }
      }
      const int pos = b0 + jj;
#pragma unroll
      for (int u = 0; u < kAttnQ / 2; ++u) {
        const int qi = qs0 + 2 * u;
        if (qi < Q) {
          const int ii = qi / G;
          const bool valid = jj < nb && pos <= base + i0 + ii;
          ps[qi * kAttnBlk + jj] = valid ? acc[u] : -INFINITY;
        }
      }
    }
    __syncthreads();
    for (int qi = warp; qi < Q; qi += 4) {
      const float s0 = ps[qi * kAttnBlk + lane], s1 = ps[qi * kAttnBlk + lane + 32];
      const float bm = warp_max(fmaxf(s0, s1));
      const float m_old = m_s[qi];
      const float m_new = fmaxf(m_old, bm);
      float e0 = 0.f, e1 = 0.f, alpha = 1.f;
      if (m_new != -INFINITY) {
        e0 = expf(s0 - m_new);
        e1 = expf(s1 - m_new);
        alpha = expf(m_old - m_new);
      }
      const float sum = warp_sum(e0 + e1);
      ps[qi * kAttnBlk + lane] = e0;
      ps[qi * kAttnBlk + lane + 32] = e1;
      __syncwarp();
      if (lane == 0) {
        l_s[qi] = l_s[qi] * alpha + sum;
        m_s[qi] = m_new;
        al_s[qi] = alpha;
      }
    }
    __syncthreads();
#pragma unroll
    for (int u = 0; u < kAttnQ; ++u) {
      const int qi = qpar + u * qstride;
      if (qi < Q) {
        float acc = o_acc[u] * al_s[qi];
        const float* pr = ps + qi * kAttnBlk;
        for (int jj = 0; jj < kAttnBlk; ++jj) acc = fmaf(pr[jj], vs[jj * hd + d_pv], acc);
        o_acc[u] = acc;
      }
    }
    __syncthreads();
  }

  const int hq_base = g * G;
  if (n_active == 1) {
#pragma unroll
    for (int u = 0; u < kAttnQ; ++u) {
      const int qi = qpar + u * qstride;
      if (qi < Q) {
        const int ii = qi / G, hh = qi % G;
        const int n = sl * a.rows_per_seq + i0 + ii;
        Act<TO>::st(static_cast<TO*>(a.o) + static_cast<size_t>(n) * a.ld_o + (hq_base + hh) * hd + d_pv, a.o_plane,
                    o_acc[u] / l_s[qi]);
      }
    }
    return;
  }
  const int slot = (sl * n_qg + qg) * a.n_kv_heads + g;
  const size_t per = static_cast<size_t>(kAttnQ) * (hd + 2);
  float* mine = a.part + (static_cast<size_t>(slot) * a.n_splits_max + split) * per;
#pragma unroll
  for (int u = 0; u < kAttnQ; ++u) {
    const int qi = qpar + u * qstride;
    if (qi < Q) mine[qi * hd + d_pv] = o_acc[u];
  }
  if (tid < Q) {
    mine[kAttnQ * hd + tid] = m_s[tid];
    mine[kAttnQ * hd + kAttnQ + tid] = l_s[tid];
  }
  if (!split_combine_arrive(a, slot, n_active, flag)) return;
  const float* all = a.part + static_cast<size_t>(slot) * a.n_splits_max * per;
#pragma unroll
  for (int u = 0; u < kAttnQ; ++u) {
    const int qi = qpar + u * qstride;
    if (qi < Q) {
      const int ii = qi / G, hh = qi % G;
      const int n = sl * a.rows_per_seq + i0 + ii;
      combine_splits<TO>(a, all, per, n_active, qi, d_pv,
                         static_cast<TO*>(a.o) + static_cast<size_t>(n) * a.ld_o + (hq_base + hh) * hd + d_pv);
    }
  }
}

static size_t attn_smem(int hd) {
  return sizeof(float) * (kAttnQ * hd + kAttnBlk * (hd + 1) + kAttnBlk * hd + kAttnQ * kAttnBlk + 3 * kAttnQ) + 16;
}

// ------------------------------------------------------------------ prefill, bf16
// Prompt passes have many query rows per (sequence, KV head).  A CTA takes
// 64 query vectors -- four warps of 16 (pass rows x the GQA heads of one KV
// head) -- and walks every 64-position chunk of the cache its rows can see,
// double-buffered by TMA; the four warps share each chunk, so the cache is
// streamed once per 64 query vectors.  Per warp and 32-position half chunk:
// S = Q K^T with the query as a bf16 pair hi + lo (two MMA chains), the
// causal mask (a position is seen by rows at or after it), an online softmax
// in base 2, then O += P V with P as a bf16 pair.  There is no position
// split and no merge: a row's result is its own online softmax over chunks
// 0 .. p/64 in order (a chunk wholly past the row leaves its state exactly
// as it was), whichever rows share the CTA or the pass.
constexpr int kPfWarpQ = 16;   // query vectors per warp (the mma M)

template <int HD>
__global__ void __launch_bounds__(128) attn_pf_kernel(const __grid_constant__ CUtensorMap mk,
                                                      const __grid_constant__ CUtensorMap mv, const AttnArgs a) {
  constexpr int kBoxes = HD / 64;                    // 64-dim TMA boxes per row
  constexpr int kBoxBytes = 64 * 128;                // 64 positions x 128 B
  constexpr int kStage = 2 * kBoxes * kBoxBytes;     // K boxes, then V boxes
  constexpr int kNT = HD / 8;                        // O n-tiles
  extern __shared__ __align__(1024) uint8_t dsm_raw[];
  __shared__ __align__(8) uint64_t full[kDecStages];
  __shared__ int abort_flag;
  const uint32_t raw = smem_u32(dsm_raw);
  uint8_t* ring = dsm_raw + (((raw + 1023u) & ~1023u) - raw);
  griddep_launch();
  griddep_wait();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int gq = lane >> 2, tq = lane & 3;           // mma fragment coordinates
  const int G = a.n_heads / a.n_kv_heads;
  const int RW = kPfWarpQ / G;                       // pass rows per warp
  const int RC = 4 * RW;                             // pass rows per CTA
  const int g = blockIdx.x;
  const int n_grp = (a.rows_per_seq + RC - 1) / RC;
  const int grp = n_grp - 1 - static_cast<int>(blockIdx.y);   // longest prefixes first
  const int sl = blockIdx.z, seq = a.seq0 + sl;
  const int base = a.lens[seq] + a.pos_off;          // position of pass row 0
  const int i0 = grp * RC;
  const int nrows = min(RC, a.rows_per_seq - i0);
  const int p_max = min(base + i0 + nrows - 1, a.max_len - 1);
  const int nch = p_max / kChunkPos + 1;
  // chunks this warp's rows can see (0 if it has no row)
  const int wr = min(RW, nrows - warp * RW);
  const int w_nch = wr > 0 ? min(base + i0 + warp * RW + wr - 1, a.max_len - 1) / kChunkPos + 1 : 0;
  const int row0 = static_cast<int>(a.kv_row0 + (static_cast<long long>(seq) * a.n_kv_heads + g) * a.max_len);

  auto issue = [&](int ch) {
    const int st = ch % kDecStages;
    const int y = row0 + ch * kChunkPos;
    mbar_arrive_expect_tx(&full[st], kStage);
    for (int b = 0; b < kBoxes; ++b) {
      tma_load_2d(ring + st * kStage + b * kBoxBytes, &mk, b * 64, y, &full[st], 0ull);
      tma_load_2d(ring + st * kStage + (kBoxes + b) * kBoxBytes, &mv, b * 64, y, &full[st], 0ull);
    }
  };
  if (tid == 0) {
    for (int st = 0; st < kDecStages; ++st) mbar_init(&full[st], 1);
    mbar_fence_init();
    tma_prefetch_desc(&mk);
    tma_prefetch_desc(&mv);
    abort_flag = 0;
  }
  __syncthreads();
  if (tid == 0)
    for (int ch = 0; ch < min(kDecStages, nch); ++ch) issue(ch);

  // Q fragments of rows gq and gq+8 of this warp, scaled by 1/sqrt(hd) *
  // log2(e), as a bf16 pair hi + lo
  uint32_t qa[HD / 16][4], qb[HD / 16][4];
  int lim0 = -1, lim1 = -1;
  {
    const float sc = a.scale * kLog2e;
    const float* qrow[2] = {nullptr, nullptr};
    for (int h = 0; h < 2; ++h) {
      const int v = warp * kPfWarpQ + gq + 8 * h;
      const int ii = v / G, hh = v % G;
      if (ii < nrows) {
        const int n = sl * a.rows_per_seq + i0 + ii;
        qrow[h] = a.q + static_cast<size_t>(n) * a.ld_q + (g * G + hh) * HD;
        if (h == 0) lim0 = base + i0 + ii;
        else lim1 = base + i0 + ii;
      }
    }
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const float* qr = qrow[r & 1];
        const int col = kk * 16 + (r >> 1) * 8 + 2 * tq;
        qa[kk][r] = 0u;
        qb[kk][r] = 0u;
        if (qr) {
          const float2 v = *reinterpret_cast<const float2*>(qr + col);
          split_bf16x2(v.x * sc, v.y * sc, qa[kk][r], qb[kk][r]);
        }
      }
    }
  }
  float o[kNT][4];
#pragma unroll
  for (int nt = 0; nt < kNT; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) o[nt][e] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;

  int ch = 0;
  for (; ch < nch; ++ch) {
    const int st = ch % kDecStages;
    if (!mbar_wait(&full[st], (ch / kDecStages) & 1, a.status)) abort_flag = 1;
    const uint8_t* ks = ring + st * kStage;
    const uint8_t* vs = ks + kBoxes * kBoxBytes;
    if (ch < w_nch) {
#pragma unroll 1
      for (int hb = 0; hb < 2; ++hb) {
        const int pc = ch * kChunkPos + hb * 32;
        // S = Q K^T for 32 positions (four n-tiles of 8)
        float sacc[4][4], slo[4][4];
#pragma unroll
        for (int nt = 0; nt < 4; ++nt)
#pragma unroll
          for (int e = 0; e < 4; ++e) sacc[nt][e] = slo[nt][e] = 0.f;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const int box = (kk * 16) / 64, c = ((kk * 16) % 64) / 8;
#pragma unroll
          for (int nt = 0; nt < 4; ++nt) {
            const int pr = hb * 32 + nt * 8 + gq;                 // row of the chunk
            const uint8_t* rowp = ks + box * kBoxBytes + pr * 128;
            const uint32_t b0 = *reinterpret_cast<const uint32_t*>(rowp + ((c ^ (pr & 7)) << 4) + 4 * tq);
            const uint32_t b1 = *reinterpret_cast<const uint32_t*>(rowp + (((c + 1) ^ (pr & 7)) << 4) + 4 * tq);
            mma_bf16_16816(sacc[nt], qa[kk], b0, b1);
            mma_bf16_16816(slo[nt], qb[kk], b0, b1);
          }
        }
        float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
        for (int nt = 0; nt < 4; ++nt)
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const int pos = pc + nt * 8 + 2 * tq + e;
            sacc[nt][e] = pos <= lim0 ? sacc[nt][e] + slo[nt][e] : -INFINITY;
            sacc[nt][2 + e] = pos <= lim1 ? sacc[nt][2 + e] + slo[nt][2 + e] : -INFINITY;
            mx0 = fmaxf(mx0, sacc[nt][e]);
            mx1 = fmaxf(mx1, sacc[nt][2 + e]);
          }
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
        const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
        // a row with nothing visible so far keeps its state untouched
        const float c0 = (mn0 == -INFINITY) ? 1.f : (m0 == -INFINITY ? 0.f : exp2f(m0 - mn0));
        const float c1 = (mn1 == -INFINITY) ? 1.f : (m1 == -INFINITY ? 0.f : exp2f(m1 - mn1));
        uint32_t pa[2][4], pb[2][4];   // P as a bf16 pair hi + lo, per 16-position k-step
        float s0 = 0.f, s1 = 0.f;
#pragma unroll
        for (int k2 = 0; k2 < 2; ++k2) {
          float pv[2][4];
#pragma unroll
          for (int h2 = 0; h2 < 2; ++h2)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const float* sv = sacc[2 * k2 + h2];
              pv[h2][e] = (sv[e] == -INFINITY) ? 0.f : exp2f(sv[e] - mn0);
              pv[h2][2 + e] = (sv[2 + e] == -INFINITY) ? 0.f : exp2f(sv[2 + e] - mn1);
            }
          s0 += (pv[0][0] + pv[0][1]) + (pv[1][0] + pv[1][1]);
          s1 += (pv[0][2] + pv[0][3]) + (pv[1][2] + pv[1][3]);
          split_bf16x2(pv[0][0], pv[0][1], pa[k2][0], pb[k2][0]);
          split_bf16x2(pv[0][2], pv[0][3], pa[k2][1], pb[k2][1]);
          split_bf16x2(pv[1][0], pv[1][1], pa[k2][2], pb[k2][2]);
          split_bf16x2(pv[1][2], pv[1][3], pa[k2][3], pb[k2][3]);
        }
        l0 = l0 * c0 + s0;
        l1 = l1 * c1 + s1;
        m0 = mn0;
        m1 = mn1;
#pragma unroll
        for (int nt = 0; nt < kNT; ++nt) {
          o[nt][0] *= c0;
          o[nt][1] *= c0;
          o[nt][2] *= c1;
          o[nt][3] *= c1;
        }
        // O += P V over the 32 positions, V read transposed
#pragma unroll
        for (int k2 = 0; k2 < 2; ++k2) {
#pragma unroll
          for (int nt = 0; nt < kNT; nt += 2) {
            const int mi = lane >> 3, rr = lane & 7;
            const int pr = hb * 32 + k2 * 16 + (mi & 1) * 8 + rr;
            const int db = nt + (mi >> 1);                          // 8-dim block
            const int box = db / 8, c = db % 8;
            const uint32_t addr = smem_u32(vs + box * kBoxBytes + pr * 128 + ((c ^ (pr & 7)) << 4));
            uint32_t r[4];
            ldmatrix_x4_trans(r, addr);
            mma_bf16_16816(o[nt], pa[k2], r[0], r[1]);
            mma_bf16_16816(o[nt], pb[k2], r[0], r[1]);
            mma_bf16_16816(o[nt + 1], pa[k2], r[2], r[3]);
            mma_bf16_16816(o[nt + 1], pb[k2], r[2], r[3]);
          }
        }
      }
    }
    __syncthreads();                      // stage `st` consumed by every warp
    if (abort_flag) break;
    if (tid == 0 && ch + kDecStages < nch) issue(ch + kDecStages);
  }
  if (abort_flag) {
    // a wait gave up at chunk ch: the copies issued from there on (chunks
    // ch .. ch + kDecStages - 1) must land, or time out, before the CTA exits
    if (tid == 0)
      for (int c = ch; c < min(nch, ch + kDecStages); ++c)
        mbar_wait(&full[c % kDecStages], (c / kDecStages) & 1, a.status);
    return;
  }
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  __nv_bfloat16* out = static_cast<__nv_bfloat16*>(a.o);
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int v = warp * kPfWarpQ + gq + 8 * h;
    const int ii = v / G, hh = v % G;
    if (ii >= nrows) continue;
    const float inv = 1.f / (h == 0 ? l0 : l1);
    const size_t row = static_cast<size_t>(sl * a.rows_per_seq + i0 + ii) * a.ld_o + (g * G + hh) * HD;
#pragma unroll
    for (int nt = 0; nt < kNT; ++nt) {
      const int d = nt * 8 + 2 * tq;
      uint32_t hi, lo;
      split_bf16x2(o[nt][2 * h] * inv, o[nt][2 * h + 1] * inv, hi, lo);
      *reinterpret_cast<uint32_t*>(out + row + d) = hi;
      *reinterpret_cast<uint32_t*>(out + row + d + a.o_plane) = lo;
    }
  }
}

static int n_qgroups(const AttnArgs& a, bool bf16) {
  const int RQ = rows_per_group(a.rows_per_seq, a.n_heads / a.n_kv_heads, bf16);
  return (a.rows_per_seq + RQ - 1) / RQ;
}

size_t attn_partial_floats(const AttnArgs& a) {
  return static_cast<size_t>(a.n_seqs) * n_qgroups(a, false) * a.n_kv_heads * a.n_splits_max * kAttnQ *
         (a.head_dim + 2);
}
int attn_counters(const AttnArgs& a) { return a.n_seqs * n_qgroups(a, false) * a.n_kv_heads; }

template <typename T>
static cudaError_t launch_attn_t(const AttnArgs& a, cudaStream_t s) {
  const bool bf16 = sizeof(T) == 2;
  dim3 grid(a.n_splits_max, a.n_kv_heads, a.n_seqs * n_qgroups(a, bf16));
  if (bf16 && a.prefill && a.n_heads / a.n_kv_heads <= kRegQ) {
    const int G = a.n_heads / a.n_kv_heads;
    const int rc = 4 * (kPfWarpQ / G);
    const dim3 pgrid(a.n_kv_heads, (a.rows_per_seq + rc - 1) / rc, a.n_seqs);
    const size_t smem = 1024 + static_cast<size_t>(kDecStages) * 2 * kChunkPos * a.head_dim * 2;
    static PerDevice pf_attr;
    pf_attr.once([] {
      cudaFuncSetAttribute(attn_pf_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, 160 * 1024);
      cudaFuncSetAttribute(attn_pf_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, 160 * 1024);
    });
    if (a.head_dim == 128) return launch_pdl(attn_pf_kernel<128>, pgrid, dim3(128), smem, s, *a.kmap, *a.vmap, a);
    return launch_pdl(attn_pf_kernel<64>, pgrid, dim3(128), smem, s, *a.kmap, *a.vmap, a);
  }
  if (bf16 && a.n_heads / a.n_kv_heads <= kRegQ) {
    // one cluster of n_splits_max (<= 8) CTAs per (sequence, query group, KV
    // head); decode and prefill chunks alike (16 / G query rows per group)
    const size_t smem = 1024 + static_cast<size_t>(kDecStages) * 2 * kChunkPos * a.head_dim * 2;
    static PerDevice mma_attr;
    mma_attr.once([] {
      cudaFuncSetAttribute(attn_mma_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, 160 * 1024);
      cudaFuncSetAttribute(attn_mma_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, 160 * 1024);
    });
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(128);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = a.n_splits_max;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    if (a.head_dim == 128) return cudaLaunchKernelEx(&cfg, attn_mma_kernel<128>, *a.kmap, *a.vmap, a);
    return cudaLaunchKernelEx(&cfg, attn_mma_kernel<64>, *a.kmap, *a.vmap, a);
  }
  if (use_reg_kernel(a.rows_per_seq, a.n_heads / a.n_kv_heads)) {
    const size_t ring = static_cast<size_t>(kDecStages) * 2 * kChunkPos * a.head_dim * sizeof(T);
    const int qmax = std::min(kRegQ, a.rows_per_seq * (a.n_heads / a.n_kv_heads));
    const int wq = qmax <= kQPW ? 1 : (qmax <= 2 * kQPW ? 2 : 4);
    static PerDevice dec_attr;
    dec_attr.once([] {
      cudaFuncSetAttribute(attn_dec_kernel<T, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize, 160 * 1024);
      cudaFuncSetAttribute(attn_dec_kernel<T, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, 160 * 1024);
    });
    if (a.head_dim == 128) return launch_pdl(attn_dec_kernel<T, 4>, grid, dim3(128), ring, s, a, wq);
    return launch_pdl(attn_dec_kernel<T, 2>, grid, dim3(128), ring, s, a, wq);
  }
  static PerDevice attr;
  attr.once([] { cudaFuncSetAttribute(attn_smem_kernel<T, T>, cudaFuncAttributeMaxDynamicSharedMemorySize, 100 * 1024); });
  return launch_pdl(attn_smem_kernel<T, T>, grid, dim3(128), attn_smem(a.head_dim), s, a);
}

bool attn_chainable(const AttnArgs& a) {
  return a.dtype == DVI_BF16 && !a.prefill && a.n_heads / a.n_kv_heads <= kRegQ;
}

int attn_grid_ctas(const AttnArgs& a) {
  const int G = a.n_heads / a.n_kv_heads;
  if (a.dtype == DVI_BF16 && a.prefill && G <= kRegQ) {
    const int rc = 4 * (kPfWarpQ / G);
    return a.n_kv_heads * ((a.rows_per_seq + rc - 1) / rc) * a.n_seqs;
  }
  return a.n_splits_max * a.n_kv_heads * a.n_seqs * n_qgroups(a, a.dtype == DVI_BF16);
}

cudaError_t launch_attn(const AttnArgs& a, cudaStream_t s) {
  const cudaError_t e = a.dtype == DVI_BF16 ? launch_attn_t<__nv_bfloat16>(a, s) : launch_attn_t<float>(a, s);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace dvi

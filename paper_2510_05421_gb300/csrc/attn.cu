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
// Decode (<= 16 rows per sequence): attn_reg_kernel keeps a query group's
// vectors, scores and accumulators in registers; each warp walks its
// positions four at a time (lane = hd/32 dims, 8-byte coalesced K/V loads),
// reduces the dot products with shuffles and runs an online softmax; the four
// warps merge through shared memory at the end.
// Prefill chunks: attn_smem_kernel stages 64-position K/V blocks in shared
// memory for 16 queries at a time.
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace dvi {

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

// Decode launches (<= 16 rows per sequence, GQA group <= 8) use the register
// kernel with 8 query vectors per CTA; others the shared-memory kernel with 16.
static __host__ __device__ inline bool use_reg_kernel(int rows_per_seq, int G) {
  return rows_per_seq <= 16 && G <= kRegQ;
}
static __host__ __device__ inline int rows_per_group(int rows_per_seq, int G) {
  return (use_reg_kernel(rows_per_seq, G) ? kRegQ : kAttnQ) / G;
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
  DT<TO>::st(dst, O / L);
}

// ------------------------------------------------------------------ decode
template <typename T, typename TO, int DPL>
__global__ void __launch_bounds__(128) attn_reg_kernel(const AttnArgs a) {
  constexpr int HD = 32 * DPL;
  __shared__ float wm[4][kRegQ], wl[4][kRegQ];
  __shared__ float wacc[4][kRegQ][HD];
  __shared__ int flag;
  griddep_launch();
  griddep_wait();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
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

  float q[kRegQ][DPL];
  int lim[kRegQ];
#pragma unroll
  for (int qi = 0; qi < kRegQ; ++qi) {
    lim[qi] = -1;
#pragma unroll
    for (int e = 0; e < DPL; ++e) q[qi][e] = 0.f;
    if (qi < Q) {
      const int ii = qi / G, hh = qi % G;
      const int n = sl * a.rows_per_seq + i0 + ii;
      const float* src = a.q + static_cast<size_t>(n) * a.ld_q + (g * G + hh) * HD + lane * DPL;
#pragma unroll
      for (int e = 0; e < DPL; ++e) q[qi][e] = src[e] * a.scale;
      lim[qi] = base + i0 + ii;          // last position row ii may see
    }
  }
  float m[kRegQ], l[kRegQ], acc[kRegQ][DPL];
#pragma unroll
  for (int qi = 0; qi < kRegQ; ++qi) {
    m[qi] = -INFINITY;
    l[qi] = 0.f;
#pragma unroll
    for (int e = 0; e < DPL; ++e) acc[qi][e] = 0.f;
  }
  const size_t head_off = (static_cast<size_t>(seq) * a.n_kv_heads + g) * a.max_len * HD + lane * DPL;
  const T* kb = static_cast<const T*>(a.kc) + head_off;
  const T* vb = static_cast<const T*>(a.vc) + head_off;

  for (int gp = p0 + warp * kRegPos; gp < p1; gp += 4 * kRegPos) {
    float kr[kRegPos][DPL], vr[kRegPos][DPL];
#pragma unroll
    for (int j = 0; j < kRegPos; ++j) {
      if (gp + j < p1) {
        load_n<T, DPL>(kb + static_cast<size_t>(gp + j) * HD, kr[j]);
        load_n<T, DPL>(vb + static_cast<size_t>(gp + j) * HD, vr[j]);
      } else {
#pragma unroll
        for (int e = 0; e < DPL; ++e) { kr[j][e] = 0.f; vr[j][e] = 0.f; }
      }
    }
    float s[kRegPos][kRegQ];
#pragma unroll
    for (int j = 0; j < kRegPos; ++j)
#pragma unroll
      for (int qi = 0; qi < kRegQ; ++qi) {
        s[j][qi] = -INFINITY;
        if (qi < Q) {                       // warp-uniform
          float t = 0.f;
#pragma unroll
          for (int e = 0; e < DPL; ++e) t = fmaf(q[qi][e], kr[j][e], t);
          t = warp_sum(t);
          if (gp + j < p1 && gp + j <= lim[qi]) s[j][qi] = t;
        }
      }
#pragma unroll
    for (int qi = 0; qi < kRegQ; ++qi) {
      if (qi >= Q) continue;
      float bm = s[0][qi];
#pragma unroll
      for (int j = 1; j < kRegPos; ++j) bm = fmaxf(bm, s[j][qi]);
      if (bm == -INFINITY) continue;      // nothing this row may see here
      const float mn = fmaxf(m[qi], bm);
      const float c = (m[qi] == -INFINITY) ? 0.f : expf(m[qi] - mn);
      l[qi] *= c;
#pragma unroll
      for (int e = 0; e < DPL; ++e) acc[qi][e] *= c;
#pragma unroll
      for (int j = 0; j < kRegPos; ++j) {
        const float pj = expf(s[j][qi] - mn);
        l[qi] += pj;
#pragma unroll
        for (int e = 0; e < DPL; ++e) acc[qi][e] = fmaf(pj, vr[j][e], acc[qi][e]);
      }
      m[qi] = mn;
    }
  }
  // merge the four warps
#pragma unroll
  for (int qi = 0; qi < kRegQ; ++qi) {
    if (lane == 0) {
      wm[warp][qi] = m[qi];
      wl[warp][qi] = l[qi];
    }
#pragma unroll
    for (int e = 0; e < DPL; ++e) wacc[warp][qi][lane * DPL + e] = acc[qi][e];
  }
  __syncthreads();
  const int hq_base = g * G;
  const int slot = (sl * n_qg + qg) * a.n_kv_heads + g;
  const size_t per = static_cast<size_t>(kAttnQ) * (HD + 2);
  float* mine = a.part + (static_cast<size_t>(slot) * a.n_splits_max + split) * per;
  for (int idx = tid; idx < Q * HD; idx += 128) {
    const int qi = idx / HD, d = idx % HD;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) M = fmaxf(M, wm[w][qi]);
    float L = 0.f, O = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float ww = (wm[w][qi] == -INFINITY) ? 0.f : expf(wm[w][qi] - M);
      L = fmaf(wl[w][qi], ww, L);
      O = fmaf(wacc[w][qi][d], ww, O);
    }
    if (n_active == 1) {
      const int ii = qi / G, hh = qi % G;
      const int n = sl * a.rows_per_seq + i0 + ii;
      DT<TO>::st(static_cast<TO*>(a.o) + static_cast<size_t>(n) * a.ld_o + (hq_base + hh) * HD + d, O / L);
    } else {
      mine[qi * HD + d] = O;
      if (d == 0) {
        mine[kAttnQ * HD + qi] = M;
        mine[kAttnQ * HD + kAttnQ + qi] = L;
      }
    }
  }
  if (n_active == 1) return;
  if (!split_combine_arrive(a, slot, n_active, &flag)) return;
  const float* all = a.part + static_cast<size_t>(slot) * a.n_splits_max * per;
  for (int idx = tid; idx < Q * HD; idx += 128) {
    const int qi = idx / HD, d = idx % HD;
    const int ii = qi / G, hh = qi % G;
    const int n = sl * a.rows_per_seq + i0 + ii;
    combine_splits<TO>(a, all, per, n_active, qi, d,
                       static_cast<TO*>(a.o) + static_cast<size_t>(n) * a.ld_o + (hq_base + hh) * HD + d);
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
        DT<TO>::st(static_cast<TO*>(a.o) + static_cast<size_t>(n) * a.ld_o + (hq_base + hh) * hd + d_pv,
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

static int n_qgroups(const AttnArgs& a) {
  const int RQ = rows_per_group(a.rows_per_seq, a.n_heads / a.n_kv_heads);
  return (a.rows_per_seq + RQ - 1) / RQ;
}

size_t attn_partial_floats(const AttnArgs& a) {
  return static_cast<size_t>(a.n_seqs) * n_qgroups(a) * a.n_kv_heads * a.n_splits_max * kAttnQ * (a.head_dim + 2);
}
int attn_counters(const AttnArgs& a) { return a.n_seqs * n_qgroups(a) * a.n_kv_heads; }

template <typename T>
static cudaError_t launch_attn_t(const AttnArgs& a, cudaStream_t s) {
  dim3 grid(a.n_splits_max, a.n_kv_heads, a.n_seqs * n_qgroups(a));
  if (use_reg_kernel(a.rows_per_seq, a.n_heads / a.n_kv_heads)) {
    if (a.head_dim == 128) return launch_pdl(attn_reg_kernel<T, T, 4>, grid, dim3(128), 0, s, a);
    return launch_pdl(attn_reg_kernel<T, T, 2>, grid, dim3(128), 0, s, a);
  }
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(attn_smem_kernel<T, T>, cudaFuncAttributeMaxDynamicSharedMemorySize, 100 * 1024);
    attr = true;
  }
  return launch_pdl(attn_smem_kernel<T, T>, grid, dim3(128), attn_smem(a.head_dim), s, a);
}

cudaError_t launch_attn(const AttnArgs& a, cudaStream_t s) {
  const cudaError_t e = a.dtype == DVI_BF16 ? launch_attn_t<__nv_bfloat16>(a, s) : launch_attn_t<float>(a, s);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace dvi

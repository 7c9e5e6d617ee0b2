// Block-causal multi-query decode attention over the KV cache.
//
// The verify pass of Sec. 3.3 evaluates h_{L,t+i-1} for i = 1..k_spec in one
// pass: query row i of a sequence's block sits at position n+i and sees
// cache positions 0..n+i (the block's own K/V rows were written into the
// cache by the QKV epilogue just before).  Draft and AR passes are the
// one-row case, prefill chunks the many-row case.
//
// One CTA = (position split, KV head, sequence x query group).  It loads its
// split's K/V rows once for every query of the group (all query heads that
// share the KV head, GQA), in 64-position sub-blocks with 16-byte loads,
// keeps an online softmax per query (one warp per query) and accumulates P.V.
// Split boundaries are fixed multiples of `split_len`, independent of the
// number of query rows, and the last CTA to finish a (sequence, group, head)
// combines the splits in split order, so a row's output does not depend on
// how many rows share the launch.
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace dvi {


template <typename T>
__device__ __forceinline__ void load8(const T* src, float* dst);
template <>
__device__ __forceinline__ void load8<__nv_bfloat16>(const __nv_bfloat16* src, float* dst) {
  const uint4 u = *reinterpret_cast<const uint4*>(src);
  dst[0] = bf16_lo(u.x); dst[1] = bf16_hi(u.x); dst[2] = bf16_lo(u.y); dst[3] = bf16_hi(u.y);
  dst[4] = bf16_lo(u.z); dst[5] = bf16_hi(u.z); dst[6] = bf16_lo(u.w); dst[7] = bf16_hi(u.w);
}
template <>
__device__ __forceinline__ void load8<float>(const float* src, float* dst) {
  const float4 a = *reinterpret_cast<const float4*>(src);
  const float4 b = *reinterpret_cast<const float4*>(src + 4);
  dst[0] = a.x; dst[1] = a.y; dst[2] = a.z; dst[3] = a.w; dst[4] = b.x; dst[5] = b.y; dst[6] = b.z; dst[7] = b.w;
}

template <typename T, typename TO>
__global__ void __launch_bounds__(128, 2) attn_kernel(const AttnArgs a) {
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
  const int base = a.lens[seq] + a.pos_off;         // position of block row 0
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
  const int qstride = 128 / hd;                      // threads per dim in P.V
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
        load8<T>(kbase + static_cast<size_t>(b0 + r) * hd + c, kv);
        load8<T>(vbase + static_cast<size_t>(b0 + r) * hd + c, vv);
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
    // scores: thread -> position jj, queries qi = qs0, qs0+2, ...
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
    // online softmax: one warp per query
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
  auto write_out = [&](int qi, float val) {
    const int ii = qi / G, hh = qi % G;
    const int n = sl * a.rows_per_seq + i0 + ii;
    DT<TO>::st(static_cast<TO*>(a.o) + static_cast<size_t>(n) * a.ld_o + (hq_base + hh) * hd + d_pv, val);
  };
  if (n_active == 1) {
#pragma unroll
    for (int u = 0; u < kAttnQ; ++u) {
      const int qi = qpar + u * qstride;
      if (qi < Q) write_out(qi, o_acc[u] / l_s[qi]);
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
  __threadfence();
  __syncthreads();
  if (tid == 0) *flag = (atomicAdd(a.counters + slot, 1) == n_active - 1);
  __syncthreads();
  if (!*flag) return;
  __threadfence();
  if (tid == 0) a.counters[slot] = 0;
  const float* all = a.part + static_cast<size_t>(slot) * a.n_splits_max * per;
#pragma unroll
  for (int u = 0; u < kAttnQ; ++u) {
    const int qi = qpar + u * qstride;
    if (qi < Q) {
      float M = -INFINITY;
      for (int s = 0; s < n_active; ++s) M = fmaxf(M, __ldcg(all + s * per + kAttnQ * hd + qi));
      float L = 0.f, O = 0.f;
      for (int s = 0; s < n_active; ++s) {
        const float ms = __ldcg(all + s * per + kAttnQ * hd + qi);
        const float w = (ms == -INFINITY) ? 0.f : expf(ms - M);
        L = fmaf(__ldcg(all + s * per + kAttnQ * hd + kAttnQ + qi), w, L);
        O = fmaf(__ldcg(all + s * per + qi * hd + d_pv), w, O);
      }
      write_out(qi, O / L);
    }
  }
}

static size_t attn_smem(int hd) {
  return sizeof(float) * (kAttnQ * hd + kAttnBlk * (hd + 1) + kAttnBlk * hd + kAttnQ * kAttnBlk + 3 * kAttnQ) + 16;
}

static int n_qgroups(const AttnArgs& a) {
  const int G = a.n_heads / a.n_kv_heads;
  const int RQ = kAttnQ / G;
  return (a.rows_per_seq + RQ - 1) / RQ;
}

size_t attn_partial_floats(const AttnArgs& a) {
  return static_cast<size_t>(a.n_seqs) * n_qgroups(a) * a.n_kv_heads * a.n_splits_max * kAttnQ * (a.head_dim + 2);
}
int attn_counters(const AttnArgs& a) { return a.n_seqs * n_qgroups(a) * a.n_kv_heads; }

cudaError_t launch_attn(const AttnArgs& a, cudaStream_t s) {
  dim3 grid(a.n_splits_max, a.n_kv_heads, a.n_seqs * n_qgroups(a));
  const size_t smem = attn_smem(a.head_dim);
  if (a.dtype == DVI_BF16) {
    static bool attr = false;
    if (!attr) {
      cudaFuncSetAttribute(attn_kernel<__nv_bfloat16, __nv_bfloat16>,
                           cudaFuncAttributeMaxDynamicSharedMemorySize, 100 * 1024);
      attr = true;
    }
    attn_kernel<__nv_bfloat16, __nv_bfloat16><<<grid, 128, smem, s>>>(a);
  } else {
    static bool attr = false;
    if (!attr) {
      cudaFuncSetAttribute(attn_kernel<float, float>, cudaFuncAttributeMaxDynamicSharedMemorySize, 100 * 1024);
      attr = true;
    }
    attn_kernel<float, float><<<grid, 128, smem, s>>>(a);
  }
  return cudaGetLastError();
}

}  // namespace dvi

// Drafter-head update (Sec. 3.4) on the replay buffer of Sec. 3.3.
//
// Rows are the buffer slots (step, sequence, block position); only rows with
// the valid flag (positions up to and including the first reject) count.
// With u = RMSNorm_final(h_k), l = logits^phi, p = softmax(z),
// z = (W^S + gamma A B) u, q = softmax(l / tau), q1 = softmax(l):
//
//  update_prep      UB[n] = B u_n                               (LoRA down)
//  (projection)     Z = U W^S^T + gamma UB A^T                  (EPI_HEAD)
//  update_rowstats  per row: log-normalisers of z, l/tau, l (one online
//                   pass); KL(p||q), KL(p||q1), H[p], -log p(a), -log p(y*)
//  update_coef      the schedule's term weights at update t, the means that
//                   form the loss, per-row gradient coefficients; the EMA
//                   baseline b moves after the loss is formed
//  update_grad_a    per vocabulary entry v, dL/dz_{n,v} from the closed forms
//                     KL:  p (log p - log q - KL)     CE to a: p - [v=a]
//                     -H:  p (log p + H)
//                   then dA[v] = gamma sum_n G[n][v] UB[n] and the optimizer
//                   step on A[v]; partial sums of G A for dB (old A)
//  update_ga_reduce GA[n] = sum over vocabulary tiles (fixed order)
//  update_grad_b    dB[j][c] = gamma sum_n GA[n][j] u_n[c], optimizer step
//  update_finish    t += 1, empty the buffer
//
// Full-head mode (W^S itself is trained; LoRA factors, if any, stay frozen)
// replaces grad_a .. grad_b by
//  update_g         G[n][v] = dL/dz_{n,v} (the same closed forms)
//  update_gw        dW[v][c] = sum_n G[n][v] u_n[c] and the optimizer step on
//                   W^S (its f32 master when the weights are bf16; the bf16
//                   rounding is written back for the next drafter passes)
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace dvi {

constexpr int kMaxRank = 64;

enum { RS_LSEZ = 0, RS_LSEQ, RS_LSEQ1, RS_KL, RS_KL1, RS_ENT, RS_NLLA, RS_NLLY, RS_N };
enum { CF_KL = 0, CF_KL1, CF_ENT, CF_A, CF_Y, CF_N };
// dev_state floats: 0 t, 1 b, 2 loss, 3 kl, 4 pg, 5 ce, 6 ent, 7 rl, 8 kl1, 9 accept rate,
// 10 skip flag, 11 adam steps
enum { DS_T = 0, DS_B, DS_LOSS, DS_KL, DS_PG, DS_CE, DS_ENT, DS_RL, DS_KL1, DS_ACC, DS_SKIP, DS_ADAM };

__device__ __forceinline__ bool row_valid(const UpdateArgs& a, int n) { return a.log_meta[n * 6] != 0; }

// grid (cap, ceil(r/4)); warp w of CTA (n, y) forms UB[n][4y + w] = B_j . u_n
// (lanes take 4 consecutive features per step, eight steps in flight).
template <typename T>
__global__ void __launch_bounds__(128) update_prep_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  const int n = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j = blockIdx.y * 4 + warp;
  if (j >= a.r) return;
  if (!row_valid(a, n)) {
    if (lane == 0) a.ub[n * a.r + j] = 0.f;
    return;
  }
  const T* u = static_cast<const T*>(a.log_u) + static_cast<size_t>(n) * a.d;
  const float4* br = reinterpret_cast<const float4*>(a.lora_b + static_cast<size_t>(j) * a.d);
  float acc = 0.f;
#pragma unroll 8
  for (int c4 = lane; c4 < a.d / 4; c4 += 32) {
    const float4 b4 = br[c4];
    const T* uc = u + c4 * 4;
    acc = fmaf(b4.x, Act<T>::ld(uc, a.log_plane), acc);
    acc = fmaf(b4.y, Act<T>::ld(uc + 1, a.log_plane), acc);
    acc = fmaf(b4.z, Act<T>::ld(uc + 2, a.log_plane), acc);
    acc = fmaf(b4.w, Act<T>::ld(uc + 3, a.log_plane), acc);
  }
  acc = warp_sum(acc);
  if (lane == 0) a.ub[n * a.r + j] = acc;
}

// (m, s) pairs of log-sum-exp: merge of two partial maxima and sums.
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
  const float M = fmaxf(m, m2);
  if (M == -INFINITY) return;
  s = (m == -INFINITY ? 0.f : s * expf(m - M)) + (m2 == -INFINITY ? 0.f : s2 * expf(m2 - M));
  m = M;
}
__device__ __forceinline__ void lse_add(float& m, float& s, float x) {
  if (x == -INFINITY) return;
  if (x > m) {
    s = (m == -INFINITY ? 0.f : s * expf(m - x)) + 1.f;
    m = x;
  } else {
    s += expf(x - m);
  }
}

// One CTA of 512 threads per buffer row: a single pass for the three
// log-normalisers (online max / sum of exponentials), then one for KL(p||q),
// KL(p||q1) and H[p]; float4 loads when V is a multiple of 4.
__global__ void __launch_bounds__(512) update_rowstats_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  __shared__ float red[16][6];
  const int n = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, nw = blockDim.x >> 5;
  float* rs = a.rowstat + n * RS_N;
  if (!row_valid(a, n)) {
    if (tid < RS_N) rs[tid] = 0.f;
    return;
  }
  const float* z = a.Z + static_cast<size_t>(n) * a.V;
  const float* l = a.log_logits + static_cast<size_t>(n) * a.V;
  const float it = 1.f / a.cfg.tau;
  const bool vec = (a.V & 3) == 0;
  const int nv = vec ? a.V / 4 : a.V;
  float mz = -INFINITY, sz = 0.f, mq = -INFINITY, sq = 0.f, mq1 = -INFINITY, sq1 = 0.f;
  for (int i = tid; i < nv; i += blockDim.x) {
    if (vec) {
      const float4 z4 = reinterpret_cast<const float4*>(z)[i];
      const float4 l4 = reinterpret_cast<const float4*>(l)[i];
      const float zz[4] = {z4.x, z4.y, z4.z, z4.w}, ll[4] = {l4.x, l4.y, l4.z, l4.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        lse_add(mz, sz, zz[e]);
        lse_add(mq, sq, ll[e] * it);
        lse_add(mq1, sq1, ll[e]);
      }
    } else {
      lse_add(mz, sz, z[i]);
      lse_add(mq, sq, l[i] * it);
      lse_add(mq1, sq1, l[i]);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lse_merge(mz, sz, __shfl_xor_sync(0xffffffffu, mz, o), __shfl_xor_sync(0xffffffffu, sz, o));
    lse_merge(mq, sq, __shfl_xor_sync(0xffffffffu, mq, o), __shfl_xor_sync(0xffffffffu, sq, o));
    lse_merge(mq1, sq1, __shfl_xor_sync(0xffffffffu, mq1, o), __shfl_xor_sync(0xffffffffu, sq1, o));
  }
  if (lane == 0) {
    red[warp][0] = mz; red[warp][1] = sz; red[warp][2] = mq; red[warp][3] = sq; red[warp][4] = mq1; red[warp][5] = sq1;
  }
  __syncthreads();
  mz = red[0][0]; sz = red[0][1]; mq = red[0][2]; sq = red[0][3]; mq1 = red[0][4]; sq1 = red[0][5];
  for (int w = 1; w < nw; ++w) {
    lse_merge(mz, sz, red[w][0], red[w][1]);
    lse_merge(mq, sq, red[w][2], red[w][3]);
    lse_merge(mq1, sq1, red[w][4], red[w][5]);
  }
  __syncthreads();
  const float lz = mz + logf(sz), lq = mq + logf(sq), lq1 = mq1 + logf(sq1);
  float kl = 0.f, kl1 = 0.f, ent = 0.f;
  for (int i = tid; i < nv; i += blockDim.x) {
    float zz[4], ll[4];
    int ne = 1;
    if (vec) {
      const float4 z4 = reinterpret_cast<const float4*>(z)[i];
      const float4 l4 = reinterpret_cast<const float4*>(l)[i];
      zz[0] = z4.x; zz[1] = z4.y; zz[2] = z4.z; zz[3] = z4.w;
      ll[0] = l4.x; ll[1] = l4.y; ll[2] = l4.z; ll[3] = l4.w;
      ne = 4;
    } else {
      zz[0] = z[i];
      ll[0] = l[i];
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      if (e < ne) {
        const float lp = zz[e] - lz;
        const float p = expf(lp);
        kl = fmaf(p, lp - (ll[e] * it - lq), kl);
        kl1 = fmaf(p, lp - (ll[e] - lq1), kl1);
        ent = fmaf(-p, lp, ent);
      }
    }
  }
  kl = warp_sum(kl);
  kl1 = warp_sum(kl1);
  ent = warp_sum(ent);
  if (lane == 0) {
    red[warp][0] = kl; red[warp][1] = kl1; red[warp][2] = ent;
  }
  __syncthreads();
  if (tid == 0) {
    kl = 0.f; kl1 = 0.f; ent = 0.f;
    for (int w = 0; w < nw; ++w) {
      kl += red[w][0]; kl1 += red[w][1]; ent += red[w][2];
    }
    const int* meta = a.log_meta + n * 6;
    rs[RS_LSEZ] = lz;
    rs[RS_LSEQ] = lq;
    rs[RS_LSEQ1] = lq1;
    rs[RS_KL] = kl;
    rs[RS_KL1] = kl1;
    rs[RS_ENT] = ent;
    rs[RS_NLLA] = -(z[meta[1]] - lz);
    rs[RS_NLLY] = -(z[meta[5]] - lz);
  }
}

// Weights of the terms at update t (Sec. 3.4's schedule; readings of the
// unnamed constants are the config's).
struct TermW { float kl, pg, ce, ent, rl, beta; };
__device__ TermW term_weights(const dvi_update_config& c, int t) {
  TermW w{0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (c.objective == 1) { w.kl = c.lambda0; return w; }
  if (c.objective == 2) { w.rl = 1.f; return w; }
  if (c.objective == 3) { w.pg = 1.f; return w; }
  if (t < c.t_warmup) {
    w.pg = 0.f;
    w.kl = c.lambda0;
  } else if (t < c.t_warmup + c.t_ramp) {
    const float f = static_cast<float>(t - c.t_warmup) / static_cast<float>(c.t_ramp);
    w.pg = f * c.lambda_pg_max;
    w.kl = c.lambda0 - f * (c.lambda0 - c.lambda_kl_min);
  } else {
    w.pg = c.lambda_pg_max;
    w.kl = c.lambda_kl_min;
  }
  w.ce = c.w_ce;
  w.ent = c.w_ent;
  if (t >= c.t_warmup) {
    const float f = c.t_ramp > 0 ? fminf(1.f, static_cast<float>(t - c.t_warmup) / c.t_ramp) : 1.f;
    w.rl = c.w_rl_max * f;
    w.beta = c.beta_min + (c.beta0 - c.beta_min) * expf(-static_cast<float>(t - c.t_warmup) / c.t_beta);
  }
  return w;
}

__global__ void update_coef_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  if (threadIdx.x != 0) return;
  const int t = static_cast<int>(a.dev_state[DS_T]);
  const float b = a.dev_state[DS_B];
  const TermW w = term_weights(a.cfg, t);
  int N = 0, nP = 0;
  float s_kl = 0.f, s_pg = 0.f, s_ce = 0.f, s_ent = 0.f, s_rl = 0.f, s_kl1 = 0.f, s_r = 0.f;
  for (int n = 0; n < a.cap; ++n) {
    if (!row_valid(a, n)) continue;
    const float* rs = a.rowstat + n * RS_N;
    const float r = static_cast<float>(a.log_meta[n * 6 + 2]);
    ++N;
    s_r += r;
    s_kl += rs[RS_KL];
    s_kl1 += rs[RS_KL1];
    s_ce += rs[RS_NLLY];
    s_ent += rs[RS_ENT];
    s_rl += (r - b) * rs[RS_NLLA];
    if (r == 1.f) { ++nP; s_pg += rs[RS_NLLA]; }
  }
  const float fN = N > 0 ? static_cast<float>(N) : 1.f;
  const float kl = N ? s_kl / fN : 0.f, kl1 = N ? s_kl1 / fN : 0.f, ce = N ? s_ce / fN : 0.f;
  const float ent = N ? s_ent / fN : 0.f, rl = N ? s_rl / fN : 0.f, pg = nP ? s_pg / nP : 0.f;
  const float loss = w.kl * kl + w.pg * pg + w.ce * ce - w.ent * ent + w.rl * rl + w.beta * kl1;
  const bool skip = (N == 0) || !isfinite(loss);
  if (N > 0 && !isfinite(loss)) flag_status(a.status, DVI_DEV_NONFINITE);
  a.dev_state[DS_LOSS] = loss;
  a.dev_state[DS_KL] = kl;
  a.dev_state[DS_PG] = pg;
  a.dev_state[DS_CE] = ce;
  a.dev_state[DS_ENT] = ent;
  a.dev_state[DS_RL] = rl;
  a.dev_state[DS_KL1] = kl1;
  a.dev_state[DS_ACC] = N ? s_r / fN : 0.f;
  a.dev_state[DS_SKIP] = skip ? 1.f : 0.f;
  for (int n = 0; n < a.cap; ++n) {
    float* cf = a.coef + n * CF_N;
    if (skip || !row_valid(a, n)) {
      for (int q = 0; q < CF_N; ++q) cf[q] = 0.f;
      continue;
    }
    const float r = static_cast<float>(a.log_meta[n * 6 + 2]);
    cf[CF_KL] = w.kl / fN;
    cf[CF_KL1] = w.beta / fN;
    cf[CF_ENT] = w.ent / fN;
    cf[CF_A] = (r == 1.f && nP ? w.pg / nP : 0.f) + w.rl * (r - b) / fN;
    cf[CF_Y] = w.ce / fN;
  }
  if (!skip) {
    const float rho = a.cfg.baseline_rho;
    a.dev_state[DS_B] = rho * b + (1.f - rho) * (s_r / fN);
    a.dev_state[DS_ADAM] += 1.f;
  }
}

__device__ __forceinline__ void opt_step(const dvi_update_config& c, float step, float g, float* p, float* m,
                                         float* v) {
  if (c.optimizer == 1) {
    *p -= c.lr * g;
    return;
  }
  const float mn = c.beta1 * *m + (1.f - c.beta1) * g;
  const float vn = c.beta2 * *v + (1.f - c.beta2) * g * g;
  *m = mn;
  *v = vn;
  const float mh = mn / (1.f - powf(c.beta1, step));
  const float vh = vn / (1.f - powf(c.beta2, step));
  *p -= c.lr * mh / (sqrtf(vh) + c.adam_eps);
}

// dL/dz_{n,v} of a valid row n from its row statistics and term coefficients:
//   KL(p||q):  p (log p - log q - KL)      KL(p||q1): p (log p - log q1 - KL1)
//   -H[p]:     p (log p + H)               CE to a / to y*: p - [v = a / y*]
__device__ __forceinline__ float logit_grad(const UpdateArgs& a, int n, int v, float it) {
  const float* rs = a.rowstat + n * RS_N;
  const float* cf = a.coef + n * CF_N;
  const float z = a.Z[static_cast<size_t>(n) * a.V + v];
  const float l = a.log_logits[static_cast<size_t>(n) * a.V + v];
  const float lp = z - rs[RS_LSEZ];
  const float p = expf(lp);
  const float lq = l * it - rs[RS_LSEQ];
  const float lq1 = l - rs[RS_LSEQ1];
  const int* meta = a.log_meta + n * 6;
  return cf[CF_KL] * p * (lp - lq - rs[RS_KL]) + cf[CF_KL1] * p * (lp - lq1 - rs[RS_KL1]) +
         cf[CF_ENT] * p * (lp + rs[RS_ENT]) + cf[CF_A] * (p - (v == meta[1] ? 1.f : 0.f)) +
         cf[CF_Y] * (p - (v == meta[5] ? 1.f : 0.f));
}

// grid = ceil(V/128); dynamic smem: G tile [cap][128] + A tile [128][r]
__global__ void __launch_bounds__(128) update_grad_a_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  extern __shared__ float sm[];
  if (a.dev_state[DS_SKIP] != 0.f) return;
  float* Gs = sm;                              // [cap][128]
  float* As = Gs + static_cast<size_t>(a.cap) * 128;   // [128][r]
  const int tid = threadIdx.x;
  const int v = blockIdx.x * 128 + tid;
  const bool ok = v < a.V;
  const float it = 1.f / a.cfg.tau;
  float dA[kMaxRank];
  float Av[kMaxRank];
  for (int j = 0; j < a.r; ++j) {
    dA[j] = 0.f;
    Av[j] = ok ? a.lora_a[static_cast<size_t>(v) * a.r + j] : 0.f;
    As[tid * a.r + j] = Av[j];
  }
  for (int n = 0; n < a.cap; ++n) {
    float G = 0.f;
    if (ok && row_valid(a, n)) {
      G = logit_grad(a, n, v, it);
      const float* ub = a.ub + n * a.r;
      for (int j = 0; j < a.r; ++j) dA[j] = fmaf(G, ub[j], dA[j]);
    }
    Gs[static_cast<size_t>(n) * 128 + tid] = G;
  }
  __syncthreads();
  // partial G A over this vocabulary tile: pairs (n, j)
  float* part = a.ga_part + static_cast<size_t>(blockIdx.x) * a.cap * a.r;
  for (int idx = tid; idx < a.cap * a.r; idx += 128) {
    const int n = idx / a.r, j = idx % a.r;
    const float* g = Gs + static_cast<size_t>(n) * 128;
    float acc = 0.f;
    for (int q = 0; q < 128; ++q) acc = fmaf(g[q], As[q * a.r + j], acc);
    part[idx] = acc;
  }
  if (!ok) return;
  const float step = a.dev_state[DS_ADAM];
  for (int j = 0; j < a.r; ++j) {
    const float g = a.gamma * dA[j];
    const size_t i = static_cast<size_t>(v) * a.r + j;
    a.grad_a[i] = g;
    opt_step(a.cfg, step, g, a.lora_a + i, a.m_a + i, a.v_a + i);
  }
}

// GA[n][j] = sum over vocabulary tiles of the partials: 256 threads per row,
// thread (part, j) sums tiles t = part (mod parts), then the parts in order.
__global__ void __launch_bounds__(256) update_ga_reduce_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  __shared__ float ps[256];
  if (a.dev_state[DS_SKIP] != 0.f) return;
  const int n = blockIdx.x, tid = threadIdx.x;
  const int parts = 256 / a.r;
  const int j = tid % a.r, part = tid / a.r;
  float acc = 0.f;
  if (part < parts) {
#pragma unroll 4
    for (int t = part; t < a.n_vtiles; t += parts) acc += a.ga_part[(static_cast<size_t>(t) * a.cap + n) * a.r + j];
  }
  ps[tid] = acc;
  __syncthreads();
  if (tid < a.r) {
    float s = 0.f;
    for (int q = 0; q < parts; ++q) s += ps[q * a.r + tid];
    a.ga[n * a.r + tid] = s;
  }
}

// grid (ceil(d/128), ceil(r/4)): thread c of CTA (x, y) forms dB[j][c] for
// the four j = 4y.. of the CTA (one pass over the buffer rows) and steps them.
template <typename T>
__global__ void __launch_bounds__(128) update_grad_b_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  if (a.dev_state[DS_SKIP] != 0.f) return;
  const int c = blockIdx.x * 128 + threadIdx.x;
  const int j0 = blockIdx.y * 4;
  if (c >= a.d) return;
  const float step = a.dev_state[DS_ADAM];
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  const T* u = static_cast<const T*>(a.log_u) + c;
#pragma unroll 4
  for (int n = 0; n < a.cap; ++n) {
    if (!row_valid(a, n)) continue;
    const float un = Act<T>::ld(u + static_cast<size_t>(n) * a.d, a.log_plane);
#pragma unroll
    for (int q = 0; q < 4; ++q)
      if (j0 + q < a.r) acc[q] = fmaf(a.ga[n * a.r + j0 + q], un, acc[q]);
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int j = j0 + q;
    if (j >= a.r) break;
    const float g = a.gamma * acc[q];
    const size_t i = static_cast<size_t>(j) * a.d + c;
    a.grad_b[i] = g;
    opt_step(a.cfg, step, g, a.lora_b + i, a.m_b + i, a.v_b + i);
  }
}

// ---------------------------------------------------------------- full-head mode

// G[n][v] for every buffer row (zeros for rows that are not valid).
// grid = (ceil(V/256), cap), 256 threads.
__global__ void __launch_bounds__(256) update_g_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  if (a.dev_state[DS_SKIP] != 0.f) return;
  const int n = blockIdx.y;
  const int v = blockIdx.x * 256 + threadIdx.x;
  if (v >= a.V) return;
  a.G[static_cast<size_t>(n) * a.V + v] = row_valid(a, n) ? logit_grad(a, n, v, 1.f / a.cfg.tau) : 0.f;
}

constexpr int kGwRows = 16;    // W^S rows per CTA (accumulators per thread: kGwRows x 4)
constexpr int kGwCols = 512;   // W^S columns per CTA: 128 threads x 4 consecutive columns
constexpr int kGwStage = 16;   // buffer rows staged in shared memory per round

// dW = G^T U for a [kGwRows x kGwCols] tile of W^S, then the optimizer step
// on it.  The contraction runs over the buffer rows (N <= 256), so it is a
// few FMAs per W^S entry; the kernel streams W^S (master), m and v once.
// grid = (ceil(V / kGwRows), ceil(d / kGwCols)), 128 threads.
template <typename T>
__global__ void __launch_bounds__(128) update_gw_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  if (a.dev_state[DS_SKIP] != 0.f) return;
  __shared__ float4 us[kGwStage][kGwCols / 4];
  __shared__ float gs[kGwStage][kGwRows];
  const int tid = threadIdx.x;
  const int v0 = blockIdx.x * kGwRows;
  const int cb = blockIdx.y * kGwCols;
  const int c = cb + tid * 4;
  float4 acc[kGwRows];
#pragma unroll
  for (int i = 0; i < kGwRows; ++i) acc[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  const T* U = static_cast<const T*>(a.log_u);
  for (int n0 = 0; n0 < a.cap; n0 += kGwStage) {
    __syncthreads();
    for (int i = tid; i < kGwStage * (kGwCols / 4); i += 128) {
      const int row = i / (kGwCols / 4), col = cb + (i % (kGwCols / 4)) * 4;
      const int n = n0 + row;
      float4 u = make_float4(0.f, 0.f, 0.f, 0.f);
      if (n < a.cap && col < a.d && row_valid(a, n)) {
        const T* src = U + static_cast<size_t>(n) * a.d + col;
        const size_t pl = a.log_plane;
        u = make_float4(Act<T>::ld(src, pl), Act<T>::ld(src + 1, pl), Act<T>::ld(src + 2, pl),
                        Act<T>::ld(src + 3, pl));
      }
      us[row][i % (kGwCols / 4)] = u;
    }
    for (int i = tid; i < kGwStage * kGwRows; i += 128) {
      const int row = i / kGwRows, vv = i % kGwRows;
      const int n = n0 + row, v = v0 + vv;
      gs[row][vv] = (n < a.cap && v < a.V) ? a.G[static_cast<size_t>(n) * a.V + v] : 0.f;
    }
    __syncthreads();
    const int rows = min(kGwStage, a.cap - n0);
    for (int row = 0; row < rows; ++row) {
      const float4 u = us[row][tid];
#pragma unroll
      for (int vv = 0; vv < kGwRows; ++vv) {
        const float g = gs[row][vv];
        acc[vv].x = fmaf(g, u.x, acc[vv].x);
        acc[vv].y = fmaf(g, u.y, acc[vv].y);
        acc[vv].z = fmaf(g, u.z, acc[vv].z);
        acc[vv].w = fmaf(g, u.w, acc[vv].w);
      }
    }
  }
  if (c >= a.d) return;
  const dvi_update_config& cf = a.cfg;
  const float step = a.dev_state[DS_ADAM];
  const float bc1 = 1.f - powf(cf.beta1, step), bc2 = 1.f - powf(cf.beta2, step);
  float* master = a.w_master ? a.w_master : static_cast<float*>(a.w_head);
  // four rows at a time: their loads are issued before any store
#pragma unroll
  for (int g0 = 0; g0 < kGwRows; g0 += 4) {
    float4 p[4], m[4], s[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int v = v0 + g0 + j;
      if (v >= a.V) continue;
      const size_t i = static_cast<size_t>(v) * a.d + c;
      p[j] = *reinterpret_cast<const float4*>(master + i);
      if (cf.optimizer == 0) {
        m[j] = *reinterpret_cast<const float4*>(a.m_w + i);
        s[j] = *reinterpret_cast<const float4*>(a.v_w + i);
      }
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int v = v0 + g0 + j;
      if (v >= a.V) continue;
      const size_t i = static_cast<size_t>(v) * a.d + c;
      const float4 g = acc[g0 + j];
      if (a.keep_grad_w) *reinterpret_cast<float4*>(a.grad_w + i) = g;
      float gv[4] = {g.x, g.y, g.z, g.w};
      float pv[4] = {p[j].x, p[j].y, p[j].z, p[j].w};
      if (cf.optimizer == 1) {
#pragma unroll
        for (int q = 0; q < 4; ++q) pv[q] -= cf.lr * gv[q];
      } else {
        float mv[4] = {m[j].x, m[j].y, m[j].z, m[j].w};
        float sv[4] = {s[j].x, s[j].y, s[j].z, s[j].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          mv[q] = cf.beta1 * mv[q] + (1.f - cf.beta1) * gv[q];
          sv[q] = cf.beta2 * sv[q] + (1.f - cf.beta2) * gv[q] * gv[q];
          pv[q] -= cf.lr * (mv[q] / bc1) / (sqrtf(sv[q] / bc2) + cf.adam_eps);
        }
        *reinterpret_cast<float4*>(a.m_w + i) = make_float4(mv[0], mv[1], mv[2], mv[3]);
        *reinterpret_cast<float4*>(a.v_w + i) = make_float4(sv[0], sv[1], sv[2], sv[3]);
      }
      *reinterpret_cast<float4*>(master + i) = make_float4(pv[0], pv[1], pv[2], pv[3]);
      if (a.w_master) {
        uint2 packed;
        packed.x = pack_bf16x2(pv[0], pv[1]);
        packed.y = pack_bf16x2(pv[2], pv[3]);
        *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(a.w_head) + i) = packed;
      }
    }
  }
}

// master[i] = W^S[i] (bf16 -> f32), once at context creation.
__global__ void update_master_init_kernel(const __nv_bfloat16* w, float* master, size_t n) {
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<size_t>(gridDim.x) * blockDim.x)
    master[i] = __bfloat162float(w[i]);
}

__global__ void update_finish_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  for (int n = blockIdx.x * blockDim.x + threadIdx.x; n < a.cap; n += gridDim.x * blockDim.x) a.log_meta[n * 6] = 0;
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    a.dev_state[DS_T] += 1.f;
    *a.log_step = 0;
    if (a.dev_state[DS_SKIP] == 0.f) a.counters[4] += 1;
  }
}

cudaError_t launch_update_prep(const UpdateArgs& a, cudaStream_t s) {
  if (a.r == 0) return cudaSuccess;
  const dim3 grid(a.cap, (a.r + 3) / 4);
  const cudaError_t e = a.dtype == DVI_BF16 ? launch_pdl(update_prep_kernel<__nv_bfloat16>, grid, dim3(128), 0, s, a)
                                            : launch_pdl(update_prep_kernel<float>, grid, dim3(128), 0, s, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
cudaError_t launch_update_rowstats(const UpdateArgs& a, cudaStream_t s) {
  const cudaError_t e = launch_pdl(update_rowstats_kernel, dim3(a.cap), dim3(512), 0, s, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
cudaError_t launch_update_coef(const UpdateArgs& a, cudaStream_t s) {
  const cudaError_t e = launch_pdl(update_coef_kernel, dim3(1), dim3(32), 0, s, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
cudaError_t launch_update_grad_a(const UpdateArgs& a, cudaStream_t s) {
  if (a.r == 0) return cudaSuccess;
  const size_t smem = sizeof(float) * (static_cast<size_t>(a.cap) * 128 + 128 * a.r);
  // set on every call above 48 KiB (once per update; the attribute is per
  // device, and this keeps it right on whichever device is current)
  if (smem > 48 * 1024)
    cudaFuncSetAttribute(update_grad_a_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  const cudaError_t e = launch_pdl(update_grad_a_kernel, dim3(a.n_vtiles), dim3(128), smem, s, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
cudaError_t launch_update_grad_b(const UpdateArgs& a, cudaStream_t s) {
  if (a.r == 0) return cudaSuccess;
  cudaError_t e = launch_pdl(update_ga_reduce_kernel, dim3(a.cap), dim3(256), 0, s, a);
  if (e != cudaSuccess) return e;
  const dim3 grid((a.d + 127) / 128, (a.r + 3) / 4);
  e = a.dtype == DVI_BF16 ? launch_pdl(update_grad_b_kernel<__nv_bfloat16>, grid, dim3(128), 0, s, a)
                          : launch_pdl(update_grad_b_kernel<float>, grid, dim3(128), 0, s, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
cudaError_t launch_update_full(const UpdateArgs& a, cudaStream_t s) {
  cudaError_t e = launch_pdl(update_g_kernel, dim3((a.V + 255) / 256, a.cap), dim3(256), 0, s, a);
  if (e != cudaSuccess) return e;
  const dim3 grid((a.V + kGwRows - 1) / kGwRows, (a.d + kGwCols - 1) / kGwCols);
  e = a.dtype == DVI_BF16 ? launch_pdl(update_gw_kernel<__nv_bfloat16>, grid, dim3(128), 0, s, a)
                          : launch_pdl(update_gw_kernel<float>, grid, dim3(128), 0, s, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
cudaError_t launch_master_init(const void* w_bf16, float* master, size_t n, cudaStream_t s) {
  update_master_init_kernel<<<1024, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(w_bf16), master, n);
  return cudaGetLastError();
}
cudaError_t launch_update_finish(const UpdateArgs& a, cudaStream_t s) {
  const cudaError_t e = launch_pdl(update_finish_kernel, dim3((a.cap + 255) / 256), dim3(256), 0, s, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace dvi

// Small kernels around the projections: embedding rows, drafter-head
// preparation, and the single-CTA finalize kernels that turn argmax keys
// into drafted / committed tokens.
//
// Every residual row these kernels write is written with its per-128-feature
// sums of squares (the next RMSNorm's statistics) and with x * g, the next
// projection's activation row (the norm gain folded in; bf16 as a hi/lo pair
// of planes).
//
// finalize_verify is the accept/commit/rollback step of Sec. 3.3: with
// y*_{n+i} the verifier's argmax at block row i-1 and t~_i the drafts,
// m = max{i <= K : t~_j = y*_{n+j} for all j <= i}; the step commits
// t~_1..t~_m and, when m < K, the correction y*_{n+m+1} -- min(m+1, K)
// tokens -- and the cache length advances by the same count, which discards
// the KV rows of rejected drafts (they are overwritten later; no data moves).
// With the bonus row (verify rows for t~_1..t~_K and one more for t~_K's
// successor) y*_{n+K+1} exists too, and every step commits m + 1 tokens.
// The replay-buffer tuples of rows 1..min(m+1, K) get r = 1 up to m and r = 0
// at the first reject (Sec. 3.3); later rows stay invalid (counterfactual).
#include "common.cuh"
#include "kernels.h"

namespace dvi {

constexpr int kMaxTiles = 64;   // d <= 8192

// One residual row from the embedding table (128 threads): x, x * g and the
// per-tile sums of squares.  All of the row's loads are issued before any is
// used (one memory round trip), then a single block barrier.
template <typename T>
__device__ void embed_row_block(const T* table, int tok, int d, float* x, const float* g, T* xg, size_t plane,
                                float* ss, int ss_ld, int row, float* red) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nt = d / kTileRows;
  const T* src = table + static_cast<size_t>(tok) * d;
  float v[kMaxTiles], gv[kMaxTiles];
#pragma unroll
  for (int t = 0; t < kMaxTiles; ++t) {
    if (t < nt) {
      v[t] = DT<T>::ld(src + t * kTileRows + tid);
      gv[t] = g[t * kTileRows + tid];
    }
  }
#pragma unroll
  for (int t = 0; t < kMaxTiles; ++t) {
    if (t < nt) {
      const int c = t * kTileRows + tid;
      x[c] = v[t];
      Act<T>::st(xg + c, plane, v[t] * gv[t]);
      const float s = warp_sum(v[t] * v[t]);
      if (lane == 0) red[t * 4 + warp] = s;
    }
  }
  __syncthreads();
  for (int t = tid; t < nt; t += blockDim.x)
    ss[static_cast<size_t>(t) * ss_ld + row] = (red[t * 4] + red[t * 4 + 1]) + (red[t * 4 + 2] + red[t * 4 + 3]);
  __syncthreads();
}

// ---------------------------------------------------------------- embed
template <typename T>
__global__ void __launch_bounds__(128) embed_kernel(const EmbedArgs a) {
  __shared__ float red[kMaxTiles * 4];
  griddep_launch();
  griddep_wait();
  const int row = blockIdx.x;
  int tok = a.tokens[row];
  if (tok < 0 || tok >= a.vocab) {
    if (threadIdx.x == 0) flag_status(a.status, DVI_DEV_BAD_TOKEN);
    tok = 0;
  }
  embed_row_block<T>(static_cast<const T*>(a.table), tok, a.d, a.x + static_cast<size_t>(row) * a.ldx, a.g,
                     static_cast<T*>(a.xg) + static_cast<size_t>(row) * a.ldxg, a.xg_plane, a.ss, a.ss_ld, row,
                     red);
}

cudaError_t launch_embed(const EmbedArgs& a, cudaStream_t s) {
  cudaError_t e = a.dtype == DVI_BF16 ? launch_pdl(embed_kernel<__nv_bfloat16>, dim3(a.rows), dim3(128), 0, s, a)
                                      : launch_pdl(embed_kernel<float>, dim3(a.rows), dim3(128), 0, s, a);
  return e != cudaSuccess ? e : cudaGetLastError();
}

// ---------------------------------------------------------------- head prep
// grid (rows, ceil(r/4) or 1); block 128.  Every CTA computes the row's
// 1/rms; CTA y == 0 logs u and hands the row to the verify stream; each CTA
// computes four entries of B u (one warp each).
// One row of the drafter-head preparation (128 threads): x = h_k, its
// per-tile sums of squares and 1/rms, u = x * rstd * gain into `us` (when
// non-null), and, when `io` is set, u into the replay buffer and h_k handed
// to the verify rows (x, x * g_copy and the sums of squares).
template <typename T>
__device__ void prep_row(const HeadPrepArgs& a, int row, bool io, float* red, float* rstd_s, float* us) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const float* x = a.x + static_cast<size_t>(row) * a.ldx;
  const int nt = a.d / kTileRows;
  float xv[kMaxTiles], gv[kMaxTiles];
#pragma unroll
  for (int t = 0; t < kMaxTiles; ++t)
    if (t < nt) {
      xv[t] = x[t * kTileRows + tid];
      gv[t] = a.gain[t * kTileRows + tid];
    }
  // per-tile sums of squares (also the hand-off's statistics), then 1/rms
#pragma unroll
  for (int t = 0; t < kMaxTiles; ++t)
    if (t < nt) {
      const float s = warp_sum(xv[t] * xv[t]);
      if (lane == 0) red[t * 4 + warp] = s;
    }
  __syncthreads();
  if (tid == 0) {
    float s = 0.f;
    for (int t = 0; t < nt; ++t) s += (red[t * 4] + red[t * 4 + 1]) + (red[t * 4 + 2] + red[t * 4 + 3]);
    *rstd_s = rsqrtf(s / static_cast<float>(a.d) + a.eps);
  }
  __syncthreads();
  const float rstd = *rstd_s;
  if (us) {
#pragma unroll
    for (int t = 0; t < kMaxTiles; ++t)
      if (t < nt) us[t * kTileRows + tid] = xv[t] * rstd * gv[t];
  }
  if (io) {
    T* lu = nullptr;
    if (a.log_u && a.log_enabled) {
      const int ls = *a.log_step;
      if (ls < a.log_cap_steps)
        lu = static_cast<T*>(a.log_u) +
             (static_cast<size_t>(ls) * a.log_rows_per_step + static_cast<size_t>(row) * a.log_row_stride +
              a.log_row_off) * a.d;
    }
    if (lu) {
#pragma unroll
      for (int t = 0; t < kMaxTiles; ++t)
        if (t < nt) Act<T>::st(lu + t * kTileRows + tid, a.log_plane, xv[t] * rstd * gv[t]);
    }
    if (a.x_copy) {
      const int crow = row * a.copy_row_stride + a.copy_row_off;
      float* xc = a.x_copy + static_cast<size_t>(crow) * a.ld_copy;
      T* xgc = static_cast<T*>(a.xg_copy) + static_cast<size_t>(crow) * a.ld_copy;
      float gc[kMaxTiles];
#pragma unroll
      for (int t = 0; t < kMaxTiles; ++t)
        if (t < nt) gc[t] = a.g_copy[t * kTileRows + tid];
#pragma unroll
      for (int t = 0; t < kMaxTiles; ++t)
        if (t < nt) {
          xc[t * kTileRows + tid] = xv[t];
          Act<T>::st(xgc + t * kTileRows + tid, a.xg_copy_plane, xv[t] * gc[t]);
        }
      for (int t = tid; t < nt; t += 128)
        a.ss_copy[static_cast<size_t>(t) * a.ss_copy_ld + crow] =
            (red[t * 4] + red[t * 4 + 1]) + (red[t * 4 + 2] + red[t * 4 + 3]);
    }
  }
}

template <typename T>
__global__ void __launch_bounds__(128) head_prep_kernel(const HeadPrepArgs a) {
  __shared__ float red[kMaxTiles * 4];
  __shared__ float rstd_s;
  __shared__ __align__(16) float us[kMaxTiles * kTileRows];   // u = x * rstd * gain
  griddep_launch();
  griddep_wait();
  const int row = blockIdx.x, grp = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  prep_row<T>(a, row, grp == 0, red, &rstd_s, us);
  if (a.r > 0 && a.bu) {
    __syncthreads();
    const int j = grp * 4 + warp;
    if (j < a.r) {
      // B row j (f32) against u from shared memory, 4 floats per lane per step
      const float4* br = reinterpret_cast<const float4*>(a.lora_b + static_cast<size_t>(j) * a.d);
      const float4* u4 = reinterpret_cast<const float4*>(us);
      float acc = 0.f;
#pragma unroll 8
      for (int c = lane; c < a.d / 4; c += 32) {
        const float4 b = br[c];
        const float4 u = u4[c];
        acc = fmaf(b.x, u.x, acc);
        acc = fmaf(b.y, u.y, acc);
        acc = fmaf(b.z, u.z, acc);
        acc = fmaf(b.w, u.w, acc);
      }
      acc = warp_sum(acc);
      if (lane == 0) a.bu[static_cast<size_t>(row) * a.r + j] = acc;
    }
  }
}

cudaError_t launch_head_prep(const HeadPrepArgs& a, cudaStream_t s) {
  dim3 grid(a.rows, (a.r > 0 && a.bu) ? (a.r + 3) / 4 : 1);
  cudaError_t e = a.dtype == DVI_BF16 ? launch_pdl(head_prep_kernel<__nv_bfloat16>, grid, dim3(128), 0, s, a)
                                      : launch_pdl(head_prep_kernel<float>, grid, dim3(128), 0, s, a);
  return e != cudaSuccess ? e : cudaGetLastError();
}

// ---------------------------------------------------------------- finalize
__device__ __forceinline__ int take_argmax(unsigned long long* slot, int* status) {
  const unsigned long long k = *slot;
  *slot = 0ull;
  if (k == 0ull) {
    flag_status(status, DVI_DEV_NONFINITE);
    return 0;
  }
  return argmax_idx(k);
}

// Embeds each sequence's next input token into the draft residual stream.
template <typename T>
__device__ void embed_rows(const StepState& st, const int* toks, float* red) {
  for (int b = 0; b < st.B; ++b)
    embed_row_block<T>(static_cast<const T*>(st.embed), toks[b], st.d, st.x_dr + static_cast<size_t>(b) * st.d,
                       st.g0, static_cast<T*>(st.xg_dr) + static_cast<size_t>(b) * st.d, st.xg_dr_plane, st.ss_dr,
                       st.ss_dr_ld, b, red);
}

// 16-byte asynchronous copy global -> shared (completes at cp_async_wait).
__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gsrc) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem_dst)), "l"(gsrc) : "memory");
}
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.commit_group;\ncp.async.wait_all;" ::: "memory");
}

// With `prep` set, the drafter-head preparation of the pass (the logged u
// and the hand-off of h_k to the verify rows; the head computed B u itself)
// runs here, for every row before its residual is overwritten by the next
// pass's embedding.  The drafted tokens are read first; with `stage` set the
// next pass's embedding rows are copied into shared memory asynchronously
// while the preparation runs, so their load is off the critical path.
template <typename T>
__global__ void __launch_bounds__(128) finalize_draft_kernel(const StepState st, int j, const HeadPrepArgs hp,
                                                             int prep, int stage) {
  __shared__ int tok_s[64];
  __shared__ float red[kMaxTiles * 4];
  __shared__ float rstd_s;
  extern __shared__ __align__(16) uint8_t emb_raw[];
  griddep_launch();
  griddep_wait();
  for (int b = threadIdx.x; b < st.B; b += blockDim.x) {
    const int t = take_argmax(st.amax + b, st.status);
    st.draft_ids[b * (st.K + 1) + j + 1] = t;
    tok_s[b] = t;
  }
  __syncthreads();
  const bool next = j + 1 < st.Kv;   // the next pass's token (t~_K feeds the bonus row)
  T* emb_s = reinterpret_cast<T*>(emb_raw);
  if (next && stage) {
    const int per_row = st.d * static_cast<int>(sizeof(T)) / 16;
    for (int i = threadIdx.x; i < st.B * per_row; i += blockDim.x) {
      const int b = i / per_row, c = i % per_row;
      int tok = tok_s[b];
      if (tok < 0 || tok >= st.vocab) tok = 0;   // flagged by the embedding below
      cp_async16(emb_raw + static_cast<size_t>(i) * 16,
                 reinterpret_cast<const uint8_t*>(static_cast<const T*>(st.embed) + static_cast<size_t>(tok) * st.d) +
                     static_cast<size_t>(c) * 16);
    }
  }
  if (prep) {
    for (int b = 0; b < hp.rows; ++b) {
      prep_row<T>(hp, b, true, red, &rstd_s, nullptr);
      __syncthreads();
    }
  }
  if (!next) return;
  if (!stage) {
    embed_rows<T>(st, tok_s, red);
    return;
  }
  cp_async_wait();
  __syncthreads();
  for (int b = 0; b < st.B; ++b) {
    if (threadIdx.x == 0 && (tok_s[b] < 0 || tok_s[b] >= st.vocab)) flag_status(st.status, DVI_DEV_BAD_TOKEN);
    embed_row_block<T>(emb_s + static_cast<size_t>(b) * st.d, 0, st.d, st.x_dr + static_cast<size_t>(b) * st.d,
                       st.g0, static_cast<T*>(st.xg_dr) + static_cast<size_t>(b) * st.d, st.xg_dr_plane, st.ss_dr,
                       st.ss_dr_ld, b, red);
  }
}

template <typename T>
__global__ void __launch_bounds__(128) finalize_verify_kernel(const StepState st) {
  __shared__ int tok_s[64];
  __shared__ float red[kMaxTiles * 4];
  griddep_launch();
  griddep_wait();
  const int K = st.K, Kv = st.Kv;
  const int ls = *st.log_step;
  const bool log_ok = st.log_enabled && ls < st.log_cap_steps;
  for (int b = threadIdx.x; b < st.B; b += blockDim.x) {
    int y[16];
    for (int i = 0; i < Kv; ++i) y[i] = take_argmax(st.amax + b * Kv + i, st.status);
    int* dr = st.draft_ids + b * (K + 1);
    int m = 0;
    while (m < K && dr[m + 1] == y[m]) ++m;
    // the correction y*_{n+m+1} exists for m < K, and for m = K with the bonus row
    const int c = m < Kv ? m + 1 : K;
    for (int i = 0; i < Kv; ++i) {
      const int id = i < m ? dr[i + 1] : (i == m ? y[m] : -1);
      st.out_ids[b * Kv + i] = id;
    }
    st.n_committed[b] = c;
    st.n_accepted[b] = m;
    if (log_ok) {
      for (int i = 0; i < K; ++i) {
        int* meta = st.log_meta + (static_cast<size_t>(ls) * st.B * K + b * K + i) * 6;
        meta[0] = i < c;
        meta[1] = dr[i + 1];
        meta[2] = i < m ? 1 : 0;
        meta[3] = i + 1;
        meta[4] = dr[i];
        meta[5] = y[i];
      }
    }
    const int newtok = st.out_ids[b * Kv + c - 1];
    st.lens[b] += c;
    st.pending[b] = newtok;
    dr[0] = newtok;
    tok_s[b] = newtok;
    atomicAdd(reinterpret_cast<unsigned long long*>(st.counters + 2), static_cast<unsigned long long>(m));
    atomicAdd(reinterpret_cast<unsigned long long*>(st.counters + 3), static_cast<unsigned long long>(c));
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    st.counters[0] += 1;
    st.counters[1] += static_cast<long long>(st.B) * K;
    if (st.log_enabled) {
      if (ls < st.log_cap_steps) *st.log_step = ls + 1;
      else flag_status(st.status, DVI_DEV_LOG_FULL);
    }
  }
  embed_rows<T>(st, tok_s, red);
}

template <typename T>
__global__ void __launch_bounds__(128) finalize_ar_kernel(const StepState st) {
  __shared__ int tok_s[64];
  __shared__ float red[kMaxTiles * 4];
  griddep_launch();
  griddep_wait();
  for (int b = threadIdx.x; b < st.B; b += blockDim.x) {
    const int y = take_argmax(st.amax + b, st.status);
    st.out_ids[b] = y;
    st.lens[b] += 1;
    st.pending[b] = y;
    st.draft_ids[b * (st.K + 1)] = y;
    tok_s[b] = y;
  }
  __syncthreads();
  embed_rows<T>(st, tok_s, red);
}

template <typename T>
__global__ void __launch_bounds__(128) finalize_prefill_kernel(const StepState st, int seq, int n_tokens,
                                                               int32_t* first_out) {
  __shared__ float red[kMaxTiles * 4];
  __shared__ int tok;
  griddep_launch();
  griddep_wait();
  if (threadIdx.x == 0) {
    const int y = take_argmax(st.amax, st.status);
    st.lens[seq] = n_tokens;
    st.pending[seq] = y;
    st.draft_ids[seq * (st.K + 1)] = y;
    if (first_out) *first_out = y;
    tok = y;
  }
  __syncthreads();
  embed_row_block<T>(static_cast<const T*>(st.embed), tok, st.d, st.x_dr + static_cast<size_t>(seq) * st.d,
                     st.g0, static_cast<T*>(st.xg_dr) + static_cast<size_t>(seq) * st.d, st.xg_dr_plane, st.ss_dr,
                     st.ss_dr_ld, seq, red);
}

__global__ void reset_seq_kernel(const StepState st, int seq) {
  griddep_launch();
  griddep_wait();
  st.lens[seq] = 0;
}

template <typename K, typename... Args>
static cudaError_t launch1(K kern, cudaStream_t s, Args... args) {
  const cudaError_t e = launch_pdl(kern, dim3(1), dim3(128), 0, s, args...);
  return e != cudaSuccess ? e : cudaGetLastError();
}

constexpr size_t kStageMax = 64 * 1024;   // shared memory for staged embedding rows

cudaError_t launch_finalize_draft(const StepState& st, int j, const HeadPrepArgs* prep, cudaStream_t s) {
  HeadPrepArgs hp{};
  if (prep) hp = *prep;
  const int on = prep ? 1 : 0;
  const size_t esz = st.dtype == DVI_BF16 ? 2 : 4;
  const size_t bytes = static_cast<size_t>(st.B) * st.d * esz;
  const int stage = bytes <= kStageMax ? 1 : 0;
  const size_t smem = stage ? bytes : 0;
  static PerDevice attr;
  attr.once([] {
    cudaFuncSetAttribute(finalize_draft_kernel<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         static_cast<int>(kStageMax));
    cudaFuncSetAttribute(finalize_draft_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         static_cast<int>(kStageMax));
  });
  const cudaError_t e =
      st.dtype == DVI_BF16
          ? launch_pdl(finalize_draft_kernel<__nv_bfloat16>, dim3(1), dim3(128), smem, s, st, j, hp, on, stage)
          : launch_pdl(finalize_draft_kernel<float>, dim3(1), dim3(128), smem, s, st, j, hp, on, stage);
  return e != cudaSuccess ? e : cudaGetLastError();
}
cudaError_t launch_finalize_verify(const StepState& st, cudaStream_t s) {
  return st.dtype == DVI_BF16 ? launch1(finalize_verify_kernel<__nv_bfloat16>, s, st)
                              : launch1(finalize_verify_kernel<float>, s, st);
}
cudaError_t launch_finalize_ar(const StepState& st, cudaStream_t s) {
  return st.dtype == DVI_BF16 ? launch1(finalize_ar_kernel<__nv_bfloat16>, s, st)
                              : launch1(finalize_ar_kernel<float>, s, st);
}
cudaError_t launch_finalize_prefill(const StepState& st, int seq, int n_tokens, int32_t* first_out,
                                    cudaStream_t s) {
  return st.dtype == DVI_BF16 ? launch1(finalize_prefill_kernel<__nv_bfloat16>, s, st, seq, n_tokens, first_out)
                              : launch1(finalize_prefill_kernel<float>, s, st, seq, n_tokens, first_out);
}
cudaError_t launch_reset_seq(const StepState& st, int seq, cudaStream_t s) {
  return launch1(reset_seq_kernel, s, st, seq);
}

}  // namespace dvi

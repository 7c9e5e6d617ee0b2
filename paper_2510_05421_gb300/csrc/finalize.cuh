// The finalize steps of the decode passes (Sec. 3.3) as device functions
// that any 128 threads of a CTA can run together: the standalone finalize
// kernels (one CTA of 128 threads) and the last CTA of a head projection,
// whose 128 epilogue threads run them once every head CTA has published its
// argmax (the fused head -> argmax -> accept -> commit path).  Their block
// barriers are a named barrier of those 128 threads (fin_sync).
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
#pragma once

#include "common.cuh"
#include "kernels.h"

namespace dvi {

constexpr int kMaxTiles = 64;   // d <= 8192
constexpr int kFinThreads = 128;

// Barrier of the 128 threads running a finalize step (the whole CTA of a
// finalize kernel, the epilogue warps of a head projection).
__device__ __forceinline__ void fin_sync() { named_bar(2, kFinThreads); }

// Shared memory of a finalize step.
struct FinSmem {
  int tok_s[64];
  float red[kMaxTiles * 4];
  float rstd_s;
  int last;   // head projection: this CTA is the last to finish
};

// One residual row from the embedding table (128 threads): x, x * g and the
// per-tile sums of squares.  All of the row's loads are issued before any is
// used (one memory round trip), then a single block barrier.
template <typename T, int NT = kMaxTiles>
__device__ void embed_row_block(const T* table, int tok, int d, float* x, const float* g, T* xg, size_t plane,
                                float* ss, int ss_ld, int row, float* red) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nt = d / kTileRows;
  const T* src = table + static_cast<size_t>(tok) * d;
  float v[NT], gv[NT];
#pragma unroll
  for (int t = 0; t < NT; ++t) {
    if (t < nt) {
      v[t] = DT<T>::ld(src + t * kTileRows + tid);
      gv[t] = g[t * kTileRows + tid];
    }
  }
#pragma unroll
  for (int t = 0; t < NT; ++t) {
    if (t < nt) {
      const int c = t * kTileRows + tid;
      x[c] = v[t];
      Act<T>::st(xg + c, plane, v[t] * gv[t]);
      const float s = warp_sum(v[t] * v[t]);
      if (lane == 0) red[t * 4 + warp] = s;
    }
  }
  fin_sync();
  for (int t = tid; t < nt; t += kFinThreads)
    ss[static_cast<size_t>(t) * ss_ld + row] = (red[t * 4] + red[t * 4 + 1]) + (red[t * 4 + 2] + red[t * 4 + 3]);
  fin_sync();
}


// One row of the drafter-head preparation (128 threads): x = h_k, its
// per-tile sums of squares and 1/rms, u = x * rstd * gain into `us` (when
// non-null), and, when `io` is set, u into the replay buffer and h_k handed
// to the verify rows (x, x * g_copy and the sums of squares).
template <typename T, int NT = kMaxTiles>
__device__ void prep_row(const HeadPrepArgs& a, int row, bool io, float* red, float* rstd_s, float* us) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const float* x = a.x + static_cast<size_t>(row) * a.ldx;
  const int nt = a.d / kTileRows;
  float xv[NT], gv[NT];
#pragma unroll
  for (int t = 0; t < NT; ++t)
    if (t < nt) {
      xv[t] = x[t * kTileRows + tid];
      gv[t] = a.gain[t * kTileRows + tid];
    }
  // per-tile sums of squares (also the hand-off's statistics), then 1/rms
#pragma unroll
  for (int t = 0; t < NT; ++t)
    if (t < nt) {
      const float s = warp_sum(xv[t] * xv[t]);
      if (lane == 0) red[t * 4 + warp] = s;
    }
  fin_sync();
  if (tid == 0) {
    float s = 0.f;
    for (int t = 0; t < nt; ++t) s += (red[t * 4] + red[t * 4 + 1]) + (red[t * 4 + 2] + red[t * 4 + 3]);
    *rstd_s = rsqrtf(s / static_cast<float>(a.d) + a.eps);
  }
  fin_sync();
  const float rstd = *rstd_s;
  if (us) {
#pragma unroll
    for (int t = 0; t < NT; ++t)
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
      for (int t = 0; t < NT; ++t)
        if (t < nt) Act<T>::st(lu + t * kTileRows + tid, a.log_plane, xv[t] * rstd * gv[t]);
    }
    if (a.x_copy) {
      const int crow = row * a.copy_row_stride + a.copy_row_off;
      float* xc = a.x_copy + static_cast<size_t>(crow) * a.ld_copy;
      T* xgc = static_cast<T*>(a.xg_copy) + static_cast<size_t>(crow) * a.ld_copy;
      float gc[NT];
#pragma unroll
      for (int t = 0; t < NT; ++t)
        if (t < nt) gc[t] = a.g_copy[t * kTileRows + tid];
#pragma unroll
      for (int t = 0; t < NT; ++t)
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


__device__ __forceinline__ int take_argmax(unsigned long long* slot, int* status) {
  const unsigned long long k = __ldcg(slot);
  *slot = 0ull;
  if (k == 0ull) {
    flag_status(status, DVI_DEV_NONFINITE);
    return 0;
  }
  return argmax_idx(k);
}

// Embeds each sequence's next input token into the draft residual stream.
template <typename T, int NT = kMaxTiles>
__device__ void embed_rows(const StepState& st, const int* toks, float* red) {
  for (int b = 0; b < st.B; ++b)
    embed_row_block<T, NT>(static_cast<const T*>(st.embed), toks[b], st.d, st.x_dr + static_cast<size_t>(b) * st.d,
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
// pass's embedding.  The drafted tokens are read first; with `emb_raw` set
// (B * d elements of shared memory) the next pass's embedding rows are
// copied into shared memory asynchronously while the preparation runs, so
// their load is off the critical path.
template <typename T, int NT = kMaxTiles>
__device__ void finalize_draft_body(const StepState& st, int j, const HeadPrepArgs& hp, int prep, FinSmem& fs,
                                    uint8_t* emb_raw) {
  for (int b = threadIdx.x; b < st.B; b += kFinThreads) {
    const int t = take_argmax(st.amax + b, st.status);
    st.draft_ids[b * (st.K + 1) + j + 1] = t;
    fs.tok_s[b] = t;
  }
  fin_sync();
  const bool next = j + 1 < st.Kv;   // the next pass's token (t~_K feeds the bonus row)
  if (next && emb_raw) {
    const int per_row = st.d * static_cast<int>(sizeof(T)) / 16;
    for (int i = threadIdx.x; i < st.B * per_row; i += kFinThreads) {
      const int b = i / per_row, c = i % per_row;
      int tok = fs.tok_s[b];
      if (tok < 0 || tok >= st.vocab) tok = 0;   // flagged by the embedding below
      cp_async16(emb_raw + static_cast<size_t>(i) * 16,
                 reinterpret_cast<const uint8_t*>(static_cast<const T*>(st.embed) + static_cast<size_t>(tok) * st.d) +
                     static_cast<size_t>(c) * 16);
    }
  }
  if (prep) {
    for (int b = 0; b < hp.rows; ++b) {
      prep_row<T, NT>(hp, b, true, fs.red, &fs.rstd_s, nullptr);
      fin_sync();
    }
  }
  if (!next) return;
  if (!emb_raw) {
    embed_rows<T, NT>(st, fs.tok_s, fs.red);
    return;
  }
  cp_async_wait();
  fin_sync();
  const T* emb_s = reinterpret_cast<const T*>(emb_raw);
  for (int b = 0; b < st.B; ++b) {
    if (threadIdx.x == 0 && (fs.tok_s[b] < 0 || fs.tok_s[b] >= st.vocab)) flag_status(st.status, DVI_DEV_BAD_TOKEN);
    embed_row_block<T, NT>(emb_s + static_cast<size_t>(b) * st.d, 0, st.d, st.x_dr + static_cast<size_t>(b) * st.d,
                       st.g0, static_cast<T*>(st.xg_dr) + static_cast<size_t>(b) * st.d, st.xg_dr_plane, st.ss_dr,
                       st.ss_dr_ld, b, fs.red);
  }
}

// Accept length, commit and rollback, the replay-buffer tuples' metadata,
// and the next pass's embedding (finalize_verify).
template <typename T, int NT = kMaxTiles>
__device__ void finalize_verify_body(const StepState& st, FinSmem& fs) {
  const int K = st.K, Kv = st.Kv;
  const int ls = *st.log_step;
  const bool log_ok = st.log_enabled && ls < st.log_cap_steps;
  for (int b = threadIdx.x; b < st.B; b += kFinThreads) {
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
    fs.tok_s[b] = newtok;
    atomicAdd(reinterpret_cast<unsigned long long*>(st.counters + 2), static_cast<unsigned long long>(m));
    atomicAdd(reinterpret_cast<unsigned long long*>(st.counters + 3), static_cast<unsigned long long>(c));
  }
  fin_sync();
  if (threadIdx.x == 0) {
    st.counters[0] += 1;
    st.counters[1] += static_cast<long long>(st.B) * K;
    if (st.log_enabled) {
      if (ls < st.log_cap_steps) *st.log_step = ls + 1;
      else flag_status(st.status, DVI_DEV_LOG_FULL);
    }
  }
  embed_rows<T, NT>(st, fs.tok_s, fs.red);
}

// Greedy AR: the argmax is the next token of every sequence (finalize_ar).
template <typename T, int NT = kMaxTiles>
__device__ void finalize_ar_body(const StepState& st, FinSmem& fs) {
  for (int b = threadIdx.x; b < st.B; b += kFinThreads) {
    const int y = take_argmax(st.amax + b, st.status);
    st.out_ids[b] = y;
    st.lens[b] += 1;
    st.pending[b] = y;
    st.draft_ids[b * (st.K + 1)] = y;
    fs.tok_s[b] = y;
  }
  fin_sync();
  embed_rows<T, NT>(st, fs.tok_s, fs.red);
}

// The finalize step after a head projection, in the head's last CTA: every
// head CTA's argmax keys are published before the count reaches the grid.
// `smem` is free shared memory of the CTA: the FinSmem, then (f.stage) the
// staged embedding rows.
// NT bounds d / 128 (the per-thread register arrays of the row steps).
template <int NT>
__device__ __forceinline__ void head_finalize(const FinArgs& f, uint8_t* smem, int tid) {
  FinSmem& fs = *reinterpret_cast<FinSmem*>(smem);
  __threadfence();
  fin_sync();
  if (tid == 0) fs.last = atomicAdd(f.ctr, 1) == static_cast<int>(gridDim.x) - 1;
  fin_sync();
  if (!fs.last) return;
  __threadfence();
  if (tid == 0) *f.ctr = 0;
  uint8_t* emb = f.stage ? smem + (sizeof(FinSmem) + 15) / 16 * 16 : nullptr;
  if (f.kind == FIN_DRAFT) finalize_draft_body<__nv_bfloat16, NT>(f.st, f.j, f.hp, f.prep, fs, emb);
  else if (f.kind == FIN_VERIFY) finalize_verify_body<__nv_bfloat16, NT>(f.st, fs);
  else finalize_ar_body<__nv_bfloat16, NT>(f.st, fs);
}

}  // namespace dvi

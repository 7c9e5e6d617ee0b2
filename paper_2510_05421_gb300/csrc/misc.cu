// Small kernels around the projections: embedding rows, drafter-head
// preparation, and the single-CTA finalize kernels that turn argmax keys
// into drafted / committed tokens.
//
// Every residual row these kernels write is written with its per-128-feature
// sums of squares (the next RMSNorm's statistics) and with x * g, the next
// projection's activation row (the norm gain folded in; bf16 as a hi/lo pair
// of planes).
//
// The finalize steps themselves are in finalize.cuh: these kernels run them
// where a head projection cannot (f32, a split head).
#include "finalize.cuh"

namespace dvi {


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

template <typename T>
__global__ void __launch_bounds__(128) finalize_draft_kernel(const StepState st, int j, const HeadPrepArgs hp,
                                                             int prep, int stage) {
  __shared__ FinSmem fs;
  extern __shared__ __align__(16) uint8_t emb_raw[];
  griddep_launch();
  griddep_wait();
  finalize_draft_body<T>(st, j, hp, prep, fs, stage ? emb_raw : nullptr);
}

template <typename T>
__global__ void __launch_bounds__(128) finalize_verify_kernel(const StepState st) {
  __shared__ FinSmem fs;
  griddep_launch();
  griddep_wait();
  finalize_verify_body<T>(st, fs);
}

template <typename T>
__global__ void __launch_bounds__(128) finalize_ar_kernel(const StepState st) {
  __shared__ FinSmem fs;
  griddep_launch();
  griddep_wait();
  finalize_ar_body<T>(st, fs);
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

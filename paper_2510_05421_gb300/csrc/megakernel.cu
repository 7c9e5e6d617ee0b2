// Draft-phase megakernel: the shallow passes of a decode step in one
// persistent launch (Sec. 3.3, draft rollout).
//
// Every CTA (one per SM, all resident) walks the same phase sequence:
//   for each draft pass j:  for each draft layer l < k:
//       QKV -> attention -> O -> gate/up (SwiGLU) -> down
//     then the hand-off of h_{k} to the verify rows and, for j < K, the
//     drafter head z = W^S u + gamma A (B u) with its argmax (the next draft).
// A phase ends with a completion counter: each CTA adds 1 with release
// semantics after its global writes, and the next phase polls the count with
// acquire semantics (bounded; a timeout sets DVI_DEV_TIMEOUT and an abort
// flag that ends every CTA's loop).
//
// Projections are row-split: each CTA owns a contiguous range of 8-row groups
// of a weight matrix's output rows with the whole K, so a row's dot product
// is finished inside one CTA and no partial sums cross CTAs.  The decode rows
// are few (at most kMkMaxRows), so every CTA rebuilds the small input vector
// of a phase itself (residual adds, RMSNorm statistics, attention combine)
// from the previous phase's outputs instead of waiting for one owner.
// Warp 8 streams the CTA's weight tiles (8 rows x 64 columns, 128-byte
// swizzle, 16 per 16 KB stage) and the attention's cached K/V rows through a
// ring of stages, running ahead across phase boundaries, so HBM keeps
// streaming while the CTAs meet at a counter.  Warps 0-7 compute: each warp
// takes 128 of a stage's 1024 columns and multiplies the 8 weight rows
// (B operand, by ldmatrix) with the activations (A operand: rows are the bf16
// hi and lo halves of each decode row, the rest zero) on the warp tensor
// cores with f32 accumulation.  A row's summation order depends on K only, so
// its result does not depend on the CTA count or on how many decode rows
// share the launch.
//
// The attention of a decode row at position pos splits [0, pos] into P equal
// ranges (a function of pos only, so a draft pass and a greedy AR step at the
// same position reduce in the same order).  The ring streams a range in
// chunks of 8192 / hd cached positions, keys then values, each one 16 KB TMA
// box; positions written earlier in this launch and the newest one are
// filled into the stage from global memory and from the pass's own K/V.
// Scores and values run on the warp tensor cores too (each warp owning a
// slice of a chunk's positions, with its own online softmax).
#include "common.cuh"
#include "kernels.h"

namespace dvi {
namespace {

constexpr int kMkThreads = 288;      // warps 0-7 compute, warp 8 streams
constexpr int kMkCompute = 256;
constexpr int kMkWarps = 8;
constexpr int kMkStage = 16384;      // bytes per ring stage
constexpr int kMkStageElems = kMkStage / 2;
constexpr int kMkGroup = 8;          // weight rows per tile (the MMA's N)
constexpr int kMkChunk = 1024;       // weight columns per stage (16 tiles of 64)
constexpr int kMkBar = 3;            // named barrier of the compute warps
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ void cbar() { named_bar(kMkBar, kMkCompute); }

__device__ __forceinline__ int ld_acquire_i32(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Four 8x8 b16 matrices; lane l supplies the row address of matrix l/8, row l%8.
__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], uint32_t saddr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(saddr)
               : "memory");
}

// Contiguous range [lo, hi) of N items for CTA c of n.
__host__ __device__ __forceinline__ void part_range(int N, int c, int n, int& lo, int& hi) {
  lo = static_cast<int>(static_cast<long long>(N) * c / n);
  hi = static_cast<int>(static_cast<long long>(N) * (c + 1) / n);
}
__host__ __device__ __forceinline__ int mk_groups(int N) { return (N + kMkGroup - 1) / kMkGroup; }
__host__ __device__ __forceinline__ int mk_chunks(int K) { return (K + kMkChunk - 1) / kMkChunk; }
// bf16 elements per plane of the A operand: every phase's K rounded up to
// whole 1024-column chunks, plus 8 (the planes start 16 bytes apart modulo
// 128, so one ldmatrix's rows fall in different banks)
__host__ __device__ __forceinline__ int mk_plane(const MkArgs& a) {
  int maxK = a.d > a.F ? a.d : a.F;
  if (a.Hq * a.hd > maxK) maxK = a.Hq * a.hd;
  return mk_chunks(maxK) * kMkChunk + 8;
}

// ------------------------------------------------------------------ layout
// Bytes of the attention scratch (per unit): the q fragments of the lanes
// with live A rows [hd / 16][min(32, 8 G)] x 16 B and the new K and V rows
// (bf16); at the unit's end the warps' partial o [8][G][hd] f32 and (max,
// sum) [8][G][2] f32 overlay them.
__host__ __device__ __forceinline__ size_t mk_att_bytes(int G, int hd) {
  const size_t ql = 8 * G < 32 ? 8 * G : 32;
  const size_t in = static_cast<size_t>(hd / 16) * ql * 16 + 2 * static_cast<size_t>(hd) * 2;
  const size_t out = static_cast<size_t>(kMkWarps) * G * hd * 4 + static_cast<size_t>(kMkWarps) * G * 2 * 4;
  return in > out ? in : out;
}

struct MkLayout {
  size_t ring, bars, act, xw, wacc, gbuf, att, misc, total;
};
__host__ __device__ __forceinline__ size_t al16(size_t x) { return (x + 15) / 16 * 16; }
__host__ __device__ inline MkLayout mk_layout(const MkArgs& a, int ns) {
  MkLayout L;
  size_t off = 0;
  L.ring = off;
  off += static_cast<size_t>(ns) * kMkStage;
  L.bars = off;
  off = al16(off + 2 * static_cast<size_t>(ns) * 8);
  // f32 rows of the residual / attention output: [B][max(d, H_q hd)]
  const int dh = a.d > a.Hq * a.hd ? a.d : a.Hq * a.hd;
  L.act = off;
  off = al16(off + static_cast<size_t>(a.B) * dh * 4);
  // the MMA's A operand: 2 B planes (hi, lo of each decode row) of
  // mk_plane(a) bf16 each, then 16 zero bytes (the A rows past 2 B)
  L.xw = off;
  off = al16(off + static_cast<size_t>(2 * a.B) * mk_plane(a) * 2 + 16);
  L.wacc = off;
  off = al16(off + static_cast<size_t>(kMkWarps) * a.rows_max * a.B * 4);
  L.gbuf = off;
  off = al16(off + static_cast<size_t>(a.rows_max) * a.B * 4);
  // attention scratch (mk_att_bytes); the O phase's combine weights
  // [B][H_q][P] reuse it
  const size_t att = mk_att_bytes(a.Hq / a.Hkv, a.hd);
  const size_t wts = static_cast<size_t>(a.B) * a.Hq * a.P * 4;
  L.att = off;
  off = al16(off + (att > wts ? att : wts));
  // misc: warp keys [8][kMkMaxRows] (u64), rstd, tokens, the wait flag, per-tile
  // sums [B][d/128], B u [B][r]
  L.misc = off;
  off = al16(off + kMkWarps * kMkMaxRows * 8 + 2 * kMkMaxRows * 4 + 16 + static_cast<size_t>(a.B) * (a.d / 128) * 4 +
             static_cast<size_t>(a.B) * a.r * 4);
  L.total = off;
  return L;
}

}  // namespace

size_t mk_smem_bytes(const MkArgs& a, int n_stages) { return mk_layout(a, n_stages).total + 1024; }

int mk_bounds(const MkArgs& a) {
  const int npass = a.mode == MK_DRAFT ? a.Kv : 1;
  const int heads = a.mode == MK_DRAFT ? a.K : 0;
  return npass * 5 * a.k + 2 * heads;
}

int mk_rows_max(const MkArgs& a, int n) {
  const int nqkv = (a.Hq + 2 * a.Hkv) * a.hd;
  auto per = [n](int N) { return (mk_groups(N) + n - 1) / n; };
  int g = per(nqkv);
  g = g > per(a.d) ? g : per(a.d);
  g = g > per(a.F) ? g : per(a.F);
  if (a.mode == MK_DRAFT && a.K > 0) g = g > per(a.V) ? g : per(a.V);
  return g * kMkGroup;
}

namespace {

// ------------------------------------------------------------------ ring
struct Ring {
  uint8_t* base;
  uint64_t* full;
  uint64_t* empty;
  int ns;
  uint32_t it;   // stages consumed so far (the same sequence as the producer's)
};

// Compute side: wait for the next stage's bytes.
__device__ __forceinline__ const uint8_t* ring_acquire(Ring& r, int* status, bool& ok) {
  const int s = static_cast<int>(r.it % r.ns);
  if (!mbar_wait(&r.full[s], (r.it / r.ns) & 1u, status)) ok = false;
  return r.base + static_cast<size_t>(s) * kMkStage;
}
// Compute side: the warp is done with the stage (one arrival per warp).
__device__ __forceinline__ void ring_release(Ring& r) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(&r.empty[r.it % r.ns]);
  ++r.it;
}

// ------------------------------------------------------------------ boundaries
__device__ __forceinline__ void mk_signal(const MkArgs& a, int i) {
  cbar();   // every compute thread's global writes of the phase precede thread 0's release
  if (threadIdx.x == 0) asm volatile("red.release.gpu.global.add.s32 [%0], 1;" ::"l"(a.ctr + i) : "memory");
}

// Wait for every CTA's signal on counter i (acquire by thread 0, then the
// compute barrier).  False when the launch is aborting.
__device__ __forceinline__ bool mk_wait(const MkArgs& a, int i, int* flag_s) {
  if (threadIdx.x == 0) {
    int ok = 1;
    const int n = static_cast<int>(gridDim.x);
    volatile int* abort_flag = a.ctr + a.n_bound;
    if (ld_acquire_i32(a.ctr + i) < n) {
      // the abort flag and the clock only every 64 polls: the counter's
      // completion is seen one load after it happens
      const uint64_t t0 = global_ns();
      for (uint32_t it = 1; ld_acquire_i32(a.ctr + i) < n; ++it) {
        if ((it & 63u) != 0) continue;
        if (*abort_flag) {
          ok = 0;
          break;
        }
        if (global_ns() - t0 > kWaitLimitNs) {
          flag_status(a.status, DVI_DEV_TIMEOUT);
          *abort_flag = 1;
          ok = 0;
          break;
        }
      }
    }
    *flag_s = ok;
  }
  cbar();
  return *flag_s != 0;
}
__device__ __forceinline__ void mk_abort(const MkArgs& a) {
  volatile int* abort_flag = a.ctr + a.n_bound;
  *abort_flag = 1;
}

// Bounded wait on an mbarrier phase that also gives up when the launch is
// aborting (checked every 256 polls).
__device__ __forceinline__ bool mbar_wait_abort(uint64_t* bar, uint32_t parity, const MkArgs& a) {
  if (mbar_try_wait(bar, parity)) return true;
  volatile int* abort_flag = a.ctr + a.n_bound;
  const uint64_t t0 = global_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 255u) == 0 && *abort_flag) return false;
    if (global_ns() - t0 > kWaitLimitNs) {
      flag_status(a.status, DVI_DEV_TIMEOUT);
      *abort_flag = 1;
      return false;
    }
  }
}

}  // namespace
}  // namespace dvi

namespace dvi {
namespace {

// ------------------------------------------------------------------ projections
// Groups [g0, g1) of 8 weight rows, K columns each: a group's stages are its
// 1024-column chunks in order.  Warp w multiplies columns [128 w, 128 w + 128)
// of every stage, 32 columns at a time: one ldmatrix.x4 of the weight tile
// (the B fragments of two k16 steps), one ldmatrix.x4 of the activation
// planes (the A fragments of the same two steps: A row p is plane p -- row
// 2m the hi, 2m + 1 the lo half of decode row m -- and rows past 2 B read
// zeros), two m16n8k16 MMAs into four independent accumulators.  At the
// group's end the hi and lo rows are added (a shuffle) and the warp's partial
// sums of the 8 rows go to wacc[warp][row_local][m].  Tiles past K are
// zero-filled by the copy and meet zero activations.
template <int M>
__device__ __forceinline__ bool gemv_groups(Ring& ring, int K, int g0, int g1, uint32_t xa, int plane, float* wacc,
                                            int rows_max, int* status) {
  constexpr int P = 2 * M;
  const int nkc = mk_chunks(K);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, g = lane >> 2, t = lane & 3;
  const int lrow = lane & 7, lmat = lane >> 3;
  // this lane's A row address at column 0 (plane lrow, or the zero block)
  const uint32_t arow = lrow < P ? xa + static_cast<uint32_t>(lrow * plane * 2 + lmat * 16)
                                 : xa + static_cast<uint32_t>(P * plane * 2);
  const uint32_t astep = lrow < P ? 2u : 0u;   // bytes per column (the zero block stays put)
  bool ok = true;
  for (int gi = g0; gi < g1; ++gi) {
    float d[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i) d[i][0] = d[i][1] = d[i][2] = d[i][3] = 0.f;
    for (int kc = 0; kc < nkc; ++kc) {
      const uint8_t* st = ring_acquire(ring, status, ok);
      if (!ok) return false;
      const uint32_t sb = smem_u32(st) + warp * 2048;
      const uint32_t ab = arow + astep * static_cast<uint32_t>(kc * kMkChunk + warp * 128);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          uint32_t b[4], af[4];
          ldmatrix_x4(b, sb + h * 1024 + lrow * 128 + (((4 * q + lmat) ^ lrow) << 4));
          ldmatrix_x4(af, ab + astep * static_cast<uint32_t>(h * 64 + q * 32));
          const uint32_t a0[4] = {af[0], 0u, af[1], 0u};
          const uint32_t a1[4] = {af[2], 0u, af[3], 0u};
          mma_bf16_16816(d[2 * h + q], a0, b[0], b[1]);
          mma_bf16_16816(d[2 * h + q], a1, b[2], b[3]);
        }
      }
      ring_release(ring);
    }
    // lane (g, t) holds rows 2t, 2t + 1 of the group for A row g
    const float s0 = (d[0][0] + d[1][0]) + (d[2][0] + d[3][0]);
    const float s1 = (d[0][1] + d[1][1]) + (d[2][1] + d[3][1]);
    const float y0 = s0 + __shfl_xor_sync(0xffffffffu, s0, 4);
    const float y1 = s1 + __shfl_xor_sync(0xffffffffu, s1, 4);
    if (g < P && (g & 1) == 0) {
      const int m = g >> 1, rl = (gi - g0) * kMkGroup + 2 * t;
      wacc[(static_cast<size_t>(warp) * rows_max + rl) * M + m] = y0;
      wacc[(static_cast<size_t>(warp) * rows_max + rl + 1) * M + m] = y1;
    }
  }
  return true;
}

// The rows' totals (warps summed in order), handed to `out(row_local, m, v)`;
// the next projection starts after the closing barrier.
template <int M, typename Out>
__device__ __forceinline__ void gemv_finish(float* wacc, int rows_max, int nrows, Out out) {
  cbar();
  for (int rl = threadIdx.x; rl < nrows; rl += kMkCompute) {
#pragma unroll
    for (int m = 0; m < M; ++m) {
      float v = 0.f;
#pragma unroll
      for (int w = 0; w < kMkWarps; ++w) v += wacc[(static_cast<size_t>(w) * rows_max + rl) * M + m];
      out(rl, m, v);
    }
  }
  cbar();
}

// The A operand of a projection over K columns: plane 2m (hi) and 2m + 1
// (lo) of row m of src (row stride ld), as bf16 pairs (columns 2w, 2w + 1 in
// word w of the plane), zero from K to the end of the last 1024-column
// chunk.  `global`: src is in global memory, written by other CTAs in the
// previous phase (four loads per thread in flight).
template <int M>
__device__ __forceinline__ void mk_pack(uint32_t* xw, int plane, const float* src, int K, int ld, bool global) {
  const int nw = mk_chunks(K) * kMkChunk / 2, kw = K / 2, pw = plane / 2;
  for (int w0 = threadIdx.x; w0 < nw; w0 += 4 * kMkCompute) {
    float2 v[4][M];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int w = w0 + u * kMkCompute;
#pragma unroll
      for (int m = 0; m < M; ++m) {
        v[u][m] = make_float2(0.f, 0.f);
        if (w < kw) {
          const float2* p = reinterpret_cast<const float2*>(src + static_cast<size_t>(m) * ld) + w;
          v[u][m] = global ? __ldcg(p) : *p;
        }
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int w = w0 + u * kMkCompute;
      if (w < nw) {
#pragma unroll
        for (int m = 0; m < M; ++m) {
          uint32_t hi, lo;
          split_bf16x2(v[u][m].x, v[u][m].y, hi, lo);
          xw[(2 * m) * pw + w] = hi;
          xw[(2 * m + 1) * pw + w] = lo;
        }
      }
    }
  }
  cbar();
}

// ------------------------------------------------------------------ phase geometry
// QKV rows are the concatenation [W_q; W_k; W_v] (each a multiple of 8 rows):
// the map and first row of group gi.
__device__ __forceinline__ const CUtensorMap* qkv_group(const MkArgs& a, int l, int gi, int& y) {
  const int nq = mk_groups(a.Hq * a.hd), nk = mk_groups(a.Hkv * a.hd);
  const CUtensorMap* m = a.wmaps + l * 7;
  if (gi < nq) {
    y = gi * kMkGroup;
    return m;
  }
  if (gi < nq + nk) {
    y = (gi - nq) * kMkGroup;
    return m + 1;
  }
  y = (gi - nq - nk) * kMkGroup;
  return m + 2;
}

// Attention unit (sequence b, KV head kvh, range p of P) of CTA c, if any,
// and its position range [r0, r1) of [0, pos] at pass j.
struct AttUnit {
  bool on;
  int b, kvh, p, pos, n_b, r0, r1;
};
__device__ __forceinline__ AttUnit att_unit(const MkArgs& a, int j, int c) {
  AttUnit u;
  u.on = c < a.B * a.Hkv * a.P;
  if (!u.on) return u;
  u.b = c / (a.Hkv * a.P);
  u.kvh = (c / a.P) % a.Hkv;
  u.p = c % a.P;
  u.n_b = a.lens[u.b];
  u.pos = u.n_b + j;
  part_range(u.pos + 1, u.p, a.P, u.r0, u.r1);
  return u;
}
// Positions of the chunk [c0, c0 + cn) of a unit that the ring streams: those
// below the sequence's committed length (stable during the launch).
__device__ __forceinline__ int att_stable(const MkArgs& a, const AttUnit& u, int c0, int cn) {
  return max(0, min(c0 + cn, min(u.n_b, a.max_len)) - c0);
}
__device__ __forceinline__ size_t kv_row(const MkArgs& a, int l, int b, int kvh, int x) {
  return ((static_cast<size_t>(l) * a.B + b) * a.Hkv + kvh) * a.max_len + x;
}

}  // namespace
}  // namespace dvi

namespace dvi {
namespace {

// ------------------------------------------------------------------ producer
// Warp 8, lane 0: the CTA's whole stage sequence, in the compute warps' order.
template <int HD>
__device__ void mk_producer(const MkArgs& a, Ring& r, int c, int n) {
  constexpr int CP = kMkStageElems / HD;
  const uint64_t pol = l2_evict_first_policy();
  uint32_t it = 0;
  auto take = [&](int& s) -> bool {
    s = static_cast<int>(it % r.ns);
    return mbar_wait_abort(&r.empty[s], ((it / r.ns) & 1u) ^ 1u, a);
  };
  // one 8-row group of a K-column matrix: its 1024-column chunks, each one
  // box of 16 tiles of 8 rows x 64 (tiles past K and rows past the matrix
  // are zero-filled and counted)
  auto group = [&](const CUtensorMap* map, int K, int y) -> bool {
    const int nkc = mk_chunks(K);
    for (int kc = 0; kc < nkc; ++kc) {
      int s;
      if (!take(s)) return false;
      mbar_arrive_expect_tx(&r.full[s], static_cast<uint32_t>(kMkStage));
      tma_load_3d(r.base + static_cast<size_t>(s) * kMkStage, map, 0, y, kc * (kMkChunk / 64), &r.full[s], pol);
      ++it;
    }
    return true;
  };
  auto groups = [&](const CUtensorMap* map, int K, int g0, int g1) -> bool {
    for (int gi = g0; gi < g1; ++gi)
      if (!group(map, K, gi * kMkGroup)) return false;
    return true;
  };
  // CP cached K or V rows from `row` on: one box of the cache's 3D map
  // ([hd / 64][rows][64], 128-byte swizzled tiles of CP rows x 64; rows past
  // the cache are zero-filled and counted)
  const uint64_t kv_pol = l2_evict_normal_policy();
  auto kv = [&](const CUtensorMap* map, int row) -> bool {
    int s;
    if (!take(s)) return false;
    mbar_arrive_expect_tx(&r.full[s], static_cast<uint32_t>(kMkStage));
    tma_load_3d(r.base + static_cast<size_t>(s) * kMkStage, map, 0, row, 0, &r.full[s], kv_pol);
    ++it;
    return true;
  };
  const int npass = a.mode == MK_DRAFT ? a.Kv : 1;
  const int nqkv = (a.Hq + 2 * a.Hkv) * HD;
  int q0, q1, o0, o1, f0, f1, v0, v1;
  part_range(mk_groups(nqkv), c, n, q0, q1);
  part_range(mk_groups(a.d), c, n, o0, o1);
  part_range(mk_groups(a.F), c, n, f0, f1);
  part_range(mk_groups(a.V), c, n, v0, v1);
  bool ok = true;
  for (int j = 0; j < npass && ok; ++j) {
    const AttUnit u = att_unit(a, j, c);
    for (int l = 0; l < a.k && ok; ++l) {
      const CUtensorMap* m = a.wmaps + l * 7;
      for (int gi = q0; gi < q1 && ok; ++gi) {
        int y;
        const CUtensorMap* map = qkv_group(a, l, gi, y);
        ok = group(map, a.d, y);
      }
      if (u.on) {
        // per chunk: its keys, then its values
        for (int c0 = u.r0; c0 < u.r1 && ok; c0 += CP) {
          const int row = static_cast<int>(kv_row(a, l, u.b, u.kvh, c0));
          ok = kv(a.wmaps + a.k * 7 + 1, row) && kv(a.wmaps + a.k * 7 + 2, row);
        }
      }
      if (ok) ok = groups(m + 3, a.Hq * HD, o0, o1);
      if (ok) ok = groups(m + 4, a.d, f0, f1);
      if (ok) ok = groups(m + 5, a.d, f0, f1);
      if (ok) ok = groups(m + 6, a.F, o0, o1);
    }
    if (ok && a.mode == MK_DRAFT && j < a.K) ok = groups(a.wmaps + a.k * 7, a.d, v0, v1);
  }
  // every issued copy lands before this thread leaves (the CTA's shared
  // memory stays live while any of its threads runs)
  const uint32_t first = it > static_cast<uint32_t>(r.ns) ? it - r.ns : 0u;
  for (uint32_t i = first; i < it; ++i) mbar_wait(&r.full[i % r.ns], (i / r.ns) & 1u, a.status);
}

// ------------------------------------------------------------------ prologues
// act[m][0..d) = the raw residual of row m: xa[m] + xb[m] (written by other
// CTAs in earlier phases) or the embedding of tok[m]; `writer` also stores it
// in xr_out.
// (Loads are issued eight per thread at a time before any result is stored.)
__device__ __forceinline__ void mk_residual(const MkArgs& a, float* act, const float* __restrict__ xa,
                                            const float* __restrict__ xb, const int* tok, float* xr_out,
                                            bool writer) {
  const int d = a.d;
  for (int m = 0; m < a.B; ++m) {
    const __nv_bfloat16* e =
        tok ? static_cast<const __nv_bfloat16*>(a.embed) + static_cast<size_t>(tok[m]) * d : nullptr;
    const size_t base = static_cast<size_t>(m) * d;
    for (int i0 = threadIdx.x; i0 < d; i0 += 8 * kMkCompute) {
      float v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int i = i0 + u * kMkCompute;
        v[u] = 0.f;
        if (i < d) v[u] = e ? __bfloat162float(e[i]) : __ldcg(xa + base + i) + __ldcg(xb + base + i);
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int i = i0 + u * kMkCompute;
        if (i < d) {
          act[base + i] = v[u];
          if (writer) xr_out[base + i] = v[u];
        }
      }
    }
  }
}

// Per-128-feature sums of squares of the act rows (tsum[m][t]) and 1/rms.
__device__ __forceinline__ void mk_rms(const MkArgs& a, const float* act, float* tsum, float* rstd) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nt = a.d / 128;
  cbar();
  for (int q = warp; q < a.B * nt; q += kMkWarps) {
    const int m = q / nt, t = q % nt;
    const float* x = act + static_cast<size_t>(m) * a.d + t * 128;
    float s = 0.f;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float v = x[u * 32 + lane];
      s = fmaf(v, v, s);
    }
    s = warp_sum(s);
    if (lane == 0) tsum[q] = s;
  }
  cbar();
  if (tid < a.B) {
    float s = 0.f;
    for (int t = 0; t < nt; ++t) s += tsum[tid * nt + t];
    rstd[tid] = rsqrtf(s / static_cast<float>(a.d) + a.eps);
  }
  cbar();
}

// act[m][i] = x * rstd[m] * g[i]
// (the gains are loaded eight per thread at a time)
__device__ __forceinline__ void mk_scale(const MkArgs& a, float* act, const float* rstd, const float* __restrict__ g) {
  for (int i0 = threadIdx.x; i0 < a.d; i0 += 8 * kMkCompute) {
    float gv[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int i = i0 + u * kMkCompute;
      gv[u] = i < a.d ? __ldg(g + i) : 0.f;
    }
    for (int m = 0; m < a.B; ++m) {
      const float r = rstd[m];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int i = i0 + u * kMkCompute;
        if (i < a.d) {
          const size_t o = static_cast<size_t>(m) * a.d + i;
          act[o] = act[o] * r * gv[u];
        }
      }
    }
  }
  cbar();
}

}  // namespace
}  // namespace dvi

namespace dvi {
namespace {

// The normed input of a projection over d columns in one pass (d <= 4096):
// x = xa + xb (or the embedding of tok), stored to xr_out by `writer`; the
// per-128-feature sums of squares (tsum) and 1/rms (rstd); the A planes of
// x * rstd * g.  Thread tid takes the column pairs tid + 256 e, whose loads
// (x and gain) are all issued before any is used; a warp's 32 pairs are half
// a 128-column tile, so the tile sums are two warp sums (hs[m][tile][half]).
constexpr int kMkPairs = 8;   // column pairs per thread: d <= 512 * kMkPairs
template <int M>
__device__ __forceinline__ void mk_norm_pack(const MkArgs& a, const float* __restrict__ xa,
                                             const float* __restrict__ xb, const int* tok, float* xr_out,
                                             bool writer, const float* __restrict__ g, uint32_t* xw, int plane,
                                             float* tsum, float* rstd, float* hs) {
  const int d = a.d, np = d / 2, nt = d / 128, pw = plane / 2;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  float2 x[M][kMkPairs], gv[kMkPairs];
#pragma unroll
  for (int e = 0; e < kMkPairs; ++e) {
    const int p = tid + e * kMkCompute;
    gv[e] = make_float2(0.f, 0.f);
#pragma unroll
    for (int m = 0; m < M; ++m) x[m][e] = make_float2(0.f, 0.f);
    if (p < np) {
      gv[e] = __ldg(reinterpret_cast<const float2*>(g) + p);
#pragma unroll
      for (int m = 0; m < M; ++m) {
        if (tok) {
          const uint32_t w = __ldg(reinterpret_cast<const uint32_t*>(static_cast<const __nv_bfloat16*>(a.embed) +
                                                                      static_cast<size_t>(tok[m]) * d) + p);
          x[m][e] = make_float2(bf16_lo(w), bf16_hi(w));
        } else {
          const float2 u = __ldcg(reinterpret_cast<const float2*>(xa + static_cast<size_t>(m) * d) + p);
          const float2 v = __ldcg(reinterpret_cast<const float2*>(xb + static_cast<size_t>(m) * d) + p);
          x[m][e] = make_float2(u.x + v.x, u.y + v.y);
        }
      }
    }
  }
#pragma unroll
  for (int e = 0; e < kMkPairs; ++e) {
    const int p = tid + e * kMkCompute;
    if (p < np) {
#pragma unroll
      for (int m = 0; m < M; ++m) {
        if (writer) reinterpret_cast<float2*>(xr_out + static_cast<size_t>(m) * d)[p] = x[m][e];
        const float sq = warp_sum(fmaf(x[m][e].x, x[m][e].x, x[m][e].y * x[m][e].y));
        if (lane == 0) hs[(m * nt + (e * kMkCompute + warp * 32) / 64) * 2 + (warp & 1)] = sq;
      }
    }
  }
  cbar();
  if (tid < M) {
    float s = 0.f;
    for (int t = 0; t < nt; ++t) {
      const float ts = hs[(tid * nt + t) * 2] + hs[(tid * nt + t) * 2 + 1];
      tsum[tid * nt + t] = ts;
      s += ts;
    }
    rstd[tid] = rsqrtf(s / static_cast<float>(d) + a.eps);
  }
  cbar();
#pragma unroll
  for (int e = 0; e < kMkPairs; ++e) {
    const int p = tid + e * kMkCompute;
    if (p < np) {
#pragma unroll
      for (int m = 0; m < M; ++m) {
        const float r = rstd[m];
        uint32_t hi, lo;
        split_bf16x2(x[m][e].x * r * gv[e].x, x[m][e].y * r * gv[e].y, hi, lo);
        xw[(2 * m) * pw + p] = hi;
        xw[(2 * m + 1) * pw + p] = lo;
      }
    }
  }
  // zero columns up to the end of the last 1024-column chunk
  const int nw = mk_chunks(d) * kMkChunk / 2;
  for (int w = np + tid; w < nw; w += kMkCompute)
#pragma unroll
    for (int q = 0; q < 2 * M; ++q) xw[q * pw + w] = 0u;
  cbar();
}

// ------------------------------------------------------------------ attention
// A K or V stage holds CP cache rows as hd / 64 tiles of CP rows x 64
// (one 3D box, 128-byte swizzled): the 16-byte chunk j of row i.
template <int HD>
__device__ __forceinline__ uint32_t kv_off(int i, int j) {
  constexpr int CP = kMkStageElems / HD;
  return static_cast<uint32_t>((j >> 3) * CP * 128 + i * 128 + (((j & 7) ^ (i & 7)) << 4));
}

// Rows [from, cn) of a K or V chunk stage whose positions were written in
// this launch (or are the newest one, `fresh`) are copied in from global
// memory, then ordered before the stage's next asynchronous write.
template <int HD>
__device__ __forceinline__ void mk_patch(const MkArgs& a, const void* cache, int l, const AttUnit& u, uint8_t* st,
                                         int c0, int from, int cn, const __nv_bfloat16* fresh) {
  constexpr int V16 = HD / 8;   // 16-byte chunks per row
  for (int e = threadIdx.x; e < (cn - from) * V16; e += kMkCompute) {
    const int i = from + e / V16, q = e % V16;
    const int x = c0 + i;
    // the newest row from shared memory (also for a position past the cache,
    // flagged KV_FULL), earlier ones from the cache in global memory
    uint4 v;
    if (x == u.pos || x >= a.max_len)
      v = reinterpret_cast<const uint4*>(fresh)[q];
    else
      v = __ldcg(reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(cache) +
                                                kv_row(a, l, u.b, u.kvh, x) * HD) + q);
    *reinterpret_cast<uint4*>(st + kv_off<HD>(i, q)) = v;
  }
  fence_proxy_async_smem();
  cbar();
}

// D (16x8 f32) += A (16x8 bf16, row) . B (8x8 bf16, col), one warp.
__device__ __forceinline__ void mma_bf16_1688(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t b0) {
  asm volatile("mma.sync.aligned.m16n8k8.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5}, {%6}, {%0,%1,%2,%3};"
               : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
               : "r"(a0), "r"(a1), "r"(b0));
}

// The halves of a bf16 pair at chunk positions p, p + 1 that lie below cn.
__device__ __forceinline__ uint32_t kv_mask(uint32_t v, int p, int cn) {
  return (p < cn ? v & 0xffffu : 0u) | (p + 1 < cn ? v & 0xffff0000u : 0u);
}

// One attention unit: G query heads of KV head kvh for the decode row of
// sequence b at position pos, over the unit's range of [0, pos]; writes the
// partial (running max, sum, o) for the O phase's combine.
//
// Both products run on the tensor cores (warp MMA, f32 accumulation) with the
// stage's CP positions split over the 8 warps, PW each.  Scores: A row 2 h
// is the bf16 hi part of query head h (pre-scaled by log2(e) / sqrt(hd), so
// the softmax uses exp2), row 2 h + 1 its lo part (heads 4..7 in rows
// 8..15); B is the warp's key rows (ldmatrix); a score is its hi row plus its
// lo row (lanes g and g ^ 1).  Each warp keeps its own online softmax (max,
// sum and o in registers), updated once per chunk: the chunk's key stage,
// the update, then its value stage as o^T += V^T p^T with A = the warp's
// value rows (ldmatrix.trans, 16 dimensions an m-tile) and B = the
// probabilities, column 2 h the hi part of head h and 2 h + 1 its lo part (a
// lane's scores are already where the B fragment wants them).  The 8 warps'
// partials are merged at the end.  Positions past the range get probability 0
// and their value rows are masked to 0.  The chunk loop is not unrolled
// (compact code: the phase runs after the projections' code has filled the
// instruction cache).
template <int HD, int G>
__device__ bool mk_attention(const MkArgs& a, int l, const AttUnit& u, Ring& ring, uint8_t* att_sm) {
  constexpr int CP = kMkStageElems / HD;   // positions per stage
  constexpr int PW = CP / kMkWarps;        // positions per warp and stage
  constexpr int NT = PW / 8;               // score n-tiles per warp
  constexpr int KS = HD / 16;              // k16 steps of a score
  constexpr int MT = HD / 16;              // m-tiles of o^T
  constexpr int NH = G > 4 ? 2 : 1;        // head tiles (4 heads: hi, lo columns)
  constexpr int half = HD / 2;
  static_assert(NT == 1 || NT == 2, "8 or 16 positions per warp and stage");
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, c = lane & 3, lrow = lane & 7, lmat = lane >> 3;
  constexpr int QL = 8 * G < 32 ? 8 * G : 32;   // lanes with live A rows (g < 2 G)
  uint4* qf = reinterpret_cast<uint4*>(att_sm);                         // [KS][QL]
  __nv_bfloat16* kn = reinterpret_cast<__nv_bfloat16*>(qf + KS * QL);   // [HD]
  __nv_bfloat16* vn = kn + HD;

  const float* qrow = a.qkv + static_cast<size_t>(u.b) * (a.Hq + 2 * a.Hkv) * HD;
  const bool pos_ok = u.pos < a.max_len;
  const int rp = pos_ok ? u.pos : a.max_len - 1;
  const float2* rope = a.rope + static_cast<size_t>(rp) * half;
  const float qscale = kLog2e * rsqrtf(static_cast<float>(HD));
  // dimension dim of head row h of this row's q | k after RoPE
  auto rot = [&](int h, int dim) {
    const float* x = qrow + static_cast<size_t>(h) * HD;
    const float v = __ldcg(x + dim), vp = __ldcg(x + (dim < half ? dim + half : dim - half));
    const float2 cs = rope[dim % half];
    return dim < half ? v * cs.x - vp * cs.y : v * cs.x + vp * cs.y;
  };
  // the A fragment of lane (gg, cc) for k-step ks: rows gg and gg + 8
  for (int i = tid; i < KS * QL; i += kMkCompute) {
    const int ks = i / QL, gg = (i % QL) >> 2, cc = i & 3;
    uint32_t f[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int row = gg + 8 * r, hq = row >> 1;
      if (hq < G) {
        const int h = u.kvh * G + hq, d0 = 16 * ks + 2 * cc;
        uint32_t hi0, lo0, hi1, lo1;
        split_bf16x2(rot(h, d0) * qscale, rot(h, d0 + 1) * qscale, hi0, lo0);
        split_bf16x2(rot(h, d0 + 8) * qscale, rot(h, d0 + 9) * qscale, hi1, lo1);
        f[r] = row & 1 ? lo0 : hi0;
        f[2 + r] = row & 1 ? lo1 : hi1;
      }
    }
    qf[i] = make_uint4(f[0], f[1], f[2], f[3]);
  }
  for (int dim = tid; dim < HD; dim += kMkCompute) {
    kn[dim] = __float2bfloat16_rn(rot(a.Hq + u.kvh, dim));
    vn[dim] = __float2bfloat16_rn(__ldcg(qrow + static_cast<size_t>(a.Hq + a.Hkv + u.kvh) * HD + dim));
  }
  cbar();
  // the newest position into the cache (the unit whose range ends at pos)
  if (u.p == a.P - 1) {
    if (pos_ok) {
      const size_t row = kv_row(a, l, u.b, u.kvh, u.pos) * HD;
      for (int dim = tid; dim < HD; dim += kMkCompute) {
        static_cast<__nv_bfloat16*>(a.kc)[row + dim] = kn[dim];
        static_cast<__nv_bfloat16*>(a.vc)[row + dim] = vn[dim];
      }
    } else if (tid == 0) {
      flag_status(a.status, DVI_DEV_KV_FULL);
    }
  }
  // lane (g, c) tracks heads g / 2 + 4 h (h < NH) for the softmax and holds
  // o^T of heads c + 4 h at dimensions 16 m + g and 16 m + g + 8
  float o[MT][NH][4];
#pragma unroll
  for (int m = 0; m < MT; ++m)
#pragma unroll
    for (int h = 0; h < NH; ++h) o[m][h][0] = o[m][h][1] = o[m][h][2] = o[m][h][3] = 0.f;
  float mrun[NH], lrun[NH];
#pragma unroll
  for (int h = 0; h < NH; ++h) {
    mrun[h] = -INFINITY;
    lrun[h] = 0.f;
  }
  const int pw0 = warp * PW;   // the warp's first position in a chunk
  // the lane's q fragments, held for the whole range
  uint32_t qa[KS][4];
#pragma unroll
  for (int ks = 0; ks < KS; ++ks) {
    const uint4 v = lane < QL ? qf[ks * QL + lane] : make_uint4(0u, 0u, 0u, 0u);
    qa[ks][0] = v.x;
    qa[ks][1] = v.y;
    qa[ks][2] = v.z;
    qa[ks][3] = v.w;
  }
  bool ok = true;
#pragma unroll 1
  for (int c0 = u.r0; c0 < u.r1; c0 += CP) {
    const int cn = min(CP, u.r1 - c0);
    const int stable = att_stable(a, u, c0, cn);
    // ---- scores of the chunk's keys: lane (g, c) gets its heads at the
    // positions pw0 + 8 t + 2 c + {0, 1} (two accumulators: even and odd k16 steps)
    float s[NT][NH][2];
    {
      uint8_t* st = const_cast<uint8_t*>(ring_acquire(ring, a.status, ok));
      if (!ok) return false;
      if (stable < cn) mk_patch<HD>(a, a.kc, l, u, st, c0, stable, cn, kn);
      const uint32_t sb = smem_u32(st);
#pragma unroll
      for (int t = 0; t < NT; ++t) {
        float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
        for (int kp = 0; kp < KS / 2; ++kp) {
          uint32_t bk[4];
          ldmatrix_x4(bk, sb + kv_off<HD>(pw0 + 8 * t + lrow, 4 * kp + lmat));
          mma_bf16_16816(acc[0], qa[2 * kp], bk[0], bk[1]);
          mma_bf16_16816(acc[1], qa[2 * kp + 1], bk[2], bk[3]);
        }
        const int i0 = pw0 + 8 * t + 2 * c;
#pragma unroll
        for (int h = 0; h < NH; ++h) {
          const float y0 = acc[0][2 * h] + acc[1][2 * h], y1 = acc[0][2 * h + 1] + acc[1][2 * h + 1];
          const float x0 = y0 + __shfl_xor_sync(0xffffffffu, y0, 4);
          const float x1 = y1 + __shfl_xor_sync(0xffffffffu, y1, 4);
          s[t][h][0] = i0 < cn ? x0 : -INFINITY;
          s[t][h][1] = i0 + 1 < cn ? x1 : -INFINITY;
        }
      }
      ring_release(ring);
    }
    // ---- the warp's online-softmax update of its heads
    uint32_t bp[NT][NH];   // the B fragments: hi (g even) or lo (g odd) of the probabilities
#pragma unroll
    for (int h = 0; h < NH; ++h) {
      float mx = -INFINITY;
#pragma unroll
      for (int t = 0; t < NT; ++t) mx = fmaxf(mx, fmaxf(s[t][h][0], s[t][h][1]));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      const float mn = fmaxf(mrun[h], mx);
      const float mu = mn == -INFINITY ? 0.f : mn;   // no position yet: every weight is 0
      const float cr = exp2f(mrun[h] - mu);
      mrun[h] = mn;
      lrun[h] *= cr;
      // o^T's columns are heads c + 4 h: their factor from lane (2 c, 0)
      const float co = __shfl_sync(0xffffffffu, cr, 8 * c);
#pragma unroll
      for (int m = 0; m < MT; ++m)
#pragma unroll
        for (int q = 0; q < 4; ++q) o[m][h][q] *= co;
#pragma unroll
      for (int t = 0; t < NT; ++t) {
        const float p0 = exp2f(s[t][h][0] - mu), p1 = exp2f(s[t][h][1] - mu);
        lrun[h] += p0 + p1;
        uint32_t hi, lo;
        split_bf16x2(p0, p1, hi, lo);
        bp[t][h] = g & 1 ? lo : hi;
      }
    }
    // ---- values: o^T += V^T p^T over the warp's positions
    {
      uint8_t* st = const_cast<uint8_t*>(ring_acquire(ring, a.status, ok));
      if (!ok) return false;
      if (stable < cn) mk_patch<HD>(a, a.vc, l, u, st, c0, stable, cn, vn);
      const uint32_t sb = smem_u32(st);
      const bool ragged = cn < CP;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        uint32_t av[4];
        if constexpr (NT == 1) {
          // k8: matrix i is the warp's 8 rows x dimensions 8 (4 q + i), the
          // A fragments of m-tiles 2 q (i = 0, 1) and 2 q + 1 (i = 2, 3)
          ldmatrix_x4_trans(av, sb + kv_off<HD>(pw0 + lrow, 4 * q + lmat));
          if (ragged)
#pragma unroll
            for (int i = 0; i < 4; ++i) av[i] = kv_mask(av[i], pw0 + 2 * c, cn);
#pragma unroll
          for (int h = 0; h < NH; ++h) {
            mma_bf16_1688(o[2 * q][h], av[0], av[1], bp[0][h]);
            mma_bf16_1688(o[2 * q + 1][h], av[2], av[3], bp[0][h]);
          }
        } else {
          // k16: matrices (rows 0..7 | 8..15) x (dimensions 16 q + 0..7 | + 8..15)
          ldmatrix_x4_trans(av, sb + kv_off<HD>(pw0 + 8 * (lmat >> 1) + lrow, 2 * q + (lmat & 1)));
          if (ragged)
#pragma unroll
            for (int i = 0; i < 4; ++i) av[i] = kv_mask(av[i], pw0 + 8 * (i >> 1) + 2 * c, cn);
#pragma unroll
          for (int h = 0; h < NH; ++h) mma_bf16_16816(o[q][h], av, bp[0][h], bp[NT - 1][h]);
        }
      }
      ring_release(ring);
    }
  }
  // ---- the warp's partials (max, sum, o of each head) overlay the q
  // fragments and new rows once every warp is done with them; then the 8
  // are merged (weights exp2(max_w - max))
  cbar();
  float* osum = reinterpret_cast<float*>(att_sm);   // [8][G][HD]
  float* wml = osum + kMkWarps * G * HD;            // [8][G][2]
#pragma unroll
  for (int h = 0; h < NH; ++h) {
    lrun[h] += __shfl_xor_sync(0xffffffffu, lrun[h], 1);
    lrun[h] += __shfl_xor_sync(0xffffffffu, lrun[h], 2);
    const int ho = c + 4 * h;   // o's head
    if (ho < G) {
      float* ow = osum + (warp * G + ho) * HD;
#pragma unroll
      for (int m = 0; m < MT; ++m) {
        ow[16 * m + g] = o[m][h][0] + o[m][h][1];
        ow[16 * m + g + 8] = o[m][h][2] + o[m][h][3];
      }
    }
    const int hs = (g >> 1) + 4 * h;   // the softmax's head
    if ((g & 1) == 0 && c == 0 && hs < G) {
      wml[(warp * G + hs) * 2] = mrun[h];
      wml[(warp * G + hs) * 2 + 1] = lrun[h];
    }
  }
  cbar();
  const size_t stride = HD + 2;
  for (int i = tid; i < G * HD; i += kMkCompute) {
    const int gg = i / HD, dd = i % HD;
    float m = -INFINITY;
#pragma unroll
    for (int w = 0; w < kMkWarps; ++w) m = fmaxf(m, wml[(w * G + gg) * 2]);
    float v = 0.f, sum = 0.f;
#pragma unroll
    for (int w = 0; w < kMkWarps; ++w) {
      const float mw = wml[(w * G + gg) * 2];
      if (mw != -INFINITY) {
        const float e = exp2f(mw - m);
        v = fmaf(e, osum[(w * G + gg) * HD + dd], v);
        if (dd == 0) sum = fmaf(e, wml[(w * G + gg) * 2 + 1], sum);
      }
    }
    float* dst = a.att + ((static_cast<size_t>(u.b) * a.Hq + u.kvh * G + gg) * a.P + u.p) * stride;
    dst[2 + dd] = v;
    if (dd == 0) {
      dst[0] = m;
      dst[1] = sum;
    }
  }
  return true;
}

// The unit's attention for the GQA group size of the model (1, 2, 4 or 8).
template <int HD>
__device__ __forceinline__ bool mk_attention_any(const MkArgs& a, int l, const AttUnit& u, Ring& ring,
                                                 uint8_t* att_sm) {
  switch (a.Hq / a.Hkv) {
    case 1: return mk_attention<HD, 1>(a, l, u, ring, att_sm);
    case 2: return mk_attention<HD, 2>(a, l, u, ring, att_sm);
    case 4: return mk_attention<HD, 4>(a, l, u, ring, att_sm);
    default:
      // a group of 8 at head_dim 128 (o^T in 64 registers a lane) is not
      // given to this kernel
      if constexpr (HD == 64) return mk_attention<HD, 8>(a, l, u, ring, att_sm);
      return false;
  }
}

// The O phase's input: for every row and query head the P partials merged
// (weights exp2(m_p - max) / sum) and packed straight into the A planes
// (column pairs of H_q hd; four pairs per thread at a time, all their
// partials' loads issued together).
template <int HD, int M>
__device__ __forceinline__ void mk_att_combine(const MkArgs& a, uint32_t* xw, int plane, float* wts) {
  const int K = a.Hq * HD, P = a.P, np = K / 2, pw = plane / 2;
  const size_t stride = HD + 2;
  for (int i = threadIdx.x; i < a.B * a.Hq; i += kMkCompute) {
    const float* base = a.att + static_cast<size_t>(i) * P * stride;
    float mx = -INFINITY;
    for (int p = 0; p < P; ++p) mx = fmaxf(mx, __ldcg(base + p * stride));
    float sum = 0.f;
    for (int p = 0; p < P; ++p) sum += __ldcg(base + p * stride + 1) * exp2f(__ldcg(base + p * stride) - mx);
    const float inv = 1.f / sum;
    for (int p = 0; p < P; ++p) wts[i * P + p] = exp2f(__ldcg(base + p * stride) - mx) * inv;
  }
  cbar();
  for (int q0 = threadIdx.x; q0 < np; q0 += 4 * kMkCompute) {
#pragma unroll
    for (int m = 0; m < M; ++m) {
      float2 s[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) s[u] = make_float2(0.f, 0.f);
      for (int p = 0; p < P; ++p) {
        float2 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int q = q0 + u * kMkCompute;
          v[u] = make_float2(0.f, 0.f);
          if (q < np)
            v[u] = __ldcg(reinterpret_cast<const float2*>(
                a.att + ((static_cast<size_t>(m) * a.Hq + (2 * q) / HD) * P + p) * stride + 2 + (2 * q) % HD));
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int q = q0 + u * kMkCompute;
          if (q < np) {
            const float wgt = wts[(m * a.Hq + (2 * q) / HD) * P + p];
            s[u].x = fmaf(v[u].x, wgt, s[u].x);
            s[u].y = fmaf(v[u].y, wgt, s[u].y);
          }
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int q = q0 + u * kMkCompute;
        if (q < np) {
          uint32_t hi, lo;
          split_bf16x2(s[u].x, s[u].y, hi, lo);
          xw[(2 * m) * pw + q] = hi;
          xw[(2 * m + 1) * pw + q] = lo;
        }
      }
    }
  }
  const int nw = mk_chunks(K) * kMkChunk / 2;
  for (int w = np + threadIdx.x; w < nw; w += kMkCompute)
#pragma unroll
    for (int q = 0; q < 2 * M; ++q) xw[q * pw + w] = 0u;
  cbar();
}

}  // namespace
}  // namespace dvi

namespace dvi {
namespace {

}  // namespace
}  // namespace dvi

namespace dvi {
namespace {

// ------------------------------------------------------------------ compute warps
template <int M, int HD>
__device__ void mk_compute(const MkArgs& a, Ring& ring, const MkLayout& L, uint8_t* sm) {
  const int c = blockIdx.x, n = gridDim.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  float* act = reinterpret_cast<float*>(sm + L.act);
  uint32_t* xw = reinterpret_cast<uint32_t*>(sm + L.xw);
  const int plane = mk_plane(a);
  const uint32_t xa = smem_u32(xw);
  const bool fused = a.d <= 512 * kMkPairs;
  float* wacc = reinterpret_cast<float*>(sm + L.wacc);
  float* gbuf = reinterpret_cast<float*>(sm + L.gbuf);
  uint8_t* att_sm = sm + L.att;
  float* hs = reinterpret_cast<float*>(att_sm);   // half-tile sums [B][d/128][2] (attention scratch is free then)
  unsigned long long* wkeys = reinterpret_cast<unsigned long long*>(sm + L.misc);   // [8][kMkMaxRows]
  float* rstd = reinterpret_cast<float*>(wkeys + kMkWarps * kMkMaxRows);               // [kMkMaxRows]
  int* tok = reinterpret_cast<int*>(rstd + kMkMaxRows);                                // [kMkMaxRows]
  int* flag_s = tok + kMkMaxRows;                                                      // [4]
  float* tsum = reinterpret_cast<float*>(flag_s + 4);                                  // [B][d/128]
  float* bu = tsum + M * (a.d / 128);                                                  // [B][r]
  const int rows_max = a.rows_max, d = a.d, nt = d / 128, K = a.K, r = a.r;
  const int nq = a.Hq * HD;
  const int npass = a.mode == MK_DRAFT ? a.Kv : 1;
  const size_t nqkv = static_cast<size_t>(a.Hq + 2 * a.Hkv) * HD;
  int q0, q1, o0, o1, f0, f1, v0, v1, h0, h1;
  part_range(mk_groups(static_cast<int>(nqkv)), c, n, q0, q1);
  part_range(mk_groups(d), c, n, o0, o1);
  part_range(mk_groups(a.F), c, n, f0, f1);
  part_range(mk_groups(a.V), c, n, v0, v1);
  part_range(d, c, n, h0, h1);
  float* xr[2] = {a.xr, a.xr + static_cast<size_t>(M) * d};
  int bn = 0;    // next completion counter
  int bw = -1;   // counter the next phase waits for
  int cur = 0;   // xr slot that holds the residual
  for (int j = 0; j < npass; ++j) {
    const bool head = a.mode == MK_DRAFT && j < K;
    const AttUnit u = att_unit(a, j, c);
    for (int l = 0; l < a.k; ++l) {
      const MkLayerW& w = a.layer[l];
      // ---------------- QKV
      if (bw >= 0 && !mk_wait(a, bw, flag_s)) return;
      if (l == 0) {
        if (tid < M) {
          int t;
          if (j == 0) {
            t = __ldcg(a.pending + tid);
          } else {
            // the previous pass's draft t~_j
            const unsigned long long key = __ldcg(a.keys + static_cast<size_t>(j - 1) * M + tid);
            t = key ? argmax_idx(key) : 0;
            if (!key) flag_status(a.status, DVI_DEV_NONFINITE);
            if (c == 0) a.draft_ids[tid * (K + 1) + j] = t;
          }
          if (t < 0 || t >= a.V) {
            flag_status(a.status, DVI_DEV_BAD_TOKEN);
            t = 0;
          }
          tok[tid] = t;
        }
        cbar();
      }
      if (fused) {
        mk_norm_pack<M>(a, xr[cur], a.y, l == 0 ? tok : nullptr, xr[cur ^ 1], c == 0, w.g_attn, xw, plane, tsum, rstd,
                        hs);
      } else {
        if (l == 0) mk_residual(a, act, nullptr, nullptr, tok, xr[cur ^ 1], c == 0);
        else mk_residual(a, act, xr[cur], a.y, nullptr, xr[cur ^ 1], c == 0);
        mk_rms(a, act, tsum, rstd);
        mk_scale(a, act, rstd, w.g_attn);
        mk_pack<M>(xw, plane, act, d, d, false);
      }
      cur ^= 1;
      if (!gemv_groups<M>(ring, d, q0, q1, xa, plane, wacc, rows_max, a.status)) {
        mk_abort(a);
        return;
      }
      gemv_finish<M>(wacc, rows_max, (q1 - q0) * kMkGroup,
                     [&](int rl, int m, float v) { a.qkv[m * nqkv + q0 * kMkGroup + rl] = v; });
      mk_signal(a, bn);
      bw = bn++;
      // ---------------- attention
      if (!mk_wait(a, bw, flag_s)) return;
      if (u.on && !mk_attention_any<HD>(a, l, u, ring, att_sm)) {
        mk_abort(a);
        return;
      }
      mk_signal(a, bn);
      bw = bn++;
      // ---------------- O
      if (!mk_wait(a, bw, flag_s)) return;
      mk_att_combine<HD, M>(a, xw, plane, reinterpret_cast<float*>(att_sm));
      if (!gemv_groups<M>(ring, nq, o0, o1, xa, plane, wacc, rows_max, a.status)) {
        mk_abort(a);
        return;
      }
      gemv_finish<M>(wacc, rows_max, (o1 - o0) * kMkGroup, [&](int rl, int m, float v) {
        a.ao[static_cast<size_t>(m) * d + o0 * kMkGroup + rl] = v;
      });
      mk_signal(a, bn);
      bw = bn++;
      // ---------------- gate / up
      if (!mk_wait(a, bw, flag_s)) return;
      if (fused) {
        mk_norm_pack<M>(a, xr[cur], a.ao, nullptr, xr[cur ^ 1], c == 0, w.g_ffn, xw, plane, tsum, rstd, hs);
      } else {
        mk_residual(a, act, xr[cur], a.ao, nullptr, xr[cur ^ 1], c == 0);
        mk_rms(a, act, tsum, rstd);
        mk_scale(a, act, rstd, w.g_ffn);
        mk_pack<M>(xw, plane, act, d, d, false);
      }
      cur ^= 1;
      if (!gemv_groups<M>(ring, d, f0, f1, xa, plane, wacc, rows_max, a.status)) {
        mk_abort(a);
        return;
      }
      gemv_finish<M>(wacc, rows_max, (f1 - f0) * kMkGroup, [&](int rl, int m, float v) { gbuf[rl * M + m] = v; });
      if (!gemv_groups<M>(ring, d, f0, f1, xa, plane, wacc, rows_max, a.status)) {
        mk_abort(a);
        return;
      }
      gemv_finish<M>(wacc, rows_max, (f1 - f0) * kMkGroup, [&](int rl, int m, float v) {
        const float g = gbuf[rl * M + m];   // written by this thread in the gate's finish
        a.hbuf[static_cast<size_t>(m) * a.F + f0 * kMkGroup + rl] = g / (1.f + expf(-g)) * v;
      });
      mk_signal(a, bn);
      bw = bn++;
      // ---------------- down
      if (!mk_wait(a, bw, flag_s)) return;
      mk_pack<M>(xw, plane, a.hbuf, a.F, a.F, true);
      if (!gemv_groups<M>(ring, a.F, o0, o1, xa, plane, wacc, rows_max, a.status)) {
        mk_abort(a);
        return;
      }
      gemv_finish<M>(wacc, rows_max, (o1 - o0) * kMkGroup, [&](int rl, int m, float v) {
        a.y[static_cast<size_t>(m) * d + o0 * kMkGroup + rl] = v;
      });
      mk_signal(a, bn);
      bw = bn++;
    }
    // ---------------- h_k: hand-off to the verify (or AR) rows, drafter head
    if (!mk_wait(a, bw, flag_s)) return;
    mk_residual(a, act, xr[cur], a.y, nullptr, nullptr, false);
    mk_rms(a, act, tsum, rstd);
    for (int m = 0; m < M; ++m) {
      const size_t row = static_cast<size_t>(m) * a.copy_row_stride + (a.mode == MK_DRAFT ? j : 0);
      for (int i = h0 + tid; i < h1; i += kMkCompute) {
        const float x = act[static_cast<size_t>(m) * d + i];
        a.x_copy[row * d + i] = x;
        Act<__nv_bfloat16>::st(static_cast<__nv_bfloat16*>(a.xg_copy) + row * d + i, a.xg_copy_plane, x * a.g_hand[i]);
      }
      for (int t = c + tid * n; t < nt; t += kMkCompute * n)
        a.ss_copy[static_cast<size_t>(t) * a.ss_copy_ld + row] = tsum[m * nt + t];
    }
    if (!head) {
      bw = -1;
      continue;
    }
    cbar();   // the hand-off read h_k before u overwrites it
    mk_scale(a, act, rstd, a.final_norm);   // u = RMSNorm_final(h_k)
    const int ls = a.log_enabled ? __ldcg(a.log_step) : a.log_cap_steps;
    const bool logged = a.log_enabled && ls < a.log_cap_steps;
    if (logged && a.log_u) {
      for (int m = 0; m < M; ++m) {
        const size_t row = (static_cast<size_t>(ls) * M + m) * K + j;
        for (int i = h0 + tid; i < h1; i += kMkCompute)
          Act<__nv_bfloat16>::st(static_cast<__nv_bfloat16*>(a.log_u) + row * d + i, a.log_plane,
                                 act[static_cast<size_t>(m) * d + i]);
      }
    }
    int bu_bound = -1;
    if (r > 0) {
      // this CTA's share of B u
      for (int q = warp; q < M * r; q += kMkWarps) {
        const int m = q / r, rr = q % r;
        const float* brow = a.lora_b + static_cast<size_t>(rr) * d;
        float s = 0.f;
        for (int i = h0 + lane; i < h1; i += 32) s = fmaf(brow[i], act[static_cast<size_t>(m) * d + i], s);
        s = warp_sum(s);
        if (lane == 0) a.bu_part[(static_cast<size_t>(c) * M + m) * r + rr] = s;
      }
      mk_signal(a, bn);
      bu_bound = bn++;
    }
    mk_pack<M>(xw, plane, act, d, d, false);
    if (!gemv_groups<M>(ring, d, v0, v1, xa, plane, wacc, rows_max, a.status)) {
      mk_abort(a);
      return;
    }
    if (r > 0) {
      if (!mk_wait(a, bu_bound, flag_s)) return;
      // B u = the CTAs' partials summed: 16 lanes per value, each a strided
      // share of the CTAs (loads in flight together), then a shuffle tree
      for (int q0 = warp * 2; q0 < M * r; q0 += 2 * kMkWarps) {
        const int q = q0 + (lane >> 4), sub = lane & 15;
        float sv = 0.f;
        if (q < M * r) {
          const int m = q / r, rr = q % r;
          float v[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const int cc = sub + 16 * i;
            v[i] = cc < n ? __ldcg(a.bu_part + (static_cast<size_t>(cc) * M + m) * r + rr) : 0.f;
          }
          for (int cc = sub + 256; cc < n; cc += 16)
            v[0] += __ldcg(a.bu_part + (static_cast<size_t>(cc) * M + m) * r + rr);
#pragma unroll
          for (int i = 0; i < 16; ++i) sv += v[i];
        }
#pragma unroll
        for (int off = 8; off > 0; off >>= 1) sv += __shfl_xor_sync(0xffffffffu, sv, off);
        if (sub == 0 && q < M * r) bu[q] = sv;
      }
    }
    float* zrow[M];
#pragma unroll
    for (int m = 0; m < M; ++m)
      zrow[m] = logged && a.zlog ? a.zlog + ((static_cast<size_t>(ls) * M + m) * K + j) * a.V : nullptr;
    unsigned long long best[M];
#pragma unroll
    for (int m = 0; m < M; ++m) best[m] = 0ull;
    gemv_finish<M>(wacc, rows_max, (v1 - v0) * kMkGroup, [&](int rl, int m, float v) {
      const int vi = v0 * kMkGroup + rl;
      if (vi >= a.V) return;
      float z = v;
      if (r > 0) {
        const float* ar = a.lora_a + static_cast<size_t>(vi) * r;
        float acc = 0.f;
        if ((r & 3) == 0 && (reinterpret_cast<uintptr_t>(a.lora_a) & 15u) == 0) {
          // the row of A four floats at a time, four loads in flight
          const int r4 = r >> 2;
          for (int q0 = 0; q0 < r4; q0 += 4) {
            float4 av[4];
#pragma unroll
            for (int q = 0; q < 4; ++q)
              if (q0 + q < r4) av[q] = __ldg(reinterpret_cast<const float4*>(ar) + q0 + q);
#pragma unroll
            for (int q = 0; q < 4; ++q)
              if (q0 + q < r4) {
                const float* b4 = bu + m * r + 4 * (q0 + q);
                acc = fmaf(av[q].x, b4[0], acc);
                acc = fmaf(av[q].y, b4[1], acc);
                acc = fmaf(av[q].z, b4[2], acc);
                acc = fmaf(av[q].w, b4[3], acc);
              }
          }
        } else {
          for (int q = 0; q < r; ++q) acc = fmaf(ar[q], bu[m * r + q], acc);
        }
        z = fmaf(a.gamma, acc, z);
      }
      if (zrow[m]) zrow[m][vi] = z;
      if (isfinite(z)) {
        const unsigned long long key = argmax_key(z, vi);
        best[m] = key > best[m] ? key : best[m];
      } else {
        flag_status(a.status, DVI_DEV_NONFINITE);
      }
    });
#pragma unroll
    for (int m = 0; m < M; ++m) {
      const unsigned long long k = warp_max_u64(best[m]);
      if (lane == 0) wkeys[warp * kMkMaxRows + m] = k;
    }
    cbar();
    if (tid < M) {
      unsigned long long k = 0ull;
      for (int q = 0; q < kMkWarps; ++q) k = wkeys[q * kMkMaxRows + tid] > k ? wkeys[q * kMkMaxRows + tid] : k;
      if (k) atomicMax(a.keys + static_cast<size_t>(j) * M + tid, k);
    }
    mk_signal(a, bn);
    bw = bn++;
  }
  // without the bonus pass no pass reads the last draft: record t~_K
  if (a.mode == MK_DRAFT && a.Kv == K && K > 0 && c == 0) {
    if (!mk_wait(a, bw, flag_s)) return;
    if (tid < M) {
      const unsigned long long key = __ldcg(a.keys + static_cast<size_t>(K - 1) * M + tid);
      if (!key) flag_status(a.status, DVI_DEV_NONFINITE);
      a.draft_ids[tid * (K + 1) + K] = key ? argmax_idx(key) : 0;
    }
  }
}

template <int M, int HD>
__global__ void __launch_bounds__(kMkThreads, 1) mk_kernel(const __grid_constant__ MkArgs a) {
  extern __shared__ __align__(16) uint8_t mk_smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(mk_smem_raw) + 1023) & ~uintptr_t(1023));
  const MkLayout L = mk_layout(a, a.n_stages);
  Ring ring;
  ring.base = sm + L.ring;
  ring.full = reinterpret_cast<uint64_t*>(sm + L.bars);
  ring.empty = ring.full + a.n_stages;
  ring.ns = a.n_stages;
  ring.it = 0;
  const int tid = threadIdx.x;
  if (tid == 0) {
    for (int s = 0; s < a.n_stages; ++s) {
      mbar_init(&ring.full[s], 1);
      mbar_init(&ring.empty[s], kMkWarps);
    }
    mbar_fence_init();
  }
  float* wacc = reinterpret_cast<float*>(sm + L.wacc);
  for (int i = tid; i < kMkWarps * a.rows_max * M; i += kMkThreads) wacc[i] = 0.f;
  // the zero block after the A planes (the A rows past 2 B)
  if (tid < 4) reinterpret_cast<uint32_t*>(sm + L.xw)[M * mk_plane(a) + tid] = 0u;
  __syncthreads();
  if (tid >= kMkCompute) {
    if (tid == kMkCompute) mk_producer<HD>(a, ring, blockIdx.x, gridDim.x);
    return;
  }
  mk_compute<M, HD>(a, ring, L, sm);
}

template <int M, int HD>
void set_mk_attr() {
  if (cudaFuncSetAttribute(mk_kernel<M, HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024) !=
      cudaSuccess)
    cudaGetLastError();   // the occupancy query then reports no room
}

void (*mk_pick(const MkArgs& a))(const MkArgs) {
  if (a.hd == 128) return a.B == 1 ? mk_kernel<1, 128> : mk_kernel<2, 128>;
  return a.B == 1 ? mk_kernel<1, 64> : mk_kernel<2, 64>;
}

void mk_attrs() {
  static PerDevice attr;
  attr.once([] {
    set_mk_attr<1, 128>();
    set_mk_attr<2, 128>();
    set_mk_attr<1, 64>();
    set_mk_attr<2, 64>();
  });
}

}  // namespace

int mk_ctas_per_sm(const MkArgs& a) {
  if (a.B < 1 || a.B > kMkMaxRows || (a.hd != 64 && a.hd != 128)) return 0;
  mk_attrs();
  int nb = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, mk_pick(a), kMkThreads, mk_smem_bytes(a, a.n_stages)) !=
      cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return nb;
}

cudaError_t launch_mk(const MkArgs& a, int n_ctas, cudaStream_t s) {
  mk_attrs();
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_ctas);
  cfg.blockDim = dim3(kMkThreads);
  cfg.dynamicSmemBytes = mk_smem_bytes(a, a.n_stages);
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeCooperative;   // every CTA resident: the phases wait on one another
  at[0].val.cooperative = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, mk_pick(a), a);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace dvi

// Internal interface between the C-ABI layer (dvi_api.cu) and the kernel
// translation units.  Host-side launchers only; no torch types anywhere.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/dvi.h"

namespace dvi {

enum Flavor : int {
  EPI_QKV = 0,     // RoPE on q/k, q -> q_out (f32), k/v -> KV cache rows
  EPI_RESID = 1,   // x += W.act, plus per-tile sums of squares for the next RMSNorm
  EPI_GATEUP = 2,  // h = SiLU(W_gate.n) * (W_up.n), two accumulators per tile
  EPI_HEAD = 3     // vocabulary logits (+ gamma A (B u)), stored and/or argmax
};

enum BMode : int {
  B_ACT = 0,       // B rows from an activation buffer in the model dtype (bf16: TMA via map `mb`)
  B_SOFT_F32 = 1   // bf16 path: float32 rows converted by warps 0-3 (dvi_linear)
};

constexpr int kBuRows = 16;   // rows of an in-kernel B u (the drafter head's batch)
constexpr int kBuRank = 16;   // LoRA rank of an in-kernel B u

struct ProjArgs {
  int flavor, b_mode, dtype;
  int M;              // token rows
  int n_pad;          // tcgen05 N: multiple of 16, >= M
  int n_out;          // rows of one weight (GATEUP: F, tiles of 64 gate + 64 up rows); QKV uses rows_q/k/v
  int K;              // input features
  int n_tiles, n_splits, kb_total, kb_per_split, n_ttiles;
  int prefetch_a;     // stream weight tiles before waiting for the previous kernel
  const void* w0;     // f32 path: weight pointers (QKV: wq, wk, wv; GATEUP: gate, up)
  const void* w1;
  const void* w2;
  int rows_q, rows_k, rows_v;
  // B operand: rows act_row0 .. act_row0+M-1 of act[.][ld_act]; bf16
  // activations hold a hi plane and a lo plane (value = hi + lo; the TMA
  // map `mb` is [2][rows][ld_act]), so the MMA runs over 2 n_pad columns
  const void* act; int ld_act; int act_row0;
  // Optional RMSNorm scale applied to every accumulator in the epilogue:
  // rstd[n] = rsqrt(sum_t ss[t*ss_ld + n] / d_norm + eps) (the norm gain is
  // already folded into the activation rows).
  const float* ss; int ss_ld; int ss_tiles; float eps; int d_norm;
  // token row -> (sequence, position)
  const int* lens; int rows_per_seq; int seq0; int pos_off;
  // split-K scratch: partial tiles and arrival counters (counters start at 0
  // and are reset to 0 by the CTA that reduces a tile)
  float* part; int* counters;
  int* status;
  // EPI_QKV
  float* q_out; int ld_q;
  void* kc; void* vc; int max_len; int head_dim;
  int n_kv_heads;
  const float2* rope;
  // EPI_RESID: x += y, per-tile sums of squares of the new x, and the next
  // projection's activation rows xg = x * g_next in the model dtype
  float* x_res; int ld_res; float* ss_out; int ss_out_ld;
  const float* g_next; void* xg_out; int ld_xg; size_t xg_plane;
  // EPI_GATEUP
  void* h_out; int ld_h; size_t h_plane;
  // EPI_HEAD
  float* logits_out; int ld_logits;
  int logits_mode;            // 0 none, 1 row n -> logits_out[n], 2 replay-buffer slot
  const int* log_step; int log_cap_steps; int log_rows_per_step;
  // mode 2: of each sequence's log_src_rows launch rows the log keeps the
  // first min(log_src_rows, log_dst_rows), at slots b * log_dst_rows +
  // log_dst_off + i of the step's rows
  int log_src_rows, log_dst_rows, log_dst_off;
  const float* lora_a; const float* lora_bu; int lora_r; float gamma;
  // bf16 drafter head, M <= kBuRows and lora_r <= kBuRank: B u computed by
  // the kernel itself (lora_bu unused), u = (x * rstd) * g from the f32
  // residual rows bu_x and the final-norm gain bu_g
  const float* lora_bmat; const float* bu_x; int bu_ldx; const float* bu_g;
  unsigned long long* amax;   // [M] argmax keys, or null
  // chained launch (decode passes): wait until *dep_wait >= dep_count (the
  // predecessor's CTAs), else for the predecessor's grid; add 1 to
  // *dep_signal after this CTA's last write (null: no signal)
  const int* dep_wait; int dep_count; int* dep_signal;
};

struct ProjMaps {
  CUtensorMap m0, m1, m2;     // bf16 path: TMA descriptors of w0, w1, w2
  CUtensorMap mb;             // bf16 path: the activation buffer (box 64 x 16 rows)
};

// Picks n_splits / kb_per_split from the weight shape only (never from M),
// so a row's result does not depend on how many rows share the launch.
void plan_splits(ProjArgs& a, int n_sms, bool tc);
size_t proj_partial_floats(const ProjArgs& a, bool tc);
bool make_weight_map(CUtensorMap* map, const void* w, int rows, int cols);
bool make_half_weight_map(CUtensorMap* map, const void* w, int rows, int cols);   // 64-row boxes (gate/up)
// W [rows][cols] (cols a multiple of 64) as [cols / 64][rows][64]: a box is
// `box_kblocks` consecutive tiles of `box_rows` rows x 64 columns, each tile
// 128-byte swizzled as a 2D box of that shape would be.
bool make_weight_map_kblocks(CUtensorMap* map, const void* w, int rows, int cols, int box_rows, int box_kblocks);
bool make_act_map(CUtensorMap* map, const void* act, int rows, int cols);   // [2 planes][rows][cols]
// The same activation buffer with boxes of `box_rows` (<= 256) rows.
bool make_act_map_box(CUtensorMap* map, const void* act, int rows, int cols, int box_rows);

// Prompt passes (bf16): the prefill kernel (prefill.cu) puts 128 token rows
// on the MMA's M side and 256 output features on N, persistent CTAs, two
// TMEM accumulators.  `a` is the decode launch's ProjArgs (flavours QKV,
// RESID, GATEUP; rows of one sequence); `act` maps the activation buffer
// with 128-row boxes; w0..w2 map the weights with 128-row boxes (QKV: wq,
// wk, wv; gate/up: gate, up).
struct PfMaps {
  CUtensorMap act, w0, w1, w2;
};
cudaError_t launch_proj_pf(const ProjArgs& a, const PfMaps& m, int n_sms, cudaStream_t s);

// Persistent projection chain (bf16): up to kChainMax projections of one
// pass in a single launch, each phase's output feeding the next phase's B
// operand (O, gate/up, down, next layer's QKV).  Every CTA takes an equal
// contiguous range of the phase's (tile, K block) sequence; a range that
// covers only part of a tile leaves its partial sum in `part`, and the last
// of the tile's CTAs to arrive sums the partials in K order and runs the
// epilogue.  A phase's activation loads wait for every tile of the phase
// before it (`phase_done`); its weight loads do not.
constexpr int kChainMax = 4;
constexpr int kChainTiles = 1024;   // tile counters per phase
constexpr int kChainMaxPad = 64;    // largest n_pad (two TMEM accumulators of 2 n_pad columns)
struct ChainArgs {
  CUtensorMap maps[kChainMax][4];   // per phase: m0, m1, m2, mb
  ProjArgs p[kChainMax];
  int n_phases;
  int n_ctas;             // grid size; fixed per context so the K ranges depend on the weight shape only
  int* phase_done;        // [kChainMax] finished tiles per phase (reset by the last CTA to leave)
  int* tile_ctr;          // [kChainMax][kChainTiles] arrivals per tile (reset by the tile's finisher)
  int* exit_ctr;
  float* part;            // [n_tiles + n_ctas][n_pad][128] partial slots (slot = tile + CTA)
};
// CTAs per SM the chain kernel keeps resident at n_pad (0 if it cannot run).
int chain_ctas_per_sm(int n_pad);
size_t chain_partial_floats(int max_tiles, int n_ctas, int n_pad);
cudaError_t launch_chain(const ChainArgs& a, cudaStream_t s);

struct AttnArgs {
  const float* q; int ld_q;          // rotated queries [M][H_q*hd]
  const void* kc; const void* vc;    // layer base of the caches [B][H_kv][max_len][hd]
  void* o; int ld_o;                 // output [M][H_q*hd] in `o_dtype` (bf16: hi/lo planes)
  size_t o_plane;
  int o_dtype;
  int dtype;                         // cache dtype
  int n_heads, n_kv_heads, head_dim, max_len;
  const int* lens; int rows_per_seq; int seq0; int n_seqs; int pos_off;
  int split_len;                     // positions per split (multiple of 64)
  int n_splits_max;
  float* part; int* counters;        // combine scratch
  int* status;
  float scale;
  long long kv_row0;                 // bf16 decode: row of (layer, seq 0, head 0, pos 0) in the cache maps
  const CUtensorMap* kmap;           // bf16 decode: the K / V caches as [rows][hd] (box 64 x 64)
  const CUtensorMap* vmap;
  int prefill;                       // a prompt pass (bf16, GQA group <= 8): the prefill attention kernel
  const int* dep_wait; int dep_count; int* dep_signal;   // chained launch (as ProjArgs; bf16 decode kernel)
};
// CTAs of the attention launch for these arguments.
int attn_grid_ctas(const AttnArgs& a);
// The decode attention kernel that takes part in completion-counter chaining
// (bf16 decode rows, at most kRegQ query heads per KV head).
bool attn_chainable(const AttnArgs& a);
bool make_kv_map(CUtensorMap* map, const void* cache, long long rows, int hd);
size_t attn_partial_floats(const AttnArgs& a);
int attn_counters(const AttnArgs& a);
cudaError_t launch_attn(const AttnArgs& a, cudaStream_t s);

// ---- small kernels (misc.cu)
struct EmbedArgs {
  const void* table; int dtype; int d; int vocab;
  const int* tokens;                 // device ids [rows]
  float* x; int ldx;                 // destination rows
  float* ss; int ss_ld;              // per-128-feature sums of squares [d/128][ss_ld]
  const float* g; void* xg; int ldxg;// activation rows x * g of the first projection (model dtype)
  size_t xg_plane;
  int rows;
  int* status;
};
cudaError_t launch_embed(const EmbedArgs& a, cudaStream_t s);

// Drafter-head preparation for draft pass j: u = RMSNorm_final(h_k) (logged
// into the replay buffer), LoRA B u, and the hand-off of h_k to the verify
// stream (x, its sums of squares, and x * g_copy for the verify's first layer).
struct HeadPrepArgs {
  const float* x; int ldx; int rows;
  const float* gain; float eps; int d;
  int dtype;
  float* x_copy; int ld_copy; int copy_row_stride; int copy_row_off;
  float* ss_copy; int ss_copy_ld;
  const float* g_copy; void* xg_copy; size_t xg_copy_plane;
  void* log_u; size_t log_plane; const int* log_step; int log_cap_steps; int log_rows_per_step; int log_row_stride;
  int log_row_off; int log_enabled;
  const float* lora_b; float* bu; int r;
};
cudaError_t launch_head_prep(const HeadPrepArgs& a, cudaStream_t s);

struct StepState {
  int B, K, d, vocab, max_len, dtype;
  int Kv, bonus;                                // verify rows per sequence (K + bonus)
  int* lens; int* pending; int* draft_ids;      // [B][K+1]
  float* x_dr; float* ss_dr; int ss_dr_ld;
  const float* g0; void* xg_dr;                 // first layer's attention-norm gain, x * g0
  size_t xg_dr_plane;
  const void* embed;
  unsigned long long* amax;
  int* out_ids; int* n_committed; int* n_accepted;
  int* log_meta; int* log_step; int log_cap_steps; int log_enabled;
  long long* counters;                          // steps, drafted, accepted, committed
  int* status;
};
// `prep` (or null): the pass's drafter-head preparation without B u, run
// before the next pass's embedding (the head computed B u itself).
cudaError_t launch_finalize_draft(const StepState& st, int j, const HeadPrepArgs* prep, cudaStream_t s);
cudaError_t launch_finalize_verify(const StepState& st, cudaStream_t s);
cudaError_t launch_finalize_ar(const StepState& st, cudaStream_t s);
cudaError_t launch_finalize_prefill(const StepState& st, int seq, int n_tokens, int32_t* first_out,
                                    cudaStream_t s);
cudaError_t launch_reset_seq(const StepState& st, int seq, cudaStream_t s);

// A finalize step run by the last CTA of a head projection (bf16, unsplit
// head): FIN_DRAFT after the drafter head of pass j (with the head
// preparation when `prep`), FIN_VERIFY after the verifier head, FIN_AR after
// the head of a greedy AR step.  `stage`: the head CTA has shared memory
// for the next pass's embedding rows.
enum FinKind : int { FIN_NONE = 0, FIN_DRAFT = 1, FIN_VERIFY = 2, FIN_AR = 3 };
struct FinArgs {
  int kind, j, prep, stage;
  int* ctr;          // arrivals of the head's CTAs; 0 before a launch, reset by the last CTA
  StepState st;
  HeadPrepArgs hp;
};
// Shared memory a finalize step needs in the head CTA (without staging).
size_t fin_smem_bytes();

cudaError_t launch_proj(const ProjArgs& a, const ProjMaps* maps, cudaStream_t s, const FinArgs* fin = nullptr);
// Whether a head launch of these arguments can run a finalize step, and
// whether its free shared memory holds `stage_bytes` of staged rows.
bool head_fin_ok(const ProjArgs& a, size_t stage_bytes, bool* stage);

// ---- drafter update (update.cu)
struct UpdateArgs {
  int cap, V, d, r, dtype, B, K;
  const void* log_u; size_t log_plane; const float* log_logits; int* log_meta; int* log_step;
  float* Z;                                     // [cap][V] drafter logits
  float* rowstat;                               // [cap][8]
  float* stat_part;                             // [cap][ceil(V / 2048)][9] merged parts of the row statistics
  float* coef;                                  // [cap][4] + globals
  float* ub;                                    // [cap][r]  U B^T
  float* ga;                                    // [cap][r]  G A
  float* ga_part; int* ga_counter; int n_vtiles;
  float* lora_a; float* lora_b; float gamma;
  float* m_a; float* v_a; float* m_b; float* v_b;
  float* grad_a; float* grad_b;
  // full-head mode: W^S (model dtype), its f32 master (bf16 only, else null),
  // Adam moments, G [cap][V], the optional gradient copy
  void* w_head; float* w_master; float* m_w; float* v_w; float* G; float* grad_w; int keep_grad_w;
  float* dev_state;                             // [0]=t, [1]=b, [2..] loss parts
  int* ctr;                                     // [4 + cap] last-CTA counters (rows done, update end, per
                                                // row; 0 between updates), grid barrier (count, generation)
  long long* counters;
  int* status;
  dvi_update_config cfg;
};
cudaError_t launch_update_prep(const UpdateArgs& a, cudaStream_t s);
cudaError_t launch_update_rowstats(const UpdateArgs& a, cudaStream_t s);
cudaError_t launch_update_grad_a(const UpdateArgs& a, cudaStream_t s);
cudaError_t launch_update_grad_b(const UpdateArgs& a, cudaStream_t s);
cudaError_t launch_update_full(const UpdateArgs& a, cudaStream_t s);
// LoRA mode: everything after the logits GEMM in one cooperative launch of
// ------------------------------------------------------------ draft-phase megakernel
// One persistent launch (one CTA per SM, every CTA resident) runs the
// shallow passes of a decode step (Sec. 3.3): the k draft layers of every
// draft pass with the drafter head, its argmax and the hand-off of h_k to the
// verify rows (MK_DRAFT), or the k shallow layers of one greedy AR step with
// the hand-off to the AR rows (MK_AR).  Phases (QKV, attention, O, gate/up,
// down, head) meet at release/acquire completion counters, one per phase
// boundary, with bounded polls.  bf16 weights only; at most kMkMaxRows
// sequences.
constexpr int kMkMaxLayers = 16;
constexpr int kMkMaxRows = 2;
constexpr int kMkMaxGroup = 8;     // query heads per KV head
enum MkMode : int { MK_DRAFT = 0, MK_AR = 1 };
struct MkLayerW {
  const void *wq, *wk, *wv, *wo, *wg, *wu, *wd;   // bf16 [out][in]
  const float *g_attn, *g_ffn;
};
struct MkArgs {
  MkLayerW layer[kMkMaxLayers];
  int mode;
  int B, k, d, Hq, Hkv, hd, F, V, max_len, K, Kv, r;
  const CUtensorMap* wmaps;   // [k][7] (wq, wk, wv, wo, wg, wu, wd), then W^S: 16 tiles of 8 rows x 64
  int P;                 // attention position splits per (sequence, KV head)
  int n_stages;          // weight ring stages of 16 KB
  int rows_max;          // output rows of one CTA in any phase
  int n_bound;           // completion counters (the abort flag follows them)
  float eps, gamma;
  const void* embed; const float* final_norm; const float* g_hand;
  const void* w_head; const float* lora_a; const float* lora_b;
  void* kc; void* vc;    // caches [L][B][H_kv][max_len][hd]; the first k layers are written
  const float2* rope;
  const int* lens; const int* pending; int* draft_ids;
  // hand-off of h_k: residual row, x * g_hand (hi/lo planes), per-tile sums of squares
  float* x_copy; int copy_row_stride; float* ss_copy; int ss_copy_ld; void* xg_copy; size_t xg_copy_plane;
  // replay buffer: u (hi/lo planes) and the drafter logits z of the logged tuples
  void* log_u; size_t log_plane; const int* log_step; int log_cap_steps; int log_enabled;
  float* zlog;
  // scratch
  float* xr;             // [2][B][d] residual stream (double buffered)
  float* qkv;            // [B][(H_q + 2 H_kv) hd] projections before RoPE
  float* att;            // [B][H_q][P][hd + 2] attention partials (max, sum, o)
  float* ao;             // [B][d] output projection
  float* hbuf;           // [B][F] SwiGLU
  float* y;              // [B][d] down projection
  float* bu_part;        // [n_ctas][r] partial B u
  unsigned long long* keys;   // [Kv][B] argmax keys, zero before the launch
  int* ctr;              // [n_bound + 1] zero before the launch
  int* status;
};
// Shared memory of the kernel with `n_stages` ring stages (0: too large).
size_t mk_smem_bytes(const MkArgs& a, int n_stages);
// Completion counters of one launch.
int mk_bounds(const MkArgs& a);
// Output rows of one CTA in the widest phase.
int mk_rows_max(const MkArgs& a, int n_ctas);
// CTAs of the kernel one SM holds with a.n_stages ring stages (0: none).
int mk_ctas_per_sm(const MkArgs& a);
cudaError_t launch_mk(const MkArgs& a, int n_ctas, cudaStream_t s);

// n_sms CTAs (grid barriers between its phases), when update_fused_ok.
bool update_fused_ok(const UpdateArgs& a, int n_sms);
cudaError_t launch_update_fused(const UpdateArgs& a, int n_sms, cudaStream_t s);
cudaError_t launch_master_init(const void* w_bf16, float* master, size_t n, cudaStream_t s);
cudaError_t launch_update_finish(const UpdateArgs& a, cudaStream_t s);

}  // namespace dvi

// Internal declarations shared by the libsdsat translation units.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace sdsat {

// ---- opt-in device trace: thread 0 of every CTA appends one record of TRACE_WORDS words:
// [0] tag << 32 | block, [1] flags << 32 | SM id, [2] t_entry, [3] t_after_wait,
// [4..6] three kernel-specific marks, [7] t_exit (%globaltimer, ns; 0 = not reached)
constexpr int TRACE_WORDS = 8;
struct Trace {
  unsigned long long* rec;   // [cap][TRACE_WORDS]
  unsigned int* count;
  unsigned int cap;
  unsigned int tag;          // kernel class << 24 | launch sequence number
};
__device__ __forceinline__ unsigned int sm_id() {
  unsigned int r;
  asm volatile("mov.u32 %0, %%smid;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void trace_write(const Trace& t, unsigned int flags, unsigned long long t0,
                                            unsigned long long tw, unsigned long long m0, unsigned long long m1,
                                            unsigned long long m2, unsigned long long t1) {
  if (!t.rec) return;
  const unsigned int i = atomicAdd(t.count, 1u);
  if (i >= t.cap) return;
  unsigned long long* r = t.rec + (size_t)i * TRACE_WORDS;
  r[0] = ((unsigned long long)t.tag << 32) | blockIdx.x;
  r[1] = ((unsigned long long)flags << 32) | sm_id();
  r[2] = t0;
  r[3] = tw;
  r[4] = m0;
  r[5] = m1;
  r[6] = m2;
  r[7] = t1;
}

// ---- skinny weight-streaming GEMM --------------------------------------------
// CTAs per SM of the skinny GEMM's grid for M <= 32 (compile-time tuning; one for M > 32).
// Every user of the grid size (the split-K partials, the fixed scratch of the
// scratch-free entry point) sizes its buffers from this constant.
#ifndef SDSAT_GEMM_CTAS_PER_SM
#define SDSAT_GEMM_CTAS_PER_SM 2
#endif
constexpr int GEMM_CTAS_PER_SM = SDSAT_GEMM_CTAS_PER_SM;
// Tiles of 128 output features x 64 K-elements; the 128 rows come from two
// 64-row TMA boxes ("halves") whose source depends on the map mode.
enum GemmMap : int {
  MAP_PLAIN = 0,    // one matrix [N][K]: tile t = rows 128t .. 128t+127
  MAP_QKV3 = 1,     // three matrices of rows_per_map rows each (q, k, v), stacked
  MAP_GATEUP = 2,   // two matrices [F][K]: tile t = gate rows 64t.. and up rows 64t..
};
enum GemmEpi : int {
  EPI_STORE = 0,    // out[m][n] = acc
  EPI_RESID = 1,    // out[m][n] += acc (residual stream)
  EPI_QKV = 2,      // RoPE on q, k; q -> out (fp32), k, v -> KV cache (bf16)
  EPI_SWIGLU = 3,   // out[m][j] = silu(gate) * up
};

struct GemmParams {
  CUtensorMap tmap[3];      // weights
  CUtensorMap tmap_x[2];    // activation operand: bf16 hi and lo [rows][K], box {64, MPAD}
  int map_mode;
  int N;              // output features (MAP_GATEUP: F)
  int K;
  int rows_per_map;   // MAP_QKV3: rows of each of q, k, v
  int n_tiles;
  int kc;             // K chunks of 64
  int P;              // CTAs
  int snap;           // stream-K split points within a tile's first `snap` units move to the tile start
  int M;              // activation rows (<= MPAD)
  // epilogue
  int epi;
  float* out;
  int out_ld;
  __nv_bfloat16* out_hi;    // EPI_SWIGLU: the down projection's operand, hi and lo parts
  __nv_bfloat16* out_lo;
  // RMSNorm folded into the GEMMs.  RMSNorm scales each row by one scalar, so the
  // operand can be stored un-normalised (h * gain) and the consuming GEMM multiplies
  // its result row m by rsqrt(sum_t ssq_in[m][t] / norm_dim + norm_eps).
  const float* ssq_in;      // [M][ssq_ld] partial sums of h^2, or null (operand already normalised)
  int ssq_n, ssq_ld;
  int norm_dim;
  float norm_eps;
  // EPI_RESID producer side: with gain_next set, also emit h * gain_next as the next
  // GEMM's bf16 hi + lo operand [M][N] and this tile's sums of h^2 into ssq_out[m][tile].
  const __nv_bfloat16* gain_next;
  __nv_bfloat16* xn_hi;
  __nv_bfloat16* xn_lo;
  float* ssq_out;
  // EPI_QKV
  __nv_bfloat16* k_layer;   // KV cache of this layer: [B][H][cap][hd]
  __nv_bfloat16* v_layer;
  int H, hd, cap, q, seq0;
  const int* len;           // committed lengths [B] (device)
  const int* positions;     // [M] or null
  const float2* rope;       // [rope_len][hd/2] (cos, sin)
  int rope_len;
  // scratch (exclusive to the running GEMM)
  float* partials;          // [P][2][MPAD][128]
  int* counters;            // [n_tiles], zero between launches
  uint32_t* err;
  Trace trace;
};

int gemm_mpad(int M);                 // 16, 32 or 64
size_t gemm_smem_bytes(int mpad);
cudaError_t gemm_prepare();           // set smem attributes (idempotent)
cudaError_t launch_gemm(GemmParams& p, int num_sms, cudaStream_t st, bool pdl);

// ---- attention -------------------------------------------------------------
constexpr int ATT_UNIT = 64;          // keys per work unit: one TMA box of cache rows
constexpr int ATT_MAX_CAP = 32768;    // KV capacity (slots per sequence) the kernel supports
constexpr int ATT_CS_MAX = 16;        // CTAs of one cluster: the most that share one (sequence, head)
#define SDSAT_ATT_MAXQ 16
struct AttnParams {
  CUtensorMap kmap;     // the K cache as a 2-D tensor [rows][hd] bf16, boxes of 64 dims x ATT_UNIT rows
  CUtensorMap vmap;     // the V cache, same geometry
  int row0;             // first row of this layer: cache row of (s, h, slot) = row0 + (s*H + h)*cap + slot
  const float* Q;       // [rows][q_ld] (row = sl*q + j), head h at column h*hd
  int q_ld;
  const int* len;       // [B]
  const uint32_t* anc;  // [nb*q] tree blocks: bit i of row j = row j attends block row i; null = causal
  int seq0, nb, q, H, hd, cap;
  float* out;           // [rows][out_ld] fp32
  int out_ld;
  __nv_bfloat16* out_hi;    // the same as bf16 hi + lo (the O projection's operand)
  __nv_bfloat16* out_lo;
  int cs, nclusters;    // set by launch_attention: CTAs per cluster, clusters in the grid
  uint32_t* err;
  Trace trace;
};
size_t attention_smem_bytes(int hd, int q);
cudaError_t attention_prepare();   // smem and cluster attributes, co-resident cluster counts (idempotent)
// grid: nclusters clusters of cs CTAs, all resident at once; cluster c takes the
// (sequence, head) pairs c, c + nclusters, ...; its CTAs split each pair's keys
cudaError_t launch_attention(const AttnParams& p, int num_sms, cudaStream_t st, bool pdl);
// the grid launch_attention picks for `pairs` (sequence, head) pairs: maxc[c] = most
// clusters of c CTAs resident at once (c = 1..ATT_CS_MAX), cluster size at most cs_cap
void attention_grid(int pairs, const int* maxc, int cs_cap, int num_sms, int* cs, int* nclusters);

// Causal attention of M consecutive prompt positions of sequence seq (a prefill chunk at
// slots len[seq] .. len[seq]+M-1, already in the cache) over the cache: position i sees
// slots [0, len + i].  One CTA per (head, 64-position block).
struct PfAttnParams {
  CUtensorMap kmap, vmap;   // the caches, as AttnParams
  int row0;                 // first cache row of this layer
  const float* Q;           // [M][q_ld] rotated queries, head h at column h*hd
  int q_ld;
  const int* len;
  int seq, M, H, hd, cap;
  float* out;               // [M][out_ld] fp32
  int out_ld;
  __nv_bfloat16* out_hi;    // the same as bf16 hi + lo (the O projection's operand)
  __nv_bfloat16* out_lo;
  uint32_t* err;
};
cudaError_t launch_prefill_attention(const PfAttnParams& p, cudaStream_t st, bool pdl);

// ---- prefill (prompt chunks of up to PF_ROWS positions) -------------------------
constexpr int PF_ROWS = 512;
struct PfGemmParams {
  CUtensorMap tmap[3];      // weights, as GemmParams::tmap (map_mode)
  CUtensorMap tmap_x[2];    // positions' operand, bf16 hi / lo [PF_ROWS][K], boxes of 64 x 128
  int map_mode, rows_per_map;
  int N;                    // output features (MAP_GATEUP: F)
  int kc;                   // 64-column chunks of K
  int n_wtiles, n_tblocks;  // tiles of 128 weight rows, blocks of 128 positions
  int M;                    // positions
  int epi;                  // EPI_STORE, EPI_RESID or EPI_SWIGLU
  float* out;               // [M][out_ld] fp32 (EPI_STORE, EPI_RESID)
  int out_ld;
  __nv_bfloat16* out_hi;    // EPI_SWIGLU: [M][out_ld] the down projection's operand
  __nv_bfloat16* out_lo;
  uint32_t* err;
};
cudaError_t prefill_prepare();
cudaError_t launch_prefill_gemm(PfGemmParams& p, int num_sms, cudaStream_t st, bool pdl);
struct RopeKvParams {
  const float* qkv;         // [M][3R]
  float* qout;              // [M][R]
  __nv_bfloat16* k_layer;   // this layer's caches [B][H][cap][hd]
  __nv_bfloat16* v_layer;
  const int* len;
  int seq, H, hd, cap;
  const float2* rope;
  int rope_len;
  uint32_t* err;
};
cudaError_t launch_rope_kv(const RopeKvParams& p, int M, cudaStream_t st, bool pdl);

// ---- embedding, acceptance, block building ------------------------------------
// x = h * rsqrt(mean h^2 + eps) * g, stored as bf16 hi + lo (tokens != null: h = E[tokens] first)
cudaError_t launch_rmsnorm(const int* tokens, const __nv_bfloat16* E, int V, float* h, int d, int M,
                           const __nv_bfloat16* gain, float eps, __nv_bfloat16* xhi, __nv_bfloat16* xlo,
                           uint32_t* err, cudaStream_t st, bool pdl);
// fp32 [M][K] -> bf16 hi + lo
cudaError_t launch_split(const float* x, int M, int K, __nv_bfloat16* xhi, __nv_bfloat16* xlo, cudaStream_t st,
                         bool pdl);

struct AcceptParams {
  const float* logits;      // [nb*q][V]
  const int* drafts;        // [nb*q]
  int seq0, nb, q, V, n_verify;
  float temperature, top_p;
  uint32_t p_fixed;         // round(top_p * 2^24)
  uint64_t seed;
  int top_k;
  int* len;                 // [B] committed lengths
  int cap;
  int commit;
  int* accepted_len;        // [nb]
  int* out_tokens;          // [nb*q]
  int* targets;             // scratch [nb*q]
  int* counters;            // scratch [nb], zero between launches
  long long* emitted;       // [B] tokens emitted per sequence (commit only), or null
  const int* n_verify_dev;  // [nb] drafts verified per sequence (pipelined blocks); null: n_verify
  const int* parent;        // tree blocks: [nb*q] parent row of every row (row 0: -1); null = chain
  int* path;                // tree blocks: [nb*q] accepted path rows, -1 past its end (optional)
  int* tree_ws;             // tree blocks: [nb][TREE_WS_STRIDE] len before the step, m, path rows
  uint32_t* err;
};
constexpr int TREE_WS_STRIDE = SDSAT_ATT_MAXQ + 2;
constexpr int TREE_MAX_ROWS = 64;   // rows of one block forward (the tree kernels run one thread per row)
cudaError_t launch_accept(const AcceptParams& p, cudaStream_t st, bool pdl);

struct BuildParams {
  int mode;                 // 1: draft step 1 block, 2: draft step 2 block
  const int* prev_out;      // [nb][prev_q] the previous block's emitted tokens
  int prev_q;
  const int* prev_acc;      // [nb] its accepted lengths
  const int* table;         // [width][table_batch][table_stride] draft tables, or null
  int table_stride, table_batch;
  const int* len;           // [B] committed lengths
  const int* adaptive;      // [SDSAT_MAX_ADAPTIVE] adaptive token ids
  int nb, q, k;             // q rows per sequence; mode 2: q = 1 + width * k; mode 3: q = 2k + 1
  int* tokens;              // [nb][q]
  int* pipe_mode;           // mode 3: [nb] in: the previous block's mode, out: this block's (0 S, 1 A)
  int* pipe_nverify;        // mode 3: [nb] out: drafts this block verifies (k in mode A, 0 in S)
};
cudaError_t launch_build_block(const BuildParams& b, cudaStream_t st, bool pdl);
// tree block rows: positions len + depth and the attention masks (ancestors and self)
cudaError_t launch_tree_prep(const int* parent, const int* len, int nb, int q, int* pos, uint32_t* anc,
                             uint32_t* err, cudaStream_t st, bool pdl);
// move the accepted path's K / V rows to contiguous slots (input: AcceptParams::tree_ws)
cudaError_t launch_tree_compact(const int* ws, int nb, int L, int H, int hd, int cap, int batch,
                                __nv_bfloat16* k, __nv_bfloat16* v, cudaStream_t st, bool pdl);
cudaError_t launch_commit(int* len, const int* new_len, int nb, int cap, uint32_t* err, cudaStream_t st,
                          bool pdl);
cudaError_t launch_add_len(int* len, int seq, int n, int cap, uint32_t* err, cudaStream_t st, bool pdl);
cudaError_t launch_exp(const float* in, float* out, int n, cudaStream_t st);
// a bounded wait that nothing satisfies: sets ERR_TIMEOUT after WAIT_LIMIT_NS (test hook)
cudaError_t launch_wait_timeout(uint32_t* err, cudaStream_t st);

}  // namespace sdsat

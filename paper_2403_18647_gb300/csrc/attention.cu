// Block-causal attention of the q block rows against the KV cache (flash decoding).
//
// In one block forward, row j of sequence s attends to the committed slots
// [0, len[s]) and to block rows 0..j (slots len[s] .. len[s]+j), which the QKV
// epilogue has just written; this is how Eq. 1-2 evaluate every appended
// position of the block in one pass.  The bytes are the K and V rows (bf16,
// hd*2 bytes each), read once per (sequence, head) for all q rows together.
//
// Work is split into units of ATT_UNIT = 64 consecutive slots of one
// (sequence, head), ordered (sequence, head, unit).  One wave of P CTAs (two
// per SM) reads the committed lengths, counts the U units and takes the
// contiguous range [iU/P, (i+1)U/P): every CTA streams the same number of
// K/V bytes.  One thread keeps a two-stage ring of K and V tiles (TMA, boxes
// of 64 dims x 64 rows, 128-byte swizzle) full; tiles made of committed slots
// only are requested before the QKV projection has finished, and the next
// ATT_PREFETCH tiles are kept on their way into L2.  Per unit, on
// the tensor cores (mma.sync m16n8k16, the q <= 16 rows fill the M = 16
// tile): S = Q K^T with each warp on 16 keys, an online-softmax update of the
// running row max and exp-sum (row reductions through shared memory), then
// O = O * alpha + P V with each warp on hd/4 dimensions.  Q and P enter as
// bf16 hi + lo pairs (two MMAs each), K and V are the cache's own bf16
// values, accumulation is fp32.
//
// A CTA's run of units of one (sequence, head) ends in a partial result (row
// max, exp-sum, unnormalised output).  The last of the <= ATT_SEG_MAX CTAs
// sharing the pair (per-pair counter, no waiting) merges the partials in CTA
// order with the usual log-sum-exp rescaling -- deterministic -- and writes
// the output in fp32 and as the O projection's bf16 hi + lo operand.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace sdsat {

constexpr int ATT_STAGES = 2;
constexpr int ATT_PREFETCH = 4;   // units past the ring requested into L2 ahead of their loads

template <int HD>
struct AttCfg {
  static constexpr int HALVES = HD / 64;                 // 64-dim column boxes per row
  static constexpr int HALF_BYTES = ATT_UNIT * 128;      // one box: 64 rows x 64 dims bf16
  static constexpr int TILE = HALF_BYTES * HALVES;       // K (or V) of one unit
  static constexpr int STAGE = 2 * TILE;                 // K then V
  static constexpr int QSTRIDE = HD * 2 + 16;            // bytes per row of the bf16 Q tiles (padded)
  static constexpr int PSTRIDE = ATT_UNIT * 2 + 16;      // bytes per row of the bf16 P tiles (padded)
  static constexpr int RED = 17;                         // floats per row of the row-reduction scratch
  static constexpr size_t OFF_Q = (size_t)ATT_STAGES * STAGE;
  static constexpr size_t OFF_P = OFF_Q + 2 * 16 * QSTRIDE;
  static constexpr size_t OFF_RED = OFF_P + 2 * 16 * PSTRIDE;                       // [16][RED]
  static constexpr size_t OFF_ROW = OFF_RED + 16 * RED * 4;                         // m, l, alpha [16]
  static constexpr size_t OFF_MERGE = OFF_ROW + 3 * 16 * 4;                         // ms, ls, w [16][SEG], inv [16]
  static constexpr size_t OFF_SEQ = OFF_MERGE + (3 * 16 * ATT_SEG_MAX + 16) * 4;    // len, units [64], first unit [65]
  static constexpr size_t OFF_BAR = (OFF_SEQ + (64 + 64 + 65) * 4 + 7) / 8 * 8;
  static constexpr size_t SMEM = 1024 + OFF_BAR + ATT_STAGES * 8 + 16;
};

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
// D (16x8 fp32) += A (16x16 bf16, row) * B (16x8 bf16, col)
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                               uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo_elem, float hi_elem) {
  return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(lo_elem)) |
         ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(hi_elem)) << 16);
}

// CTA owning unit u when U units are split over P CTAs as [iU/P, (i+1)U/P)
__device__ __forceinline__ int att_cta_of(int u, int U, int P) {
  return (int)(((long long)(u + 1) * P - 1) / U);
}

template <int HD>
__global__ void __launch_bounds__(128) attention_kernel(const __grid_constant__ AttnParams p) {
  using C = AttCfg<HD>;
  constexpr int KSTEPS = HD / 16;          // MMA k-steps over the head dimension
  constexpr int DT = HD / 32;              // 8-wide dimension tiles per warp in P.V
  constexpr int D4 = HD / 4;               // float4 columns of an output row
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* Qh = smem + C::OFF_Q;                    // bf16 [16][HD] (scaled q, hi part), padded rows
  uint8_t* Ql = Qh + 16 * C::QSTRIDE;               // lo part
  uint8_t* Ph = smem + C::OFF_P;                    // bf16 [16][ATT_UNIT] softmax numerators, hi part
  uint8_t* Pl = Ph + 16 * C::PSTRIDE;
  float* red = reinterpret_cast<float*>(smem + C::OFF_RED);     // [16 rows][RED]: one value per (warp, quad lane)
  float* m_run = reinterpret_cast<float*>(smem + C::OFF_ROW);   // [16] running row max
  float* l_run = m_run + 16;                                    // [16] running exp-sum
  float* alpha = l_run + 16;                                    // [16] rescale of the units before
  float* ms = reinterpret_cast<float*>(smem + C::OFF_MERGE);    // [16][ATT_SEG_MAX] partial maxima
  float* ls = ms + 16 * ATT_SEG_MAX;                            // partial exp-sums
  float* wg = ls + 16 * ATT_SEG_MAX;                            // merge weights
  float* inv = wg + 16 * ATT_SEG_MAX;                           // [16] 1 / L
  int* len_seq = reinterpret_cast<int*>(smem + C::OFF_SEQ);     // [64] committed length of each sequence
  int* nu_seq = len_seq + 64;                                   // [64] units per head of each sequence
  int* base = nu_seq + 64;                                      // [65] first unit of each sequence
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);   // [ATT_STAGES] K and V of the stage landed
  volatile int* abort_flag = reinterpret_cast<volatile int*>(full + ATT_STAGES);
  int* s_last = reinterpret_cast<int*>(full + ATT_STAGES) + 1;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, tig = lane & 3;
  const int mi = lane >> 3, r8 = lane & 7;        // ldmatrix: this thread's matrix and row
  const int q = p.q, H = p.H;
  const unsigned long long t_entry = p.trace.rec ? globaltimer_ns() : 0;
  pdl_trigger();

  // The committed lengths are final before this kernel can start: the block forward's
  // first kernel (RMSNorm) lets its dependents launch only after every earlier kernel
  // has completed.  Slots below them are not written during this forward either.
  if (tid < p.nb) {
    const int len = __ldcg(p.len + p.seq0 + tid);
    len_seq[tid] = len;
    nu_seq[tid] = (min(len + q, p.cap) + ATT_UNIT - 1) / ATT_UNIT;
  }
  if (tid == 0) {
    for (int s = 0; s < ATT_STAGES; ++s) mbar_init(&full[s], 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (tid == 0) {
    int acc = 0;
    for (int s = 0; s < p.nb; ++s) {
      base[s] = acc;
      acc += H * nu_seq[s];
    }
    base[p.nb] = acc;
  }
  __syncthreads();
  const int U = base[p.nb];
  const int P = min((int)gridDim.x, U);           // every CTA below P owns at least one unit
  const int cta = blockIdx.x;
  if (cta >= P) return;
  const int u0 = (int)((long long)cta * U / P), u1 = (int)((long long)(cta + 1) * U / P);
  const int n = u1 - u0;

  // unit u -> (sequence sl, head h, unit c of the pair)
  auto locate = [&](int u, int& s, int& hh, int& cc) {
    s = 0;
    while (base[s + 1] <= u) ++s;
    const int r = u - base[s];
    hh = r / nu_seq[s];
    cc = r % nu_seq[s];
  };
  // first cache row of unit u, and whether all of its slots are committed
  auto unit_row = [&](int u, bool& committed) {
    int s, hh, cc;
    locate(u, s, hh, cc);
    committed = (cc + 1) * ATT_UNIT <= len_seq[s];
    return p.row0 + ((p.seq0 + s) * H + hh) * p.cap + cc * ATT_UNIT;
  };
  uint64_t pol = 0;
  auto issue = [&](int k, int row) {   // unit u0 + k into stage k % ATT_STAGES
    uint8_t* st = smem + (size_t)(k % ATT_STAGES) * C::STAGE;
    uint64_t* bar = &full[k % ATT_STAGES];
    mbar_arrive_expect_tx(bar, C::STAGE);
#pragma unroll
    for (int hh = 0; hh < C::HALVES; ++hh) tma_load_2d(st + hh * C::HALF_BYTES, &p.kmap, bar, hh * 64, row, pol);
#pragma unroll
    for (int hh = 0; hh < C::HALVES; ++hh)
      tma_load_2d(st + C::TILE + hh * C::HALF_BYTES, &p.vmap, bar, hh * 64, row, pol);
  };
  auto prefetch = [&](int row) {   // a unit's K and V tiles into L2
#pragma unroll
    for (int hh = 0; hh < C::HALVES; ++hh) {
      tma_prefetch_l2_2d(&p.kmap, hh * 64, row);
      tma_prefetch_l2_2d(&p.vmap, hh * 64, row);
    }
  };
  int issued = 0;   // units whose loads were issued (thread 0)
  if (tid == 0) {
    tma_prefetch_desc(&p.kmap);
    tma_prefetch_desc(&p.vmap);
    pol = l2_policy_evict_first();
    // Tiles of committed slots do not depend on the QKV projection: the first ones go
    // to the ring now, the next ATT_PREFETCH into L2 (and one more each time the ring is
    // refilled), so that the ring's loads are L2 hits instead of HBM round trips.
    for (; issued < min(n, ATT_STAGES); ++issued) {
      bool committed;
      const int row = unit_row(u0 + issued, committed);
      if (!committed) break;
      issue(issued, row);
    }
    for (int k = ATT_STAGES; k < min(n, ATT_STAGES + ATT_PREFETCH); ++k) {
      bool committed;
      const int row = unit_row(u0 + k, committed);
      if (committed) prefetch(row);
    }
  }
  pdl_wait();   // q and this forward's new K/V rows come from the QKV projection
  const unsigned long long t_wait = p.trace.rec ? globaltimer_ns() : 0;
  if (tid == 0) {
    for (; issued < min(n, ATT_STAGES); ++issued) {
      bool committed;
      issue(issued, unit_row(u0 + issued, committed));
    }
  }
  unsigned long long t_k = 0, t_part = 0, t_merge = 0;
  unsigned merges = 0;

  const float scale = rsqrtf((float)HD);
  const int kb = warp * 16;                       // first key (within the unit) of this warp's scores
  const int db = warp * (HD / 4);                 // first dimension of this warp's outputs
  float O[DT][4], Ol[DT][4];   // P.V with the hi and with the lo part of P, summed when published
  int sl = 0, h = 0, c = 0;
  locate(u0, sl, h, c);
  int seg_first = u0;                             // first unit of the current (sequence, head) run
  for (int k = 0; k < n; ++k) {
    const int u = u0 + k;
    if (u == seg_first) {
      // ---- a new (sequence, head): q (scaled by 1/sqrt(hd)) as bf16 hi + lo, rows >= q zero
      for (int i = tid; i < 16 * (HD / 2); i += 128) {
        const int j = i / (HD / 2), d = (i % (HD / 2)) * 2;
        float x0 = 0.f, x1 = 0.f;
        if (j < q) {
          const float2 v = __ldcg(reinterpret_cast<const float2*>(p.Q + (size_t)(sl * q + j) * p.q_ld + h * HD + d));
          x0 = v.x * scale;
          x1 = v.y * scale;
        }
        const __nv_bfloat16 h0 = __float2bfloat16_rn(x0), h1 = __float2bfloat16_rn(x1);
        *reinterpret_cast<uint32_t*>(Qh + j * C::QSTRIDE + d * 2) =
            (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
        *reinterpret_cast<uint32_t*>(Ql + j * C::QSTRIDE + d * 2) =
            pack_bf16(x0 - __bfloat162float(h0), x1 - __bfloat162float(h1));
      }
      if (tid < 16) {
        m_run[tid] = -INFINITY;
        l_run[tid] = 0.f;
      }
#pragma unroll
      for (int nt = 0; nt < DT; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) O[nt][e] = Ol[nt][e] = 0.f;
      __syncthreads();
    }
    const int len = len_seq[sl];
    const int nkeys = min(len + q, p.cap);
    const int c0 = c * ATT_UNIT;                  // slot of the unit's first key
    const uint8_t* Kt = smem + (size_t)(k % ATT_STAGES) * C::STAGE;
    const uint8_t* Vt = Kt + C::TILE;
    const bool ok = mbar_wait_bounded(&full[k % ATT_STAGES], (k / ATT_STAGES) & 1, abort_flag, p.err);
    __syncwarp();   // lanes leave the polling loop at different times: reconverge
    if (k == 0 && p.trace.rec) t_k = globaltimer_ns();

    // ---- S = Q K^T for this warp's 16 keys (2 tiles of 8), fp32 in registers
    float S[2][4], Sl[2][4];   // products with the hi and the lo part of q, summed after the loop
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) S[nt][e] = Sl[nt][e] = 0.f;
    if (ok) {
#pragma unroll
      for (int kk = 0; kk < KSTEPS; ++kk) {
        uint32_t ah[4], al[4];
        const int qrow = r8 + 8 * (mi & 1), qcol = kk * 16 + 8 * (mi >> 1);
        ldsm_x4(smem_u32(Qh + qrow * C::QSTRIDE + qcol * 2), ah[0], ah[1], ah[2], ah[3]);
        ldsm_x4(smem_u32(Ql + qrow * C::QSTRIDE + qcol * 2), al[0], al[1], al[2], al[3]);
        const int hh = kk >> 2, cg = 2 * (kk & 3);  // 64-dim half and first 16-byte granule
        const int key = kb + 8 * (mi >> 1) + r8;
        const int cc = cg + (mi & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(smem_u32(Kt + hh * C::HALF_BYTES + key * 128 + ((cc ^ (key & 7)) << 4)), b0, b1, b2, b3);
        mma_bf16_16816(S[0], ah[0], ah[1], ah[2], ah[3], b0, b1);
        mma_bf16_16816(Sl[0], al[0], al[1], al[2], al[3], b0, b1);
        mma_bf16_16816(S[1], ah[0], ah[1], ah[2], ah[3], b2, b3);
        mma_bf16_16816(Sl[1], al[0], al[1], al[2], al[3], b2, b3);
      }
#pragma unroll
      for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) S[nt][e] += Sl[nt][e];
    }
    // mask: row j sees key slot kp iff kp <= len + j (and kp < nkeys, j < q)
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int j = g + 8 * (e >> 1);
        const int kp = c0 + kb + 8 * nt + 2 * tig + (e & 1);
        if (!ok || j >= q || kp >= nkeys || kp > len + j) S[nt][e] = -INFINITY;
      }
    // ---- the unit's row max -> running max, and the rescale of the units before
    red[g * C::RED + warp * 4 + tig] = fmaxf(fmaxf(S[0][0], S[0][1]), fmaxf(S[1][0], S[1][1]));
    red[(g + 8) * C::RED + warp * 4 + tig] = fmaxf(fmaxf(S[0][2], S[0][3]), fmaxf(S[1][2], S[1][3]));
    __syncthreads();
    if (tid < 16) {
      float mc = -INFINITY;
#pragma unroll
      for (int i = 0; i < 16; ++i) mc = fmaxf(mc, red[tid * C::RED + i]);
      const float mo = m_run[tid], mn = fmaxf(mo, mc);
      alpha[tid] = (mn == -INFINITY) ? 1.f : expf(mo - mn);
      m_run[tid] = mn;
    }
    __syncthreads();
    // ---- P = exp(S - m) as bf16 hi + lo, and its row sums
    const float mr0 = m_run[g], mr1 = m_run[g + 8];
    float l0 = 0.f, l1 = 0.f;
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
      float pv[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) pv[e] = (S[nt][e] == -INFINITY) ? 0.f : expf(S[nt][e] - ((e < 2) ? mr0 : mr1));
      l0 += pv[0] + pv[1];
      l1 += pv[2] + pv[3];
      const int key = kb + 8 * nt + 2 * tig;
      const __nv_bfloat16 h0 = __float2bfloat16_rn(pv[0]), h1 = __float2bfloat16_rn(pv[1]);
      const __nv_bfloat16 h2 = __float2bfloat16_rn(pv[2]), h3 = __float2bfloat16_rn(pv[3]);
      *reinterpret_cast<uint32_t*>(Ph + g * C::PSTRIDE + key * 2) =
          (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
      *reinterpret_cast<uint32_t*>(Ph + (g + 8) * C::PSTRIDE + key * 2) =
          (uint32_t)__bfloat16_as_ushort(h2) | ((uint32_t)__bfloat16_as_ushort(h3) << 16);
      *reinterpret_cast<uint32_t*>(Pl + g * C::PSTRIDE + key * 2) =
          pack_bf16(pv[0] - __bfloat162float(h0), pv[1] - __bfloat162float(h1));
      *reinterpret_cast<uint32_t*>(Pl + (g + 8) * C::PSTRIDE + key * 2) =
          pack_bf16(pv[2] - __bfloat162float(h2), pv[3] - __bfloat162float(h3));
    }
    red[g * C::RED + warp * 4 + tig] = l0;
    red[(g + 8) * C::RED + warp * 4 + tig] = l1;
    __syncthreads();   // P tiles and the row sums are complete
    if (tid < 16) {
      float lc = 0.f;
#pragma unroll
      for (int i = 0; i < 16; ++i) lc += red[tid * C::RED + i];
      l_run[tid] = l_run[tid] * alpha[tid] + lc;
    }
    // ---- O = O * alpha + P V for this warp's HD/4 dimensions (DT tiles of 8), all 64 keys
    {
      const float a0 = alpha[g], a1 = alpha[g + 8];
#pragma unroll
      for (int nt = 0; nt < DT; ++nt) {
        O[nt][0] *= a0;
        O[nt][1] *= a0;
        O[nt][2] *= a1;
        O[nt][3] *= a1;
        Ol[nt][0] *= a0;
        Ol[nt][1] *= a0;
        Ol[nt][2] *= a1;
        Ol[nt][3] *= a1;
      }
    }
    if (ok) {
#pragma unroll
      for (int kk = 0; kk < ATT_UNIT / 16; ++kk) {
        uint32_t ah[4], al[4];
        const int prow = r8 + 8 * (mi & 1), pcol = kk * 16 + 8 * (mi >> 1);
        ldsm_x4(smem_u32(Ph + prow * C::PSTRIDE + pcol * 2), ah[0], ah[1], ah[2], ah[3]);
        ldsm_x4(smem_u32(Pl + prow * C::PSTRIDE + pcol * 2), al[0], al[1], al[2], al[3]);
#pragma unroll
        for (int np = 0; np < DT / 2; ++np) {       // two dimension tiles per ldmatrix.x4.trans
          const int key = kk * 16 + 8 * (mi & 1) + r8;
          const int dim = db + 8 * (2 * np + (mi >> 1));
          const int hh = dim >> 6, cc = (dim & 63) >> 3;
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(smem_u32(Vt + hh * C::HALF_BYTES + key * 128 + ((cc ^ (key & 7)) << 4)), b0, b1, b2, b3);
          mma_bf16_16816(O[2 * np], ah[0], ah[1], ah[2], ah[3], b0, b1);
          mma_bf16_16816(Ol[2 * np], al[0], al[1], al[2], al[3], b0, b1);
          mma_bf16_16816(O[2 * np + 1], ah[0], ah[1], ah[2], ah[3], b2, b3);
          mma_bf16_16816(Ol[2 * np + 1], al[0], al[1], al[2], al[3], b2, b3);
        }
      }
    }
    __syncthreads();   // the stage, P and the row statistics are consumed
    if (tid == 0 && issued < n && !*abort_flag) {   // refill the freed stage, extend the L2 window
      bool committed;
      issue(issued, unit_row(u0 + issued, committed));
      if (issued + ATT_PREFETCH < n) prefetch(unit_row(u0 + issued + ATT_PREFETCH, committed));
      ++issued;
    }

    // ---- end of this CTA's run of units of the pair: publish the partial result
    const int nu = nu_seq[sl];
    if (k == n - 1 || c == nu - 1) {
      const int hu0 = base[sl] + h * nu;                       // the pair's units [hu0, hu0 + nu)
      const int j0 = att_cta_of(hu0, U, P), j1 = att_cta_of(hu0 + nu - 1, U, P);
      const int slot = cta - j0, nseg = j1 - j0 + 1;           // <= (nu-1)P/U + 2 <= P/H + 2 <= ATT_SEG_MAX
      const size_t pair = (size_t)h * ATT_SEG_MAX;
      const bool fits = nseg <= ATT_SEG_MAX;                   // always, for grids launch_attention makes
      if (!fits && tid == 0) set_error(p.err, ERR_CAPACITY);
      if (tid < q && fits) {   // m_run[tid] and l_run[tid] were last written by this thread
        float* ml = p.part_ml + ((size_t)(sl * q + tid) * H * ATT_SEG_MAX + pair + slot) * 2;
        ml[0] = m_run[tid];
        ml[1] = l_run[tid];
      }
#pragma unroll
      for (int nt = 0; nt < DT; ++nt)
#pragma unroll
        for (int e = 0; e < 4; e += 2) {
          const int j = g + 8 * (e >> 1);
          if (j < q && fits) {
            const int dim = db + 8 * nt + 2 * tig;
            *reinterpret_cast<float2*>(p.part_o + ((size_t)(sl * q + j) * H * ATT_SEG_MAX + pair + slot) * HD + dim) =
                make_float2(O[nt][e] + Ol[nt][e], O[nt][e + 1] + Ol[nt][e + 1]);
          }
        }
      if (p.trace.rec) t_part = globaltimer_ns();
      // the CTA's stores, then one release/acquire counter update by thread 0
      __syncthreads();
      if (tid == 0) {
        __threadfence();
        *s_last = (atomicAdd(p.counters + sl * H + h, 1) == nseg - 1);
        __threadfence();
      }
      __syncthreads();
      if (*s_last && fits) {
        // ---- merge the pair's partials: w[j][s] = exp(m_s - max m), L_j = sum_s w[j][s] l_s
        for (int t = tid; t < q * nseg; t += 128) {
          const int j = t / nseg, s = t % nseg;
          const float2 v = __ldcg(reinterpret_cast<const float2*>(
              p.part_ml + ((size_t)(sl * q + j) * H * ATT_SEG_MAX + pair + s) * 2));
          ms[j * ATT_SEG_MAX + s] = v.x;
          ls[j * ATT_SEG_MAX + s] = v.y;
        }
        __syncthreads();
        if (tid < q) {
          float mx = -INFINITY;
          for (int s = 0; s < nseg; ++s) mx = fmaxf(mx, ms[tid * ATT_SEG_MAX + s]);
          float L = 0.f;
          for (int s = 0; s < nseg; ++s) {
            const float m = ms[tid * ATT_SEG_MAX + s];
            const float w = (m == -INFINITY) ? 0.f : expf(m - mx);
            wg[tid * ATT_SEG_MAX + s] = w;
            L += w * ls[tid * ATT_SEG_MAX + s];
          }
          inv[tid] = 1.0f / L;
        }
        __syncthreads();
        // O_j = (sum_s w[j][s] o_s) / L_j: one (row, 4 dimensions) per thread, all partials in flight
        for (int t = tid; t < q * D4; t += 128) {
          const int j = t / D4, d4 = t % D4;
          const float4* po =
              reinterpret_cast<const float4*>(p.part_o + ((size_t)(sl * q + j) * H * ATT_SEG_MAX + pair) * HD) + d4;
          float4 v[ATT_SEG_MAX];
#pragma unroll
          for (int s = 0; s < ATT_SEG_MAX; ++s)
            if (s < nseg) v[s] = __ldcg(po + (size_t)s * D4);
          float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
          for (int s = 0; s < ATT_SEG_MAX; ++s) {
            if (s < nseg) {
              const float w = wg[j * ATT_SEG_MAX + s];
              a.x += w * v[s].x;
              a.y += w * v[s].y;
              a.z += w * v[s].z;
              a.w += w * v[s].w;
            }
          }
          const float iv = inv[j];
          const float4 o = make_float4(a.x * iv, a.y * iv, a.z * iv, a.w * iv);
          const size_t idx = (size_t)(sl * q + j) * p.out_ld + h * HD + 4 * d4;
          *reinterpret_cast<float4*>(p.out + idx) = o;
          const __nv_bfloat16 h0 = __float2bfloat16_rn(o.x), h1 = __float2bfloat16_rn(o.y);
          const __nv_bfloat16 h2 = __float2bfloat16_rn(o.z), h3 = __float2bfloat16_rn(o.w);
          uint2 hi, lo;
          hi.x = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
          hi.y = (uint32_t)__bfloat16_as_ushort(h2) | ((uint32_t)__bfloat16_as_ushort(h3) << 16);
          lo.x = pack_bf16(o.x - __bfloat162float(h0), o.y - __bfloat162float(h1));
          lo.y = pack_bf16(o.z - __bfloat162float(h2), o.w - __bfloat162float(h3));
          *reinterpret_cast<uint2*>(p.out_hi + idx) = hi;
          *reinterpret_cast<uint2*>(p.out_lo + idx) = lo;
        }
        if (tid == 0) p.counters[sl * H + h] = 0;
        ++merges;
        if (p.trace.rec) t_merge = globaltimer_ns();
        __syncthreads();   // merge scratch free again
      }
      if (k + 1 < n) {     // the next unit starts the next pair
        seg_first = u + 1;
        locate(u + 1, sl, h, c);
      }
    } else {
      ++c;
    }
  }
  if (*abort_flag && tid == 0) {   // let the copies in flight land before the CTA exits
    for (int i = max(0, issued - ATT_STAGES); i < issued; ++i) {
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&full[i % ATT_STAGES], (i / ATT_STAGES) & 1))
        if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) break;
    }
  }
  if (tid == 0 && p.trace.rec)
    trace_write(p.trace, merges | ((unsigned)n << 8), t_entry, t_wait, t_k, t_part, t_merge, globaltimer_ns());
}

size_t attention_smem_bytes(int hd) { return hd == 64 ? AttCfg<64>::SMEM : AttCfg<128>::SMEM; }

cudaError_t attention_prepare() {
  cudaError_t e = cudaFuncSetAttribute(attention_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)AttCfg<64>::SMEM);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(attention_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)AttCfg<128>::SMEM);
}

cudaError_t launch_attention(const AttnParams& p, int num_sms, cudaStream_t st, bool pdl) {
  // One wave of two CTAs per SM.  A pair of nu units is shared by at most
  // (nu-1)P/U + 2 <= P/H + 2 CTAs, so P <= 14 H keeps that within ATT_SEG_MAX.
  const long long units_max = (long long)p.nb * p.H * ((p.cap + ATT_UNIT - 1) / ATT_UNIT);
  const int grid = (int)std::min<long long>(std::min(2 * num_sms, (ATT_SEG_MAX - 2) * p.H), units_max);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = attention_smem_bytes(p.hd);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  if (p.hd == 64) return cudaLaunchKernelEx(&cfg, attention_kernel<64>, p);
  return cudaLaunchKernelEx(&cfg, attention_kernel<128>, p);
}

}  // namespace sdsat

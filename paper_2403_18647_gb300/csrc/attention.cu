// Block-causal split-KV attention of the q block rows against the KV cache.
//
// In one block forward, row j of sequence s attends to the committed slots
// [0, len[s]) and to block rows 0..j (slots len[s] .. len[s]+j), which the QKV
// epilogue has just written; this is how Eq. 1-2 evaluate every appended
// position of the block in one pass.  The bytes are the K and V rows (bf16,
// hd*2 bytes each), read once per (sequence, head) for all q rows together.
//
// Grid (chunk, head, sequence): each CTA owns ATT_CHUNK = 128 consecutive
// slots.  One thread issues TMA loads of the chunk's K and V tiles (boxes of
// 64 dims x 128 rows, 128-byte swizzle) as soon as the previous kernel has
// finished; K and V land on separate mbarriers so the scores are computed
// while V is still in flight.  Both products run on the tensor cores
// (mma.sync m16n8k16, the q <= 16 rows fill the M = 16 tile): S = Q K^T with
// each warp on 32 keys, then O = P V with each warp on hd/4 dimensions.  Q
// and P enter as bf16 hi + lo pairs (two MMAs each), K and V are the cache's
// own bf16 values, accumulation is fp32.  Each CTA
// writes its chunk's max score, exp-sum and unnormalised output per row; the
// last CTA of a (sequence, head) (per-pair counter, no waiting) merges the
// chunks in chunk order with the usual log-sum-exp rescaling --
// deterministic -- and writes the output in fp32 and as the O projection's
// bf16 hi + lo operand.
#include "common.cuh"
#include "internal.h"

namespace sdsat {

template <int HD>
struct AttCfg {
  static constexpr int HALVES = HD / 64;                 // 64-dim column boxes per row
  static constexpr int TILE = ATT_CHUNK * 128 * HALVES;  // bytes of one K (or V) chunk
  static constexpr int QSTRIDE = HD * 2 + 16;            // bytes per row of the bf16 Q / P tiles (padded)
  static constexpr int PSTRIDE = ATT_CHUNK * 2 + 16;
  static constexpr size_t SMEM = 1024 + 2 * (size_t)TILE + 2 * 16 * QSTRIDE + 2 * 16 * PSTRIDE +
                                 2 * 4 * 16 * 4 + 2 * 16 * 4 + 64;
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

template <int HD>
__global__ void __launch_bounds__(128) attention_kernel(const __grid_constant__ AttnParams p) {
  using C = AttCfg<HD>;
  constexpr int CH = ATT_CHUNK;
  constexpr int KSTEPS = HD / 16;          // MMA k-steps over the head dimension
  constexpr int DT = HD / 32;              // 8-wide dimension tiles per warp in P.V
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* Ktile = smem;
  uint8_t* Vtile = smem + C::TILE;
  uint8_t* Qh = smem + 2 * C::TILE;                 // bf16 [16][HD] (scaled q, hi part), padded rows
  uint8_t* Ql = Qh + 16 * C::QSTRIDE;               // lo part
  uint8_t* Ph = Ql + 16 * C::QSTRIDE;               // bf16 [16][CH] softmax numerators, hi part
  uint8_t* Pl = Ph + 16 * C::PSTRIDE;
  float* red_m = reinterpret_cast<float*>(Pl + 16 * C::PSTRIDE);   // [4 warps][16 rows]
  float* red_l = red_m + 64;
  float* Ms = red_l + 64;                           // [16] chunk max per row
  float* Ls = Ms + 16;                              // [16] chunk exp-sum per row
  uint64_t* bar = reinterpret_cast<uint64_t*>(Ls + 16);   // [0] K landed, [1] V landed
  int* s_last = reinterpret_cast<int*>(bar + 2);

  const int ch = blockIdx.x, h = blockIdx.y, sl = blockIdx.z, s = p.seq0 + sl;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, tig = lane & 3;
  const int q = p.q;
  const unsigned long long t_entry = p.trace.rec ? globaltimer_ns() : 0;
  pdl_trigger();
  // The committed length is final before this kernel can start: the block forward's
  // first kernel (RMSNorm) lets its dependents launch only after every earlier kernel
  // has completed.  Slots below it are not written during this forward either, so a
  // chunk that lies entirely below it can be loaded before the QKV projection finishes.
  const int len = __ldcg(p.len + s);
  const int nkeys = min(len + q, p.cap);
  const int c0 = ch * CH;
  if (c0 >= nkeys) return;
  const int nch = (nkeys + CH - 1) / CH;
  const int row0 = p.row0 + (s * p.H + h) * p.cap + c0;   // first cache row of the chunk
  const bool early = c0 + CH <= len;                        // chunk holds committed slots only
  uint64_t pol = 0;
  auto issue_loads = [&]() {
    mbar_arrive_expect_tx(&bar[0], C::TILE);
#pragma unroll
    for (int hh = 0; hh < C::HALVES; ++hh) tma_load_2d(Ktile + hh * CH * 128, &p.kmap, &bar[0], hh * 64, row0, pol);
    mbar_arrive_expect_tx(&bar[1], C::TILE);
#pragma unroll
    for (int hh = 0; hh < C::HALVES; ++hh) tma_load_2d(Vtile + hh * CH * 128, &p.vmap, &bar[1], hh * 64, row0, pol);
  };
  if (tid == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    fence_mbar_init();
    pol = l2_policy_evict_first();
    if (early) issue_loads();
  }
  pdl_wait();   // q and this forward's new K/V rows come from the QKV projection
  const unsigned long long t_wait = p.trace.rec ? globaltimer_ns() : 0;
  if (tid == 0 && !early) issue_loads();
  // q (scaled by 1/sqrt(hd)) as bf16 hi + lo; rows >= q are zero
  const float scale = rsqrtf((float)HD);
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
  __syncthreads();   // Q tiles and the barrier initialisation are visible to all threads

  volatile int no_abort = 0;
  bool ok = mbar_wait_bounded(&bar[0], 0, &no_abort, p.err);
  __syncwarp();   // lanes leave the polling loop at different times: reconverge
  const unsigned long long t_k = p.trace.rec ? globaltimer_ns() : 0;

  // ---- S = Q K^T for this warp's 32 keys (4 tiles of 8), fp32 in registers
  const int kb = warp * 32;                       // first key (within the chunk) of this warp
  float S[4][4];
#pragma unroll
  for (int nt = 0; nt < 4; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) S[nt][e] = 0.f;
  const int mi = lane >> 3, r8 = lane & 7;        // ldmatrix: this thread's matrix and row
  if (ok) {
#pragma unroll
    for (int kk = 0; kk < KSTEPS; ++kk) {
      uint32_t ah[4], al[4];
      const int qrow = r8 + 8 * (mi & 1), qcol = kk * 16 + 8 * (mi >> 1);
      ldsm_x4(smem_u32(Qh + qrow * C::QSTRIDE + qcol * 2), ah[0], ah[1], ah[2], ah[3]);
      ldsm_x4(smem_u32(Ql + qrow * C::QSTRIDE + qcol * 2), al[0], al[1], al[2], al[3]);
      const int hh = kk >> 2, cg = 2 * (kk & 3);  // 64-dim half and first 16-byte granule
#pragma unroll
      for (int np = 0; np < 2; ++np) {            // two key tiles per ldmatrix.x4
        const int key = kb + 8 * (2 * np + (mi >> 1)) + r8;
        const int c = cg + (mi & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(smem_u32(Ktile + hh * CH * 128 + key * 128 + ((c ^ (key & 7)) << 4)), b0, b1, b2, b3);
        mma_bf16_16816(S[2 * np], ah[0], ah[1], ah[2], ah[3], b0, b1);
        mma_bf16_16816(S[2 * np], al[0], al[1], al[2], al[3], b0, b1);
        mma_bf16_16816(S[2 * np + 1], ah[0], ah[1], ah[2], ah[3], b2, b3);
        mma_bf16_16816(S[2 * np + 1], al[0], al[1], al[2], al[3], b2, b3);
      }
    }
  }
  // mask: row j sees chunk key k iff c0 + k <= len + j (and c0 + k < nkeys, j < q)
#pragma unroll
  for (int nt = 0; nt < 4; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int j = g + 8 * (e >> 1);
      const int kp = c0 + kb + 8 * nt + 2 * tig + (e & 1);
      if (!ok || j >= q || kp >= nkeys || kp > len + j) S[nt][e] = -INFINITY;
    }
  // ---- row max and exp-sum over the chunk's 128 keys (4 threads x 4 warps share a row)
  float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
  for (int nt = 0; nt < 4; ++nt) {
    mx0 = fmaxf(mx0, fmaxf(S[nt][0], S[nt][1]));
    mx1 = fmaxf(mx1, fmaxf(S[nt][2], S[nt][3]));
  }
#pragma unroll
  for (int o = 1; o < 4; o <<= 1) {
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
  }
  if (tig == 0) {
    red_m[warp * 16 + g] = mx0;
    red_m[warp * 16 + g + 8] = mx1;
  }
  __syncthreads();
  mx0 = fmaxf(fmaxf(red_m[g], red_m[16 + g]), fmaxf(red_m[32 + g], red_m[48 + g]));
  mx1 = fmaxf(fmaxf(red_m[8 + g], red_m[24 + g]), fmaxf(red_m[40 + g], red_m[56 + g]));
  float l0 = 0.f, l1 = 0.f;
#pragma unroll
  for (int nt = 0; nt < 4; ++nt) {
    float pv[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float m = (e < 2) ? mx0 : mx1;
      pv[e] = (S[nt][e] == -INFINITY) ? 0.f : expf(S[nt][e] - m);
    }
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
#pragma unroll
  for (int o = 1; o < 4; o <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, o);
    l1 += __shfl_xor_sync(0xffffffffu, l1, o);
  }
  if (tig == 0) {
    red_l[warp * 16 + g] = l0;
    red_l[warp * 16 + g + 8] = l1;
  }
  __syncthreads();   // P tiles and the partial sums are complete
  if (tid < 16) {
    Ms[tid] = fmaxf(fmaxf(red_m[tid], red_m[16 + tid]), fmaxf(red_m[32 + tid], red_m[48 + tid]));
    Ls[tid] = red_l[tid] + red_l[16 + tid] + red_l[32 + tid] + red_l[48 + tid];
  }

  // ---- O = P V for this warp's HD/4 dimensions (DT tiles of 8), all 128 keys
  ok = ok && mbar_wait_bounded(&bar[1], 0, &no_abort, p.err);
  __syncwarp();
  float O[DT][4];
#pragma unroll
  for (int nt = 0; nt < DT; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) O[nt][e] = 0.f;
  const int db = warp * (HD / 4);                 // first dimension of this warp
  if (ok) {
#pragma unroll
    for (int kk = 0; kk < CH / 16; ++kk) {
      uint32_t ah[4], al[4];
      const int prow = r8 + 8 * (mi & 1), pcol = kk * 16 + 8 * (mi >> 1);
      ldsm_x4(smem_u32(Ph + prow * C::PSTRIDE + pcol * 2), ah[0], ah[1], ah[2], ah[3]);
      ldsm_x4(smem_u32(Pl + prow * C::PSTRIDE + pcol * 2), al[0], al[1], al[2], al[3]);
#pragma unroll
      for (int np = 0; np < DT / 2; ++np) {       // two dimension tiles per ldmatrix.x4.trans
        const int key = kk * 16 + 8 * (mi & 1) + r8;
        const int dim = db + 8 * (2 * np + (mi >> 1));
        const int hh = dim >> 6, c = (dim & 63) >> 3;
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(smem_u32(Vtile + hh * CH * 128 + key * 128 + ((c ^ (key & 7)) << 4)), b0, b1, b2, b3);
        mma_bf16_16816(O[2 * np], ah[0], ah[1], ah[2], ah[3], b0, b1);
        mma_bf16_16816(O[2 * np], al[0], al[1], al[2], al[3], b0, b1);
        mma_bf16_16816(O[2 * np + 1], ah[0], ah[1], ah[2], ah[3], b2, b3);
        mma_bf16_16816(O[2 * np + 1], al[0], al[1], al[2], al[3], b2, b3);
      }
    }
  }
  const size_t prow_base = (size_t)h * p.nch_max + ch;
  if (tid < q) {   // Ms / Ls of row tid were written by this thread; read before the stores below
    float* ml = p.part_ml + ((size_t)(sl * q + tid) * p.H * p.nch_max + prow_base) * 2;
    ml[0] = Ms[tid];
    ml[1] = Ls[tid];
  }
#pragma unroll
  for (int nt = 0; nt < DT; ++nt)
#pragma unroll
    for (int e = 0; e < 4; e += 2) {
      const int j = g + 8 * (e >> 1);
      if (j < q) {
        const int dim = db + 8 * nt + 2 * tig;
        *reinterpret_cast<float2*>(p.part_o + ((size_t)(sl * q + j) * p.H * p.nch_max + prow_base) * HD + dim) =
            make_float2(O[nt][e], O[nt][e + 1]);
      }
    }

  // the last chunk CTA of this (sequence, head) merges the chunks: the CTA's stores, then
  // one release/acquire counter update by thread 0
  const unsigned long long t_part = p.trace.rec ? globaltimer_ns() : 0;
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    *s_last = (atomicAdd(p.counters + sl * p.H + h, 1) == nch - 1);
    __threadfence();
  }
  __syncthreads();
  if (!*s_last) {
    if (tid == 0 && p.trace.rec)
      trace_write(p.trace, (unsigned)nch << 8, t_entry, t_wait, t_k, t_part, 0, globaltimer_ns());
    return;
  }
  // Merge weights: warp w takes rows j = w, w + 4, ...; its lanes hold the chunks.
  // w[j][c] = exp(m_c - max_c m_c) goes to shared memory (the K tile is free now),
  // 1 / L_j with L_j = sum_c w[j][c] l_c to Ms[j].
  float* wgt = reinterpret_cast<float*>(Ktile);   // [q][nch]; q * nch <= 16 * ATT_MAX_CHUNKS floats
  constexpr int CPL = ATT_MAX_CHUNKS / 32;        // chunks per lane
  for (int j = warp; j < q; j += 4) {
    const float* mlr = p.part_ml + ((size_t)(sl * q + j) * p.H * p.nch_max + (size_t)h * p.nch_max) * 2;
    float mc[CPL], lc[CPL];
#pragma unroll
    for (int u = 0; u < CPL; ++u) {
      const int c = lane + 32 * u;
      mc[u] = -INFINITY;
      lc[u] = 0.f;
      if (c < nch) {
        const float2 v = __ldcg(reinterpret_cast<const float2*>(mlr) + c);
        mc[u] = v.x;
        lc[u] = v.y;
      }
    }
    float mx = -INFINITY;
#pragma unroll
    for (int u = 0; u < CPL; ++u) mx = fmaxf(mx, mc[u]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float L = 0.f;
#pragma unroll
    for (int u = 0; u < CPL; ++u) {
      const int c = lane + 32 * u;
      const float wc = (mc[u] == -INFINITY) ? 0.f : expf(mc[u] - mx);
      if (c < nch) wgt[j * nch + c] = wc;
      L += wc * lc[u];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
    if (lane == 0) Ms[j] = 1.0f / L;
  }
  __syncthreads();
  const unsigned long long t_stats = p.trace.rec ? globaltimer_ns() : 0;
  // O_j = (sum_c w[j][c] o_c) / L_j: thread = (row group, 4 dimensions); every row of the
  // group advances four chunks at a time, so up to 16 float4 loads are in flight
  {
    constexpr int D4 = HD / 4;                 // float4 columns of a row
    constexpr int RG = 128 / D4;               // row groups
    constexpr int RPT = (16 + RG - 1) / RG;    // rows per thread (q <= 16)
    const int d4 = tid % D4, jg = tid / D4;
    float4 acc[RPT];
#pragma unroll
    for (int k = 0; k < RPT; ++k) acc[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int c0 = 0; c0 < nch; c0 += 4) {
      float4 v[RPT][4];
#pragma unroll
      for (int k = 0; k < RPT; ++k) {
        const int j = jg + RG * k;
        const float4* po = reinterpret_cast<const float4*>(
                               p.part_o + ((size_t)(sl * q + j) * p.H * p.nch_max + (size_t)h * p.nch_max) * HD) + d4;
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (j < q && c0 + u < nch) v[k][u] = __ldcg(po + (size_t)(c0 + u) * D4);
      }
#pragma unroll
      for (int k = 0; k < RPT; ++k) {
        const int j = jg + RG * k;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          if (j < q && c0 + u < nch) {
            const float wc = wgt[j * nch + c0 + u];
            acc[k].x += wc * v[k][u].x;
            acc[k].y += wc * v[k][u].y;
            acc[k].z += wc * v[k][u].z;
            acc[k].w += wc * v[k][u].w;
          }
        }
      }
    }
#pragma unroll
    for (int k = 0; k < RPT; ++k) {
      const int j = jg + RG * k;
      if (j < q) {
        const float inv = Ms[j];
        const float4 o = make_float4(acc[k].x * inv, acc[k].y * inv, acc[k].z * inv, acc[k].w * inv);
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
    }
  }
  if (tid == 0) {
    p.counters[sl * p.H + h] = 0;
    if (p.trace.rec)
      trace_write(p.trace, 1u | ((unsigned)nch << 8), t_entry, t_wait, t_k, t_part, t_stats, globaltimer_ns());
  }
}

size_t attention_smem_bytes(int hd) { return hd == 64 ? AttCfg<64>::SMEM : AttCfg<128>::SMEM; }

cudaError_t attention_prepare() {
  cudaError_t e = cudaFuncSetAttribute(attention_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)AttCfg<64>::SMEM);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(attention_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)AttCfg<128>::SMEM);
}

cudaError_t launch_attention(const AttnParams& p, cudaStream_t st, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.nch_max, p.H, p.nb);
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

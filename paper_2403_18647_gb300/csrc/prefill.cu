// Prefill: the prompt's positions through the model in chunks of up to PF_ROWS, before the
// decode loop.  Unlike the decode step (a handful of rows, bound by the weight stream), a
// chunk of hundreds of positions makes every projection a dense contraction, so it runs
// on a tiled tensor-core GEMM:
//
//   Y[m][n] = sum_k X[m][k] W[n][k], one CTA tile = 128 weight rows x 128 positions.
//
// The weight tile is the MMA's A operand (M = 128), the positions its B operand: the
// bf16 hi and lo parts of X stacked into one N = 256 operand, so one tcgen05.mma per
// 16-wide k-step computes W*Xhi and W*Xlo side by side in TMEM and the epilogue adds the
// two halves (fp32-like activations, exact bf16 weights, fp32 accumulation -- the decode
// path's precision).  One persistent CTA per SM (four 48 KB TMA stages, two 256-column
// TMEM accumulators so a tile's epilogue overlaps the next tile's MMAs); warp 0 streams
// TMA, warp 1 issues the MMAs, warps 2-5 drain TMEM.  Tiles are numbered weight-tile
// major, so the CTAs working at the same time share weight tiles through L2.
//
// Epilogues: store (q, k, v before RoPE), residual add (O and down projections), and
// SiLU(gate) * up written as the down projection's bf16 hi + lo operand.  RMSNorm and
// RoPE + the KV append are small row kernels here (the decode path folds them into the
// GEMMs); attention is the causal flash-attention kernel at the end of attention.cu.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace sdsat {

constexpr int PF_STAGES = 4;
constexpr int PF_TOK = 128;                              // positions per tile
constexpr int PF_W_BYTES = 128 * 128;                    // 128 weight rows x 64 bf16
constexpr int PF_X_BYTES = PF_TOK * 128;                 // 128 positions x 64 bf16 (hi or lo)
constexpr int PF_STAGE = PF_W_BYTES + 2 * PF_X_BYTES;    // 48 KB
constexpr int PF_ACC = 2 * PF_TOK;                       // TMEM columns of one accumulator (hi, lo)
constexpr int PF_CHUNK = 32;                             // positions per epilogue round
constexpr int PF_STAGING = 64 * (PF_CHUNK + 1);          // [64 up rows][32 positions] exchange (fp32)
constexpr int PF_NBAR = 2 * PF_STAGES + 5;
constexpr size_t PF_SMEM = 1024 + (size_t)PF_STAGES * PF_STAGE + PF_STAGING * 4 + PF_NBAR * 8 + 64;

__device__ __forceinline__ void pf_tile_half_src(int map_mode, int rows_per_map, int t, int h, int& map, int& row) {
  if (map_mode == MAP_GATEUP) {
    map = h;
    row = 64 * t;
  } else if (map_mode == MAP_QKV3) {
    const int g = 128 * t;
    map = g / rows_per_map;
    row = g % rows_per_map + 64 * h;
  } else {
    map = 0;
    row = 128 * t + 64 * h;
  }
}

__global__ void __launch_bounds__(192, 1) prefill_gemm_kernel(const __grid_constant__ PfGemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* stages = smem;
  float* staging = reinterpret_cast<float*>(smem + (size_t)PF_STAGES * PF_STAGE);
  uint64_t* bars = reinterpret_cast<uint64_t*>(staging + PF_STAGING);
  uint64_t* full = bars;                  // the stage's weights and positions landed (TMA)
  uint64_t* empty = bars + PF_STAGES;     // the stage was consumed by the tensor core
  uint64_t* acc_full = bars + 2 * PF_STAGES;   // [2] accumulator ready
  uint64_t* acc_empty = acc_full + 2;          // [2] accumulator drained (4 epilogue warps)
  uint64_t* drain = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int T = p.n_wtiles * p.n_tblocks;
  const int P = gridDim.x;
  if (threadIdx.x == 0) {
    for (int s = 0; s < PF_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, 2 * PF_ACC);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();

  if (warp == 0) {
    // ------------------------------------------------ weight + position stream (TMA)
    if (lane == 0) {
      const int nmaps = p.map_mode == MAP_QKV3 ? 3 : (p.map_mode == MAP_GATEUP ? 2 : 1);
      for (int i = 0; i < nmaps; ++i) tma_prefetch_desc(&p.tmap[i]);
      tma_prefetch_desc(&p.tmap_x[0]);
      tma_prefetch_desc(&p.tmap_x[1]);
      const uint64_t pol_w = l2_policy_evict_normal();  // a weight tile is read by the CTAs of every position block
      const uint64_t pol_x = l2_policy_evict_last();    // a position block is read by every weight tile
      pdl_wait();   // the positions are the previous kernel's output
      int it = 0;
      for (int t = blockIdx.x; t < T && !*abort_flag; t += P) {
        const int wt = t / p.n_tblocks, tb = t % p.n_tblocks;
        for (int kc = 0; kc < p.kc; ++kc, ++it) {
          const int s = it % PF_STAGES;
          if (!mbar_wait_bounded(&empty[s], ((it / PF_STAGES) & 1) ^ 1, abort_flag, p.err)) break;
          mbar_arrive_expect_tx(&full[s], PF_STAGE);
          uint8_t* dst = stages + (size_t)s * PF_STAGE;
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            int map, row;
            pf_tile_half_src(p.map_mode, p.rows_per_map, wt, h, map, row);
            tma_load_2d(dst + h * 8192, &p.tmap[map], &full[s], kc * 64, row, pol_w);
          }
          tma_load_2d(dst + PF_W_BYTES, &p.tmap_x[0], &full[s], kc * 64, tb * PF_TOK, pol_x);
          tma_load_2d(dst + PF_W_BYTES + PF_X_BYTES, &p.tmap_x[1], &full[s], kc * 64, tb * PF_TOK, pol_x);
        }
      }
      if (*abort_flag) {   // let every copy in flight land before the CTA exits
        for (int i = std::max(0, it - PF_STAGES); i < it; ++i) {
          const uint64_t t0 = globaltimer_ns();
          while (!mbar_try_wait(&full[i % PF_STAGES], (i / PF_STAGES) & 1))
            if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) break;
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ tensor-core issue
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(128, PF_ACC);
      int it = 0, seg = 0;
      bool ok = true;
      for (int t = blockIdx.x; ok && t < T; t += P, ++seg) {
        const int buf = seg & 1;
        if (!mbar_wait_bounded(&acc_empty[buf], ((seg >> 1) & 1) ^ 1, abort_flag, p.err)) break;
        tc_fence_after();
        const uint32_t d = tmem + buf * PF_ACC;
        for (int kc = 0; kc < p.kc; ++kc, ++it) {
          const int s = it % PF_STAGES;
          if (!mbar_wait_bounded(&full[s], (it / PF_STAGES) & 1, abort_flag, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t wa = smem_u32(stages + (size_t)s * PF_STAGE);
          const uint32_t xb = wa + PF_W_BYTES;   // [Xhi; Xlo]: 256 rows of 128 B
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            umma_bf16(d, sdesc_sw128(wa + kk * 32), sdesc_sw128(xb + kk * 32), idesc, (kc > 0 || kk > 0) ? 1u : 0u);
          umma_commit(&empty[s]);
        }
        if (!ok) break;
        umma_commit(&acc_full[buf]);
      }
      if (*abort_flag) {   // wait for issued MMAs before shared memory goes away
        umma_commit(drain);
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(drain, 0))
          if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) break;
      }
    }
  } else {
    // ------------------------------------------------ epilogue (TMEM -> registers -> global)
    const int e = warp & 3;   // TMEM lane quarter this warp may access
    const int r = e * 32 + lane;
    pdl_wait();   // residual rows and outputs belong to the previous kernels' results
    int seg = 0;
    for (int t = blockIdx.x; t < T; t += P, ++seg) {
      const int wt = t / p.n_tblocks, tb = t % p.n_tblocks;
      const int buf = seg & 1;
      const bool got = named_bar_and(1, 128, mbar_wait_bounded(&acc_full[buf], (seg >> 1) & 1, abort_flag, p.err));
      if (!got) break;
      tc_fence_after();
      const uint32_t lane_addr = tmem + ((uint32_t)(e * 32) << 16) + buf * PF_ACC;
      for (int c0 = 0; c0 < PF_TOK; c0 += PF_CHUNK) {
        const int m0 = tb * PF_TOK + c0;
        if (m0 >= p.M) break;   // (uniform over the CTA)
        float y[PF_CHUNK], ya[16], yb[16], la[16], lb[16];
        tmem_ld16(lane_addr + c0, ya);
        tmem_ld16(lane_addr + c0 + 16, yb);
        tmem_ld16(lane_addr + PF_TOK + c0, la);
        tmem_ld16(lane_addr + PF_TOK + c0 + 16, lb);
        tmem_wait_ld();
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          y[j] = ya[j] + la[j];
          y[16 + j] = yb[j] + lb[j];
        }
        if (c0 + PF_CHUNK >= PF_TOK || m0 + PF_CHUNK >= p.M) {   // the accumulator is drained
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[buf]);
        }
        if (p.epi == EPI_SWIGLU) {
          // tile rows 0-63: gate features 64*wt + r, rows 64-127: the matching up features
          if (r >= 64)
#pragma unroll
            for (int j = 0; j < PF_CHUNK; ++j) staging[(r - 64) * (PF_CHUNK + 1) + j] = y[j];
          named_bar_sync(1, 128);
          const int f = 64 * wt + r;
          if (r < 64 && f < p.N) {
#pragma unroll
            for (int j = 0; j < PF_CHUNK; ++j) {
              const int m = m0 + j;
              if (m < p.M) {
                const float g = y[j];
                const float a = g / (1.0f + expf(-g)) * staging[r * (PF_CHUNK + 1) + j];
                const __nv_bfloat16 hi = __float2bfloat16_rn(a);
                p.out_hi[(size_t)m * p.out_ld + f] = hi;
                p.out_lo[(size_t)m * p.out_ld + f] = __float2bfloat16_rn(a - __bfloat162float(hi));
              }
            }
          }
          named_bar_sync(1, 128);
        } else {
          const int n = 128 * wt + r;
          if (n < p.N) {
            if (p.epi == EPI_RESID) {
              float hv[PF_CHUNK];
#pragma unroll
              for (int j = 0; j < PF_CHUNK; ++j)
                hv[j] = (m0 + j < p.M) ? __ldcg(p.out + (size_t)(m0 + j) * p.out_ld + n) : 0.f;
#pragma unroll
              for (int j = 0; j < PF_CHUNK; ++j) y[j] += hv[j];
            }
#pragma unroll
            for (int j = 0; j < PF_CHUNK; ++j)
              if (m0 + j < p.M) p.out[(size_t)(m0 + j) * p.out_ld + n] = y[j];
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * PF_ACC);
  }
}

cudaError_t prefill_prepare() {
  return cudaFuncSetAttribute(prefill_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)PF_SMEM);
}

cudaError_t launch_prefill_gemm(PfGemmParams& p, int num_sms, cudaStream_t st, bool pdl) {
  const int T = p.n_wtiles * p.n_tblocks;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(std::max(1, std::min(num_sms, T)));
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = PF_SMEM;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, prefill_gemm_kernel, p);
}

// ---- RoPE + KV append of a prefill chunk ------------------------------------------------
// qkv [M][3R] (q | k | v, head-major columns) -> q rotated into qout [M][R]; k rotated and v
// into the cache slots len[seq] + m at position len[seq] + m (rotate-half pairing (i, i + hd/2)).
__global__ void __launch_bounds__(256) rope_kv_kernel(RopeKvParams p) {
  pdl_wait();
  pdl_trigger();
  const int m = blockIdx.x;
  const int R = p.H * p.hd, half = p.hd >> 1;
  const int slot = __ldcg(p.len + p.seq) + m;
  int pos = slot;
  if (pos >= p.rope_len) {
    if (threadIdx.x == 0) set_error(p.err, ERR_POSITION);
    pos = p.rope_len - 1;
  }
  const bool fits = slot < p.cap;
  if (!fits && threadIdx.x == 0) set_error(p.err, ERR_CAPACITY);
  const float* row = p.qkv + (size_t)m * 3 * R;
  for (int idx = threadIdx.x; idx < R; idx += blockDim.x) {
    const int h = idx / p.hd, i = idx % p.hd;
    const int partner = i < half ? idx + half : idx - half;
    const float2 cs = p.rope[(size_t)pos * half + (i % half)];
    const float qa = row[idx], qp = row[partner];
    const float ka = row[R + idx], kp = row[R + partner];
    p.qout[(size_t)m * R + idx] = i < half ? qa * cs.x - qp * cs.y : qa * cs.x + qp * cs.y;
    if (fits) {
      const size_t o = (((size_t)p.seq * p.H + h) * p.cap + slot) * p.hd + i;
      p.k_layer[o] = __float2bfloat16_rn(i < half ? ka * cs.x - kp * cs.y : ka * cs.x + kp * cs.y);
      p.v_layer[o] = __float2bfloat16_rn(row[2 * R + idx]);
    }
  }
}

cudaError_t launch_rope_kv(const RopeKvParams& p, int M, cudaStream_t st, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(M);
  cfg.blockDim = dim3(256);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, rope_kv_kernel, p);
}

}  // namespace sdsat

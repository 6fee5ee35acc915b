// Block-causal split-KV attention of the q block rows against the KV cache.
//
// In one block forward, row j of sequence s attends to the committed slots
// [0, len[s]) and to block rows 0..j (slots len[s] .. len[s]+j), which the QKV
// epilogue has just written; this is how Eq. 1-2 evaluate every appended
// position of the block in one pass.  The bytes are the K and V rows (bf16,
// hd*2 bytes each), read once per (sequence, head) for all q rows together.
//
// Grid (chunk, head, sequence): each CTA owns ATT_CHUNK = 128 consecutive
// slots, computes for every block row the chunk's max score, exp-sum and
// unnormalised output, and writes them to a workspace; the last CTA of a
// (sequence, head) (per-pair counter, no waiting) merges the chunks in chunk
// order with the usual log-sum-exp rescaling -- deterministic.
#include "common.cuh"
#include "internal.h"

namespace sdsat {

template <int HD>
__global__ void __launch_bounds__(128) attention_kernel(const AttnParams p) {
  constexpr int CH = ATT_CHUNK;
  __shared__ __align__(16) float Qs[SDSAT_ATT_MAXQ][HD];
  __shared__ float Ps[SDSAT_ATT_MAXQ][CH];
  __shared__ float Ms[SDSAT_ATT_MAXQ], Ls[SDSAT_ATT_MAXQ];
  __shared__ int s_last;

  pdl_wait();
  pdl_trigger();
  const int ch = blockIdx.x, h = blockIdx.y, sl = blockIdx.z, s = p.seq0 + sl;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int q = p.q;
  const int len = __ldcg(p.len + s);
  const int nkeys = min(len + q, p.cap);
  const int c0 = ch * CH;
  if (c0 >= nkeys) return;
  const int nch = (nkeys + CH - 1) / CH;
  const float scale = rsqrtf((float)HD);

  for (int i = tid; i < q * HD; i += 128) {
    const int j = i / HD, d = i % HD;
    Qs[j][d] = __ldcg(p.Q + (size_t)(sl * q + j) * p.q_ld + h * HD + d) * scale;
  }
  __syncthreads();

  // scores: thread t <-> slot c0 + t
  const size_t head_base = ((size_t)s * p.H + h) * p.cap;
  {
    const int kp = c0 + tid;
    float sc[SDSAT_ATT_MAXQ];
#pragma unroll
    for (int j = 0; j < SDSAT_ATT_MAXQ; ++j) sc[j] = 0.f;
    if (kp < nkeys) {
      const uint4* kr = reinterpret_cast<const uint4*>(p.k + (head_base + kp) * HD);
#pragma unroll 4
      for (int gi = 0; gi < HD / 8; ++gi) {
        const uint4 raw = __ldcg(kr + gi);
        const __nv_bfloat162* k2 = reinterpret_cast<const __nv_bfloat162*>(&raw);
        float kf[8];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __bfloat1622float2(k2[e]);
          kf[2 * e] = f.x;
          kf[2 * e + 1] = f.y;
        }
#pragma unroll
        for (int j = 0; j < SDSAT_ATT_MAXQ; ++j) {
          if (j < q) {
            const float4 a = *reinterpret_cast<const float4*>(&Qs[j][gi * 8]);
            const float4 b = *reinterpret_cast<const float4*>(&Qs[j][gi * 8 + 4]);
            sc[j] += a.x * kf[0] + a.y * kf[1] + a.z * kf[2] + a.w * kf[3] + b.x * kf[4] + b.y * kf[5] +
                     b.z * kf[6] + b.w * kf[7];
          }
        }
      }
    }
#pragma unroll
    for (int j = 0; j < SDSAT_ATT_MAXQ; ++j)
      if (j < q) Ps[j][tid] = (kp < nkeys && kp <= len + j) ? sc[j] : -INFINITY;
  }
  __syncthreads();

  // per-row max and exp-sum over the chunk: warp w takes rows w, w+4, ...
  for (int j = warp; j < q; j += 4) {
    float m = -INFINITY;
    for (int t = lane; t < CH; t += 32) m = fmaxf(m, Ps[j][t]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    float l = 0.f;
    for (int t = lane; t < CH; t += 32) {
      const float e = (m == -INFINITY) ? 0.f : expf(Ps[j][t] - m);
      Ps[j][t] = e;
      l += e;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
    if (lane == 0) {
      Ms[j] = m;
      Ls[j] = l;
    }
  }
  __syncthreads();

  // unnormalised output of the chunk: thread d <-> dimension d
  const int nk = min(CH, nkeys - c0);
  const size_t prow = (size_t)h * p.nch_max + ch;
  if (tid < HD) {
    float o[SDSAT_ATT_MAXQ];
#pragma unroll
    for (int j = 0; j < SDSAT_ATT_MAXQ; ++j) o[j] = 0.f;
    const __nv_bfloat16* vcol = p.v + head_base * HD + (size_t)c0 * HD + tid;
    for (int t = 0; t < nk; ++t) {
      const float v = __bfloat162float(vcol[(size_t)t * HD]);
#pragma unroll
      for (int j = 0; j < SDSAT_ATT_MAXQ; ++j)
        if (j < q) o[j] += Ps[j][t] * v;
    }
#pragma unroll
    for (int j = 0; j < SDSAT_ATT_MAXQ; ++j)
      if (j < q) p.part_o[((size_t)(sl * q + j) * p.H * p.nch_max + prow) * HD + tid] = o[j];
  }
  if (tid < q) {
    float* ml = p.part_ml + ((size_t)(sl * q + tid) * p.H * p.nch_max + prow) * 2;
    ml[0] = Ms[tid];
    ml[1] = Ls[tid];
  }

  // the last chunk CTA of this (sequence, head) merges the chunks
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = (atomicAdd(p.counters + sl * p.H + h, 1) == nch - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (tid < HD) {
    for (int j = 0; j < q; ++j) {
      const size_t rb = (size_t)(sl * q + j) * p.H * p.nch_max + (size_t)h * p.nch_max;
      float mx = -INFINITY;
      for (int c = 0; c < nch; ++c) mx = fmaxf(mx, __ldcg(p.part_ml + (rb + c) * 2));
      float L = 0.f, O = 0.f;
      for (int c = 0; c < nch; ++c) {
        const float mc = __ldcg(p.part_ml + (rb + c) * 2);
        const float w = (mc == -INFINITY) ? 0.f : expf(mc - mx);
        L += w * __ldcg(p.part_ml + (rb + c) * 2 + 1);
        O += w * __ldcg(p.part_o + (rb + c) * HD + tid);
      }
      p.out[(size_t)(sl * q + j) * p.out_ld + h * HD + tid] = O / L;
    }
  }
  if (tid == 0) p.counters[sl * p.H + h] = 0;
}

cudaError_t launch_attention(const AttnParams& p, cudaStream_t st, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.nch_max, p.H, p.nb);
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = 0;
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

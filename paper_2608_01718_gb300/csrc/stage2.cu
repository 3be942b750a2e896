// Candidate merge, stage 2 (the lookahead check) and the decision, fused in one kernel.
//
// One CTA (8 warps) per query:
//  1. merge the stage-1 partial lists (per split a record of its best score and candidate count, and that many
//     packed candidates) into C_q, the top_c candidates by (key score desc, entry id asc): every thread keeps a
//     sorted top-c of the candidates it reads (four splits in flight), each warp reduces its lanes' lists by top_c
//     rounds of a warp-wide max, and warp 0 merges the eight warp lists the same way;
//  2. the candidates are checked in parallel, one warp per candidate: r = <p_q, P_j> (the prefix-embedding cosine
//     sim(f_k(x), f_k(x'))) in fp32, each lane's 8-element chunks in order, then a butterfly sum (every lane ends
//     with the same bits); m = number of positions i < k with equal token ids;
//  3. the served entry is the first candidate in C_q order that passes (Algorithm 1); status HIT / REJECT /
//     MISS_KEY.
#include "internal.cuh"

namespace lc {
namespace {

constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;
constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

// Warp-wide maximum of a packed candidate, as two 32-bit warp reductions: the largest high word (score order),
// then the largest low word (~id) among the lanes that hold it. Unsigned 64-bit order is (high, low)
// lexicographic, so this is the 64-bit maximum.
__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
  const uint32_t hi = (uint32_t)(v >> 32), lo = (uint32_t)v;
  const uint32_t mhi = __reduce_max_sync(kFull, hi);
  const uint32_t mlo = __reduce_max_sync(kFull, hi == mhi ? lo : 0u);
  return ((uint64_t)mhi << 32) | mlo;
}

__device__ __forceinline__ float dot8(const uint4& u, const uint4& v, float acc) {
  const __nv_bfloat162* a = reinterpret_cast<const __nv_bfloat162*>(&u);
  const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float2 x = __bfloat1622float2(a[e]);
    const float2 y = __bfloat1622float2(b[e]);
    acc = fmaf(x.x, y.x, acc);
    acc = fmaf(x.y, y.y, acc);
  }
  return acc;
}

template <int CPAD>
__device__ __forceinline__ void keep(uint64_t (&loc)[CPAD], uint64_t x) {
  if (x > loc[CPAD - 1]) {
#pragma unroll
    for (int i = 0; i < CPAD; ++i) {
      if (x > loc[i]) {
        const uint64_t t = loc[i];
        loc[i] = x;
        x = t;
      }
    }
  }
}

template <int CPAD>
__global__ void __launch_bounds__(kThreads) stage2_kernel(Stage2Args a) {
  __shared__ uint64_t warp_top[kWarps][CPAD];
  __shared__ uint64_t cand[CPAD];
  __shared__ float cand_rm[CPAD][kMaxModels];   // every model's r per candidate
  __shared__ int cand_emb_ok[CPAD];             // all models pass
  __shared__ int cand_m[CPAD];
  __shared__ float warp_best[kWarps];
  __shared__ int s_ncand;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q = blockIdx.x;
  const int C = a.top_c;

  // Launched as a programmatic dependent of stage 1: wait until every preceding grid on the stream has completed
  // and its writes are visible, before reading anything (a no-op when launched without the attribute).
  asm volatile("griddepcontrol.wait;" ::: "memory");
  // The next lookup's stage 1 may be scheduled now; it too waits for this grid before touching memory.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  // 1a + 1b. Every thread takes splits tid, tid + kThreads, ...: a split's record (best score, candidate count) and
  // the first two slots of its list are loaded together, before the count is known, so lists of at most two
  // candidates (the common case) take one memory round trip; longer ones load their other slots after it. Then the
  // maximum of the best scores, and every thread's sorted top-c of the candidates it read.
  uint64_t loc[CPAD];
#pragma unroll
  for (int i = 0; i < CPAD; ++i) loc[i] = 0;
  constexpr int U = 4;   // splits in flight per thread
  float best = -INFINITY;
  auto take = [&](uint64_t x) {
    if ((int64_t)cand_id(x) >= a.n) x = 0;   // never gather outside the store
    keep(loc, x);
  };
  for (int s0 = threadIdx.x; s0 < a.splits; s0 += U * kThreads) {
    PartMeta m[U];
    uint64_t x0[U], x1[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int sp = s0 + u * kThreads;
      m[u] = PartMeta{-INFINITY, 0u};
      x0[u] = x1[u] = 0;
      if (sp < a.splits) {
        const int64_t r = (int64_t)sp * a.B + q;
        m[u] = a.part_meta[r];
        x0[u] = a.part_cand[r * C];
        if (C > 1) x1[u] = a.part_cand[r * C + 1];
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      best = fmaxf(best, m[u].best);
      const int cnt = (int)m[u].count < C ? (int)m[u].count : C;
      if (cnt > 0) take(x0[u]);
      if (cnt > 1) take(x1[u]);
      for (int i = 2; i < cnt; ++i) take(a.part_cand[((int64_t)(s0 + u * kThreads) * a.B + q) * C + i]);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) best = fmaxf(best, __shfl_xor_sync(kFull, best, o));
  if (lane == 0) warp_best[warp] = best;
  // 1c. per-warp top-c (rounds stop at the first empty maximum: every later one is empty too)
  for (int r = 0; r < C; ++r) {
    const uint64_t m = warp_max_u64(loc[0]);
    if (lane == 0) warp_top[warp][r] = m;
    if (m == 0) {
      for (int i = r + 1 + lane; i < C; i += 32) warp_top[warp][i] = 0;
      break;
    }
    if (loc[0] == m) {
#pragma unroll
      for (int i = 0; i < CPAD - 1; ++i) loc[i] = loc[i + 1];
      loc[CPAD - 1] = 0;
    }
  }
  __syncthreads();
  // 1d. warp 0 merges the eight warp lists: lane l < kWarps walks list l
  if (warp == 0) {
    int head = 0;
    int n = 0;
    for (int r = 0; r < C; ++r) {
      const uint64_t h = (lane < kWarps && head < C) ? warp_top[lane][head] : 0;
      const uint64_t m = warp_max_u64(h);
      if (m == 0) break;
      if (h == m) ++head;
      if (lane == 0) cand[r] = m;
      ++n;
    }
    if (lane == 0) {
      s_ncand = n;
      float b = warp_best[0];
      for (int w = 1; w < kWarps; ++w) b = fmaxf(b, warp_best[w]);
      warp_best[0] = b;
    }
  }
  __syncthreads();
  const int n_cand = s_ncand;

  // 2. lookahead check of every candidate, one warp per candidate; one dot product per model segment
  const int pd = a.pd, k = a.k;
  const uint4* pq = reinterpret_cast<const uint4*>(a.q_prefix + (int64_t)q * pd);
  const int32_t* tq = a.q_ids + (int64_t)q * k;
  for (int i = warp; i < n_cand; i += kWarps) {
    const uint32_t j = cand_id(cand[i]);
    const uint4* pj = reinterpret_cast<const uint4*>(a.prefix + (int64_t)j * pd);
    const int32_t* tj = a.ids + (int64_t)j * k;
    // the first 32 token ids of both prefixes, loaded with the prefix rows below rather than after them
    const bool tl = lane < k;
    const int32_t tq0 = tl ? __ldg(tq + lane) : 0, tj0 = tl ? __ldg(tj + lane) : 0;
    int emb_ok = 1;
    for (int h = 0; h < a.m; ++h) {
      float acc = 0.f;
      for (int c8 = a.seg[h] / 8 + lane; c8 < a.seg[h + 1] / 8; c8 += 32)
        acc = dot8(__ldg(pq + c8), __ldg(pj + c8), acc);
      const float r = warp_sum(acc);
      emb_ok &= r >= a.tau_m[h] ? 1 : 0;
      if (lane == 0) cand_rm[i][h] = r;
    }
    int eq = tl && tq0 == tj0 ? 1 : 0;
    for (int t = lane + 32; t < k; t += 32) eq += (__ldg(tq + t) == __ldg(tj + t)) ? 1 : 0;
    const int m = __reduce_add_sync(kFull, eq);
    if (lane == 0) {
      cand_emb_ok[i] = emb_ok;
      cand_m[i] = m;
    }
  }
  __syncthreads();

  // candidate i passes the lookahead check under the check mode
  const int tmin = a.token_match_min > 0 ? a.token_match_min : k;
  auto passes = [&](int i) {
    const bool emb_ok = cand_emb_ok[i] != 0;
    const bool tok_ok = cand_m[i] >= tmin;
    return a.check_mode == LACACHE_CHECK_EMB ? emb_ok
           : a.check_mode == LACACHE_CHECK_TOKENS ? tok_ok
                                                  : (emb_ok && tok_ok);
  };

  // optional per-candidate outputs
  const float qnan = __int_as_float(0x7fc00000);
  for (int i = threadIdx.x; i < C; i += kThreads) {
    const int64_t o = (int64_t)q * C + i;
    const bool v = i < n_cand;
    if (a.out.cand_id) a.out.cand_id[o] = v ? (int32_t)cand_id(cand[i]) : -1;
    if (a.out.cand_score) a.out.cand_score[o] = v ? cand_score(cand[i]) : qnan;
    if (a.out.cand_prefix_score) a.out.cand_prefix_score[o] = v ? cand_rm[i][0] : qnan;
    if (a.out.cand_matches) a.out.cand_matches[o] = v ? cand_m[i] : -1;
    if (a.out.cand_pass) a.out.cand_pass[o] = v && passes(i) ? 1 : 0;
    if (a.out.cand_prefix_scores)
      for (int h = 0; h < a.m; ++h) a.out.cand_prefix_scores[o * a.m + h] = v ? cand_rm[i][h] : qnan;
  }

  // 3. decision: the first candidate, in C_q order, that passes
  if (threadIdx.x == 0) {
    int served = -1;
    for (int i = 0; i < n_cand && served < 0; ++i)
      if (passes(i)) served = i;
    const int shown = served >= 0 ? served : 0;   // the candidate whose scores are reported
    if (served >= 0) {
      a.out.status[q] = LACACHE_HIT;
      a.out.entry_id[q] = (int32_t)cand_id(cand[served]);
      a.out.key_score[q] = cand_score(cand[served]);
    } else {
      a.out.status[q] = n_cand ? LACACHE_REJECT : LACACHE_MISS_KEY;
      a.out.entry_id[q] = -1;
      a.out.key_score[q] = warp_best[0];
    }
    a.out.prefix_score[q] = n_cand ? cand_rm[shown][0] : qnan;
    a.out.token_matches[q] = n_cand ? cand_m[shown] : -1;
    if (a.out.prefix_scores)
      for (int h = 0; h < a.m; ++h) a.out.prefix_scores[(int64_t)q * a.m + h] = n_cand ? cand_rm[shown][h] : qnan;
    a.out.n_cand[q] = n_cand;
    if (a.counters) atomicAdd(a.counters + (served >= 0 ? 0 : n_cand ? 1 : 2), 1ull);
  }
}

}  // namespace

// Programmatic dependent launch: the grid may be scheduled while stage 1 is still running (its CTAs then sit in
// griddepcontrol.wait), which hides the launch gap between the two kernels.
template <int CPAD>
cudaError_t launch_cpad(const Stage2Args& a, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.B);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, stage2_kernel<CPAD>, a);
}

cudaError_t launch_stage2(const Stage2Args& a, cudaStream_t st) {
  cudaError_t e;
  if (a.top_c <= 4)
    e = launch_cpad<4>(a, st);
  else if (a.top_c <= 8)
    e = launch_cpad<8>(a, st);
  else if (a.top_c <= 16)
    e = launch_cpad<16>(a, st);
  else
    e = launch_cpad<32>(a, st);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace lc

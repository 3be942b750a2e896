// Merge of entry-range shards: the whole-store result of a lookup from the results of its shards.
//
// Shard g holds global entries [id_base_g, id_base_g + n_g) and has run the full lookup (both checks) on them.
// For each query:
//   C_q    = the first top_c of the union of the shards' candidate lists by (key score desc, global id asc).
//            Every member of the global list is among its own shard's first top_c, so this is the exact C_q.
//   j*     = the first member of C_q whose lookahead check passed on its shard (Algorithm 1); a pass bit
//            depends only on the candidate's row and the query.
//   status = HIT / REJECT (C_q not empty) / MISS_KEY; key score on a non-HIT = the maximum over the shards.
//
// One warp per query. The shards' candidates (at most 16 x 32) are loaded as packed (score order, ~global id)
// keys into shared memory; top_c rounds of a warp-wide maximum take them in order (each key is unique, and its
// owner lane clears it). Lane i then fills output slot i of the candidate list, and a ballot finds j*.
#include "internal.cuh"

namespace lc {
namespace {

constexpr int kWarps = 4;
constexpr unsigned kFull = 0xffffffffu;

struct MergeArgs {
  int G, B, C, m;
  lacache_shard_result s[LACACHE_MAX_SHARDS];
  lacache_result out;
};

__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
  const uint32_t hi = (uint32_t)(v >> 32), lo = (uint32_t)v;
  const uint32_t mhi = __reduce_max_sync(kFull, hi);
  const uint32_t mlo = __reduce_max_sync(kFull, hi == mhi ? lo : 0u);
  return ((uint64_t)mhi << 32) | mlo;
}

__global__ void __launch_bounds__(kWarps * 32) merge_shards_kernel(const __grid_constant__ MergeArgs a) {
  extern __shared__ uint64_t smem_keys[];   // [kWarps][G * C]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q = blockIdx.x * kWarps + warp;
  if (q >= a.B) return;   // whole warps leave together
  const int C = a.C, items = a.G * C;
  uint64_t* keys = smem_keys + (size_t)warp * items;

  // the shards' candidates as packed keys (0 = empty slot); the best key score over all entries
  for (int e = lane; e < items; e += 32) {
    const int g = e / C, i = e - g * C;
    const lacache_shard_result& sh = a.s[g];
    uint64_t key = 0;
    if (i < sh.n_cand[q]) {
      const int64_t gid = sh.id_base + sh.cand_id[(int64_t)q * C + i];
      key = pack_cand(sh.cand_score[(int64_t)q * C + i], (uint32_t)gid);
    }
    keys[e] = key;
  }
  float best = -INFINITY;
  for (int g = lane; g < a.G; g += 32) {
    const lacache_shard_result& sh = a.s[g];
    best = fmaxf(best, sh.n_cand[q] > 0 ? sh.cand_score[(int64_t)q * C] : sh.key_score[q]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) best = fmaxf(best, __shfl_xor_sync(kFull, best, o));
  __syncwarp();

  // C rounds of the warp maximum; lane r remembers the item of round r
  int mine = -1;
  int n = 0;
  for (int r = 0; r < C; ++r) {
    uint64_t local = 0;
    int at = -1;
    for (int e = lane; e < items; e += 32)
      if (keys[e] > local) {
        local = keys[e];
        at = e;
      }
    const uint64_t m = warp_max_u64(local);
    if (m == 0) break;
    const unsigned owner = __ballot_sync(kFull, local == m);
    const int src = __shfl_sync(kFull, at, __ffs(owner) - 1);
    if (lane == __ffs(owner) - 1) keys[src] = 0;
    if (lane == r) mine = src;
    ++n;
    __syncwarp();
  }

  // slot `lane` of the merged list
  const float qnan = __int_as_float(0x7fc00000);
  const bool v = lane < n;
  int g = 0, i = 0;
  if (v) {
    g = mine / C;
    i = mine - g * C;
  }
  const lacache_shard_result& sh = a.s[g];
  const int64_t si = (int64_t)q * C + i;
  const bool pass = v && sh.cand_pass[si] != 0;
  const unsigned passing = __ballot_sync(kFull, pass);
  const int served = passing ? __ffs(passing) - 1 : -1;
  const int shown = served >= 0 ? served : 0;
  const lacache_result& out = a.out;
  if (lane < C) {
    const int64_t o = (int64_t)q * C + lane;
    const int32_t gid = v ? (int32_t)(sh.id_base + sh.cand_id[si]) : -1;
    if (out.cand_id) out.cand_id[o] = gid;
    if (out.cand_score) out.cand_score[o] = v ? sh.cand_score[si] : qnan;
    if (out.cand_prefix_score) out.cand_prefix_score[o] = v ? sh.cand_prefix_score[si] : qnan;
    if (out.cand_matches) out.cand_matches[o] = v ? sh.cand_matches[si] : -1;
    if (out.cand_pass) out.cand_pass[o] = pass ? 1 : 0;
    if (out.cand_prefix_scores)
      for (int h = 0; h < a.m; ++h)
        out.cand_prefix_scores[o * a.m + h] =
            !v ? qnan : (sh.cand_prefix_scores ? sh.cand_prefix_scores[si * a.m + h] : sh.cand_prefix_score[si]);
  }
  if (n > 0 && lane == shown) {
    out.prefix_score[q] = sh.cand_prefix_score[si];
    out.token_matches[q] = sh.cand_matches[si];
    if (out.prefix_scores)
      for (int h = 0; h < a.m; ++h)
        out.prefix_scores[(int64_t)q * a.m + h] =
            sh.cand_prefix_scores ? sh.cand_prefix_scores[si * a.m + h] : sh.cand_prefix_score[si];
    out.status[q] = served >= 0 ? LACACHE_HIT : LACACHE_REJECT;
    out.entry_id[q] = served >= 0 ? (int32_t)(sh.id_base + sh.cand_id[si]) : -1;
    out.key_score[q] = served >= 0 ? sh.cand_score[si] : best;
  }
  if (lane == 0) {
    out.n_cand[q] = n;
    if (n == 0) {
      out.status[q] = LACACHE_MISS_KEY;
      out.entry_id[q] = -1;
      out.key_score[q] = best;
      out.prefix_score[q] = qnan;
      out.token_matches[q] = -1;
      if (out.prefix_scores)
        for (int h = 0; h < a.m; ++h) out.prefix_scores[(int64_t)q * a.m + h] = qnan;
    }
  }
}

}  // namespace
}  // namespace lc

extern "C" lacache_status lacache_merge_shards(int32_t G, const lacache_shard_result* shards, int32_t B,
                                               int32_t top_c, int32_t m, const lacache_result* out,
                                               void* cuda_stream) {
  lc::NvtxRange nvtx("lacache_merge_shards");
  if (G < 1 || G > LACACHE_MAX_SHARDS || !shards || B < 1 || top_c < 1 || top_c > lc::kMaxTopC || m < 1 ||
      m > LACACHE_MAX_MODELS || !out)
    return LACACHE_ERR_INVALID_ARG;
  if (!out->entry_id || !out->status || !out->key_score || !out->prefix_score || !out->token_matches ||
      !out->n_cand)
    return LACACHE_ERR_INVALID_ARG;
  lc::MergeArgs a{};
  a.G = G;
  a.B = B;
  a.C = top_c;
  a.m = m;
  for (int g = 0; g < G; ++g) {
    const lacache_shard_result& s = shards[g];
    if (!s.cand_id || !s.cand_score || !s.cand_prefix_score || !s.cand_matches || !s.cand_pass || !s.key_score ||
        !s.n_cand || (m > 1 && !s.cand_prefix_scores) || s.id_base < 0 || (g > 0 && s.id_base < shards[g - 1].id_base))
      return LACACHE_ERR_INVALID_ARG;
    a.s[g] = s;
  }
  a.out = *out;
  const size_t smem = (size_t)lc::kWarps * G * top_c * sizeof(uint64_t);
  const int grid = (B + lc::kWarps - 1) / lc::kWarps;
  lc::merge_shards_kernel<<<grid, lc::kWarps * 32, smem, (cudaStream_t)cuda_stream>>>(a);
  return cudaGetLastError() == cudaSuccess ? LACACHE_OK : LACACHE_ERR_CUDA;
}

// Internal declarations shared by the lookup kernels and the C-ABI host code of liblacache.so.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include <nvtx3/nvToolsExt.h>

#include "lacache.h"

namespace lc {

// An NVTX range over the enclosing scope: each public call appears by name on a profiler's timeline (a no-op when
// no tool is attached).
class NvtxRange {
 public:
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

constexpr int kMaxTopC = 32;
constexpr int kMaxD = 8192;
constexpr int kMaxK = 256;
constexpr int kMaxModels = LACACHE_MAX_MODELS;

// Bits of the device status word.
constexpr unsigned int kDevTimeout = 1u;

// ---------------------------------------------------------------------------------------------------------------
// Candidate keys. A stage-1 candidate (score s, entry id j) is packed into one uint64 whose unsigned order is the
// candidate order of the lookup: higher score first, then lower entry id. The high word is the score's bits mapped
// to an unsigned order; the low word is ~j. The value 0 is never produced by a finite score and marks "empty".
// -0.0 and +0.0 are equal scores, so both map to the order of +0.0: equal scores then fall to the id rule.
// ---------------------------------------------------------------------------------------------------------------
__host__ __device__ __forceinline__ uint32_t score_order(float s) {
  uint32_t u;
#ifdef __CUDA_ARCH__
  u = __float_as_uint(s);
#else
  memcpy(&u, &s, 4);
#endif
  if (u == 0x80000000u) u = 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__host__ __device__ __forceinline__ float score_of_order(uint32_t o) {
  uint32_t u = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
  float s;
#ifdef __CUDA_ARCH__
  s = __uint_as_float(u);
#else
  memcpy(&s, &u, 4);
#endif
  return s;
}

__host__ __device__ __forceinline__ uint64_t pack_cand(float s, uint32_t j) {
  return ((uint64_t)score_order(s) << 32) | (uint64_t)(~j);
}
__host__ __device__ __forceinline__ float cand_score(uint64_t c) { return score_of_order((uint32_t)(c >> 32)); }
__host__ __device__ __forceinline__ uint32_t cand_id(uint64_t c) { return ~(uint32_t)c; }

// Stage-1 output, per split s and query q: a record of the split's best key score (over all its entries: a miss
// reports the best over the store) and of how many candidates its partial list holds, and the list itself, sorted,
// in its first `count` slots (later slots are not written: most lists hold few candidates, or none).
//   part_meta[s * B + q], part_cand[(s * B + q) * top_c + i] for i < count
struct __align__(8) PartMeta {
  float best;
  uint32_t count;
};

struct Stage1Args {
  const __nv_bfloat16* keys;  // [n x d] store keys
  int64_t n;
  int d;
  const __nv_bfloat16* q;     // [B x d] query embeddings
  int B;
  float tau_c;
  int top_c;
  uint64_t* part_cand;
  PartMeta* part_meta;
  unsigned int* dev_status;
  int inject_stall;           // test support: CTA 0 of the tensor kernel, or of the SimHash scan's ring form,
                              // withholds one load (see lacache.h)
  int* tile_ctr;              // tensor kernel, one query tile: dynamic tile schedule on these two counters
                              // [next tile, CTAs done], zero at launch and zero again when the grid ends
                              // (nullptr: static schedule)
  int inputs_from_previous;   // tensor kernel: the queries are written by the grid launched just before (the
                              // host-input gather), so wait for it before reading anything
};

struct Stage2Args {
  int64_t n;                     // valid entries: candidate ids at or past n are dropped
  const uint64_t* part_cand;
  const PartMeta* part_meta;
  int splits;
  int B;
  int pd;                        // prefix row length: sum of the models' dimensions
  int k;
  int top_c;
  int m;                         // lookahead checks (models)
  int seg[kMaxModels + 1];       // model h owns prefix row elements [seg[h], seg[h+1]), multiples of 8
  float tau_m[kMaxModels];       // model h's threshold
  int check_mode;
  int token_match_min;
  const __nv_bfloat16* prefix;   // [n x pd] store prefix embeddings
  const int32_t* ids;            // [n x k] store prefix token ids
  const __nv_bfloat16* q_prefix; // [B x pd]
  const int32_t* q_ids;          // [B x k]
  lacache_result out;            // device pointers
  unsigned long long* counters;  // decision counters [hits, rejects, key misses], or nullptr
};

// cuTensorMapEncodeTiled, obtained from the driver at run time.
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// Launchers (host). Each returns the CUDA error of the launch. `splits` is the number of partial lists written.
// The streaming CUDA-core scan (warp per key tile); batches past its shared-memory budget take several launches.
cudaError_t launch_stage1_stream(const Stage1Args& a, int num_sms, int max_splits, cudaStream_t st, int* splits);
// Encodes its own TMA descriptors for a.q and a.keys with `encode`.
// *paired (if not null) is set when the batch ran on CTA pairs.
cudaError_t launch_stage1_tensor(const Stage1Args& a, EncodeTiledFn encode, int num_sms, int max_splits,
                                 cudaStream_t st, int* splits, bool* paired = nullptr);
cudaError_t launch_stage2(const Stage2Args& a, cudaStream_t st);

// SimHash signatures of n rows ([n x d] bf16) against `bits` hyperplanes ([bits x d] bf16), bits a multiple of 32:
// sig[j * bits/32 + w] bit i is set iff <hyperplane 32w + i, row j> >= 0 (tensor-core GEMM, sign epilogue).
// rows_from_previous: the rows are written by the grid launched just before (wait for it before reading).
cudaError_t launch_signatures(const __nv_bfloat16* rows, int64_t n, int d, const __nv_bfloat16* hyperplanes,
                              int bits, uint32_t* sig, unsigned int* dev_status, EncodeTiledFn encode, int num_sms,
                              cudaStream_t st, bool rows_from_previous = false);

// Query signatures of a batch of at most kSignCudaCoreMaxBatch queries on the CUDA cores, in the bit layout of
// launch_signatures (one CTA per query and 32-bit word). q_from_previous: the queries are written by the grid
// launched just before. Measured per lookup on mid-1m at b = 256 against the tensor-core GEMM: 27.4 -> 18.2 us at
// B = 1, 64.6 -> 61.7 us at B = 40, level at 128-256 queries, slower at 512.
constexpr int kSignCudaCoreMaxBatch = 128;
cudaError_t launch_sign_queries(const __nv_bfloat16* q, int B, int d, const __nv_bfloat16* hyperplanes, int bits,
                                uint32_t* qsig, cudaStream_t st, bool q_from_previous);

// The SimHash-indexed key check: entries whose signature is within `radius` of the query's get the exact key
// check (threshold + top-c partial lists, as the other stage-1 kernels).
struct LshArgs {
  const uint32_t* sig;     // [n x words] entry signatures
  const uint32_t* qsig;    // [B x words] query signatures
  int words;
  int radius;
  const uint8_t* index;    // the same signatures as e4m3 +-1 bytes in swizzled 128-entry blocks (lsh_tc.cu)
};
// Popcount scan (small batches) and the tensor-core scan over the expanded index (batches of at least
// lsh_tensor_min_batch(bits) queries).
// *ring: the launch runs the scan's shared-memory ring form (the only form with bounded waits, so the only one a
// stall injection, a.inject_stall, acts on).
cudaError_t launch_stage1_lsh(const Stage1Args& a, const LshArgs& l, int num_sms, int max_splits, cudaStream_t st,
                              int* splits, bool* ring);
cudaError_t launch_stage1_lsh_tc(const Stage1Args& a, const LshArgs& l, int num_sms, int max_splits,
                                 cudaStream_t st, int* splits);
// The switch between them, measured per lookup step on mid-1m with both scans forced (popcount scan with its prefix
// test / tensor-core scan, us): 128 bits, B = 32 48.1 / 56.7, B = 40 61.0 / 57.4; 256 bits, B = 40 74.0 / 80.8,
// B = 48 81.6 / 81.6, B = 64 97.5 / 82.4; 512 bits, B = 32 77.5 / 97.6, B = 40 104.2 / 98.9. Past 32 queries the
// popcount scan makes a second pass over the index.
inline int lsh_tensor_min_batch(int bits) { return bits == 256 ? 48 : 40; }
// Bytes of the expanded index for `capacity` entries (whole 128-entry blocks of `bits` bytes each), and its update
// from the packed signatures of entries [first, first + n).
size_t lsh_index_bytes(int64_t capacity, int bits);
cudaError_t launch_expand_signatures(const uint32_t* sig, int64_t first, int64_t n, int bits, uint8_t* index,
                                     int num_sms, cudaStream_t st);

// LACACHE_STAGE1_AUTO's choice for a lookup of B queries against n keys of d elements, from measurements of both
// kernels. Once the keys stream from HBM, the tensor-core scan holds the copy bandwidth at every batch size (1.05-1.09
// of it from 1 to 128 queries). The streaming scan matches or passes it for one or two queries at d = 1024, where
// every lane has its whole share of a row, four 16-byte chunks, in flight per tile (585.6 against 590.9 us at
// 2M x 1024 and one query), and falls behind with fewer chunks per lane, several phases or more queries (d = 800,
// 896 and 1280 trail by 1-2 %). On stores of up to some tens of MB the scan is bound by latency: the tensor-core
// scan takes a nearly flat 9-16 us a lookup, while the streaming scan's time grows with its multiply-adds, n d B.
// Back-to-back lookups cross over at about 2^25 of them: 4,096 x 384, B = 16: 13.7 against 14.0 us a lookup;
// 16,384 x 768, B = 2: 8.9 against 8.9, B = 4: 10.4 against 8.9; 43,690 x 768 (67 MB of keys), B = 1: 10.6 against
// 13.3, B = 2: 13.6 against 13.1. A single lookup on an idle device crosses later (16,384 x 768, B = 4: 18.2
// against 21.2 us), and from a flushed L2 the streaming scan's stage 1 is also the shorter one at that size (22.3
// against 25.9 us at 43,690 x 768, B = 1). So the streaming scan takes the lookups with n d B <= 2^25 (at most
// 64 MiB of keys, at one query).
constexpr int64_t kStreamAutoMacs = (int64_t)1 << 25;
inline int auto_stage1(int64_t n, int d, int B) {
  if (n * d * B <= kStreamAutoMacs) return LACACHE_STAGE1_STREAM;
  if (B <= 2 && d == 1024) return LACACHE_STAGE1_STREAM;
  return LACACHE_STAGE1_TENSOR;
}

// Largest split count the stage-1 launchers may use on a handle (sizes its partial-list scratch). The SimHash scan
// runs two CTAs per SM and the single-CTA kernels one split per SM. The CTA-pair schedule wants small splits, so
// that the pairs sharing a key range read it from L2 (about 600 for 6 GB of keys); it may use up to 4 per SM while
// the scratch of max_batch x top_c candidates per split stays within 1 GiB.
inline int max_splits_for(int num_sms, int max_batch, int top_c) {
  const int64_t per_split = (int64_t)max_batch * top_c * 8;
  const int64_t budget = ((int64_t)1 << 30) / per_split;
  const int64_t more = budget < 4 * (int64_t)num_sms ? budget : 4 * (int64_t)num_sms;
  return more > 2 * num_sms ? (int)more : 2 * num_sms;
}

}  // namespace lc

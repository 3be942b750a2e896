// Stage 1 through the SimHash index (Eq. 1; Algorithm 1's "search semantic cache with key h(x)"): the key check
// sim(x, x') >= tau_c applied only to the entries whose signature is within `radius` bits of the query's.
//
// One CTA per contiguous split of the entries (two per SM); one entry per thread per tile of 512. A thread counts
// the differing bits of its entry's signature against each of up to 32 query signatures held in shared memory. The
// signatures arrive in one of two ways (bulk_ring() picks one per launch):
//  - registers: each thread loads its entry's words with 16-byte loads one tile ahead. The fewest instructions
//    around the distance arithmetic, so the form for the ALU-bound scans (several queries at 128 or 256 bits).
//  - a ring of tile-sized shared-memory stages, one bulk copy (cp.async.bulk) per tile, issued by thread 0 and
//    completed on the stage's mbarrier; a stage is refilled after the tile's CTA barrier, so kStages - 1 tiles are
//    in flight while one is counted. Twice the bytes in flight, and W registers free: the form for the scans bound
//    by memory (one query on a large store) and for 512-bit signatures.
// The distance test first counts the differing bits of a prefix of P of the W words (the kernel's P parameter): a
// pair whose prefix distance already exceeds the radius is out, since the prefix distance never exceeds the whole
// one. With the radii the thresholds give, nearly every pair of unrelated signatures is out after the prefix
// (use_prefix() keeps the test where the binomial tail of a random pair's prefix distance says so), and the few
// left in each thread's mask get the whole distance in a loop over that mask. P = W tests the whole signature.
// Admitted (query, entry) pairs are queued in shared memory.
// When the queue passes three quarters of its capacity, and at the end of the split, all warps take queue items two
// at a time and compute the exact fp32 score over the gathered key row (each lane's 8-element chunks in order,
// then a butterfly sum). The warp of each query then folds the scores that clear tau_c into that query's top-c
// list. A tile can admit more pairs than the queue has room for (up to 512 x 32, e.g. with radius = bits): a pair
// that finds the queue full stays in its thread's pending mask and is queued again after the next flush. The
// partial lists have the format of the other stage-1 kernels, so stage 2 is shared.
#include <cmath>

#include "internal.cuh"
#include "tcgen05.cuh"

namespace lc {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kTile = kThreads;     // entries per tile, one per thread
constexpr int kQC = 32;             // queries per pass over the entries (one bit each in a thread's masks)
constexpr unsigned kFull = 0xffffffffu;

// Per signature width (W words) and form: the queue capacity and the depth of the signature ring. Two CTAs share an
// SM's 228 KB. Without a ring the queue takes 8,192 items (12 bytes each); with one, the queue and the ring
// (kTile * W * 4 bytes a stage: 8 / 16 / 32 KB at W = 4 / 8 / 16) split about 100 KB, and kStages - 1 tiles, 40 /
// 32 / 32 KB, are in flight per CTA while one is counted.
template <int W, bool Bulk>
struct Geo {
  static constexpr int kCap = !Bulk ? 8192 : W == 16 ? 2048 : 4096;
  static constexpr int kStages = !Bulk ? 1 : W == 4 ? 6 : W == 8 ? 3 : 2;
  static constexpr int kFlushAt = kCap - kCap / 4;   // a tile that leaves more items than this is followed by a flush
  static constexpr int kRingWords = Bulk ? kTile * W : 4;   // a stage (a placeholder without the ring)
};

struct Item {
  int32_t j;      // entry id
  int32_t q;      // query within the pass
};

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

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

// The ring and the query signatures are read as 16-byte vectors (and the ring is a bulk-copy destination), so
// both sit on 16-byte boundaries (checked in launch_w).
template <int W, bool Bulk>
struct Shared {
  using G = Geo<W, Bulk>;
  alignas(16) uint32_t ring[G::kStages][G::kRingWords];   // entry t of a tile at words [t W, t W + W) of its stage
  alignas(16) uint32_t qsig[kQC][W];
  uint64_t bar[G::kStages];       // stage full: thread 0's arrive with the bytes, then the copy's
  uint64_t list[kQC][kMaxTopC];   // per query: sorted packed candidates of this split, 0 = empty
  unsigned int best[kQC];         // score_order of the best admitted score
  int count;                      // queued items
  Item items[G::kCap];
  float score[G::kCap];
};

// Exact scores of the queued items, then each query's warp folds its items into the query's list.
template <int W, bool Bulk>
__device__ void flush(Shared<W, Bulk>& sh, const Stage1Args& a, int q0, int qn) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int total = min(sh.count, Geo<W, Bulk>::kCap);   // pairs that found the queue full were not stored
  const int v = a.d / 8;
  for (int base = warp * 2; base < total; base += kWarps * 2) {
    float acc0 = 0.f, acc1 = 0.f;
    const Item i0 = sh.items[base];
    const bool two = base + 1 < total;
    const Item i1 = two ? sh.items[base + 1] : i0;
    const uint4* k0 = reinterpret_cast<const uint4*>(a.keys + (int64_t)i0.j * a.d);
    const uint4* k1 = reinterpret_cast<const uint4*>(a.keys + (int64_t)i1.j * a.d);
    const uint4* x0 = reinterpret_cast<const uint4*>(a.q + (int64_t)(q0 + i0.q) * a.d);
    const uint4* x1 = reinterpret_cast<const uint4*>(a.q + (int64_t)(q0 + i1.q) * a.d);
    for (int c = lane; c < v; c += 32) {
      acc0 = dot8(__ldg(x0 + c), __ldg(k0 + c), acc0);
      acc1 = dot8(__ldg(x1 + c), __ldg(k1 + c), acc1);
    }
    acc0 = warp_sum(acc0);
    acc1 = warp_sum(acc1);
    if (lane == 0) {
      sh.score[base] = acc0;
      if (two) sh.score[base + 1] = acc1;
    }
  }
  __syncthreads();
  const int C = a.top_c;
  for (int qq = warp; qq < qn; qq += kWarps) {
    float best = -INFINITY;
    for (int base = 0; base < total; base += 32) {
      const int idx = base + lane;
      const bool mine = idx < total && sh.items[idx].q == qq;
      const float sc = mine ? sh.score[idx] : -INFINITY;
      best = fmaxf(best, sc);
      unsigned pass = __ballot_sync(kFull, mine && sc >= a.tau_c);
      while (pass) {   // lane 0 inserts the passing items of this group one by one
        const int src = __ffs(pass) - 1;
        pass &= pass - 1;
        const float s = __shfl_sync(kFull, sc, src);
        const int j = __shfl_sync(kFull, mine ? sh.items[idx].j : 0, src);
        if (lane == 0) {
          uint64_t x = pack_cand(s, (uint32_t)j);
          uint64_t* L = sh.list[qq];
          if (x > L[C - 1]) {
            int p = C - 1;
            while (p > 0 && L[p - 1] < x) {
              L[p] = L[p - 1];
              --p;
            }
            L[p] = x;
          }
        }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) best = fmaxf(best, __shfl_xor_sync(kFull, best, o));
    if (lane == 0 && best > -INFINITY) atomicMax(&sh.best[qq], score_order(best));
  }
  __syncthreads();
  if (threadIdx.x == 0) sh.count = 0;
  __syncthreads();
}

// Carry-save adder on 32 bit positions at once: a + b + c = lo + 2 hi in every position (two LOP3 operations).
__device__ __forceinline__ void csa(uint32_t& hi, uint32_t& lo, uint32_t a, uint32_t b, uint32_t c) {
  const uint32_t u = a ^ b;
  lo = u ^ c;
  hi = (a & b) | (u & c);
}

// Number of set bits in x[0..N) (N = 4, 8 or 16). Population count runs at 16 per clock per SM, the logic
// operations at 64, so carry-save adders first fold words into sum and carry words, each group of 8 words into 5
// popcounts (3 adders):
//   x0 + x1 + x2 = sa + 2 ca,  x3 + x4 + x5 = sb + 2 cb,  sa + sb + x6 = sc + 2 cc,
//   |x0..x7| = |sc| + |x7| + 2 (|ca| + |cb| + |cc|);
// a group of 4 words into 3 (one adder). The count is exact.
template <int N, int W>
__device__ __forceinline__ int hamming(const uint32_t (&x)[W]) {
  static_assert(N <= W, "a prefix of the signature");
  int h = 0;
  if constexpr (N % 8 == 0) {
#pragma unroll
    for (int g = 0; g < N; g += 8) {
      uint32_t ca, sa, cb, sb, cc, sc;
      csa(ca, sa, x[g], x[g + 1], x[g + 2]);
      csa(cb, sb, x[g + 3], x[g + 4], x[g + 5]);
      csa(cc, sc, sa, sb, x[g + 6]);
      h += __popc(sc) + __popc(x[g + 7]) + 2 * (__popc(ca) + __popc(cb) + __popc(cc));
    }
  } else {
    static_assert(N % 4 == 0, "signature words come in groups of 4");
#pragma unroll
    for (int g = 0; g < N; g += 4) {
      uint32_t c, s;
      csa(c, s, x[g], x[g + 1], x[g + 2]);
      h += __popc(s) + __popc(x[g + 3]) + 2 * __popc(c);
    }
  }
  return h;
}

// Number of set bits in x[0..N) for a prefix of N = 3 or 5 words (one or two carry-save adders):
//   N = 3: x0 + x1 + x2 = s + 2 c;                        |x| = |s| + 2 |c|
//   N = 5: x0 + x1 + x2 = s1 + 2 c1, s1 + x3 + x4 = s2 + 2 c2;  |x| = |s2| + 2 (|c1| + |c2|)
// and hamming() for N = 4, 8 or 16.
template <int N, int W>
__device__ __forceinline__ int prefix_count(const uint32_t (&x)[W]) {
  if constexpr (N == 3) {
    uint32_t c, s;
    csa(c, s, x[0], x[1], x[2]);
    return __popc(s) + 2 * __popc(c);
  } else if constexpr (N == 5) {
    uint32_t c1, s1, c2, s2;
    csa(c1, s1, x[0], x[1], x[2]);
    csa(c2, s2, s1, x[3], x[4]);
    return __popc(s2) + 2 * (__popc(c1) + __popc(c2));
  } else {
    return hamming<N, W>(x);
  }
}

// Signature words of entry j into e (zeros past the split's end).
template <int W>
__device__ __forceinline__ void load_sig(const uint32_t* sig, int64_t j, int64_t j_end, uint32_t (&e)[W]) {
  if (j < j_end) {
    const uint4* src = reinterpret_cast<const uint4*>(sig + j * W);
#pragma unroll
    for (int w = 0; w < W / 4; ++w) {
      const uint4 u = __ldg(src + w);
      e[4 * w] = u.x;
      e[4 * w + 1] = u.y;
      e[4 * w + 2] = u.z;
      e[4 * w + 3] = u.w;
    }
  } else {
#pragma unroll
    for (int w = 0; w < W; ++w) e[w] = 0u;
  }
}

// Thread 0: tile `ti` of the split (entries j_begin + ti * kTile ..., at most j_end) into stage `st`, as one bulk
// copy completing on the stage's barrier. The split's signatures are contiguous and 16-byte aligned (W >= 4 words an
// entry), and a tile's byte count is a multiple of 16.
template <int W>
__device__ __forceinline__ void fetch_tile(Shared<W, true>& sh, const uint32_t* sig, int64_t j_begin, int64_t j_end,
                                           int64_t ti, int st) {
  const int64_t t0 = j_begin + ti * kTile;
  const uint32_t bytes = (uint32_t)min((int64_t)kTile, j_end - t0) * W * 4;
  const uint32_t bar = smem_u32(&sh.bar[st]);
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // the stage's last generic reads come first
  mbar_expect_tx(bar, bytes);
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               ::"r"(smem_u32(sh.ring[st])), "l"(sig + t0 * W), "r"(bytes), "r"(bar)
               : "memory");
}

template <int W, bool Bulk, int P>
__global__ void __launch_bounds__(kThreads, 2) lsh_scan_kernel(Stage1Args a, LshArgs l, int splits) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  using G = Geo<W, Bulk>;
  Shared<W, Bulk>& sh = *reinterpret_cast<Shared<W, Bulk>*>(smem_raw);
  constexpr int S = G::kStages;
  if (Bulk && threadIdx.x == 0) {
    for (int st = 0; st < S; ++st) mbar_init(smem_u32(&sh.bar[st]), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int s = blockIdx.x;
  const int64_t j_begin = a.n * s / splits, j_end = a.n * (s + 1) / splits;
  const int64_t tiles = (j_end - j_begin + kTile - 1) / kTile;
  const int C = a.top_c;
  // Ring form: stage uses are numbered across the passes: use u sits in stage u % S, and its copy completes the stage
  // barrier's phase of parity (u / S) & 1. A thread whose wait for a tile runs out (about a second) records the
  // timeout and reads no further tiles, but keeps to the CTA's barriers, so every pass still ends and writes its
  // lists (the host reads the timeout from the status word). Thread 0 then issues no further copies and, before the
  // CTA exits, waits (again with a limit) for the copies it had issued past the tile it gave up on.
  uint32_t u0 = 0;           // first use of this pass
  bool live = true;
  int64_t issued = 0;        // thread 0: copies issued in this pass
  uint32_t drain_first = 0;  // thread 0, once it gave up: the first use still in flight, and how many
  int64_t drain_count = 0;
  for (int q0 = 0; q0 < a.B; q0 += kQC) {
    const int qn = min(kQC, a.B - q0);
    if constexpr (Bulk) {
      if (threadIdx.x == 0 && live) {
        // test support: CTA 0 withholds the copy of its first tile (no arrive either), so every thread's wait for
        // it runs out; the withheld copy counts as issued, and the drain below waits for it in vain (bounded)
        const bool withhold = a.inject_stall && blockIdx.x == 0 && q0 == 0;
        for (issued = 0; issued < min((int64_t)S, tiles); ++issued)
          if (!(withhold && issued == 0))
            fetch_tile<W>(sh, l.sig, j_begin, j_end, issued, (int)((u0 + issued) % S));
      }
    }
    for (int i = threadIdx.x; i < kQC * W; i += kThreads) {
      const int qq = i / W;
      sh.qsig[qq][i % W] = qq < qn ? l.qsig[(int64_t)(q0 + qq) * W + i % W] : 0u;
    }
    for (int i = threadIdx.x; i < kQC * kMaxTopC; i += kThreads) sh.list[i / kMaxTopC][i % kMaxTopC] = 0;
    if (threadIdx.x < kQC) sh.best[threadIdx.x] = score_order(-INFINITY);
    if (threadIdx.x == 0) sh.count = 0;
    __syncthreads();
    const unsigned qmask = qn >= 32 ? kFull : (1u << qn) - 1u;
    // register form: the next tile's signatures are loaded before the current tile is counted
    uint32_t nxt[W];
    if constexpr (!Bulk) load_sig<W>(l.sig, j_begin + threadIdx.x, j_end, nxt);
    for (int64_t ti = 0; ti < tiles; ++ti) {
      const int64_t j = j_begin + ti * kTile + threadIdx.x;
      const uint32_t use = u0 + (uint32_t)ti;
      const int st = (int)(use % S);
      bool ok = true;
      uint32_t e[W];
      if constexpr (Bulk) {
        ok = false;
        if (live) {
          ok = mbar_wait(smem_u32(&sh.bar[st]), (use / S) & 1u, nullptr);
          if (!ok) {
            live = false;
            atomicOr(a.dev_status, kDevTimeout);
            if (threadIdx.x == 0) {   // tiles ti .. issued - 1 of this pass may still be in flight
              drain_first = use;
              drain_count = issued - ti;
            }
          }
        }
        const uint4* src = reinterpret_cast<const uint4*>(&sh.ring[st][threadIdx.x * W]);
#pragma unroll
        for (int c = 0; c < W / 4; ++c) {
          const uint4 v = ok ? src[c] : make_uint4(0u, 0u, 0u, 0u);
          e[4 * c] = v.x;
          e[4 * c + 1] = v.y;
          e[4 * c + 2] = v.z;
          e[4 * c + 3] = v.w;
        }
      } else {
#pragma unroll
        for (int w = 0; w < W; ++w) e[w] = nxt[w];
        load_sig<W>(l.sig, j + kTile, j_end, nxt);
      }
      // every query's distance first, as a mask of the admitted queries (the queue stores below could alias the
      // query signatures for the compiler): whole groups of 8 queries unrolled, then the pass's remaining queries
      // (a uniform count), so a pass of one query computes one distance. With a prefix test (P < W) the loop
      // leaves the queries within the radius on the first P words in `cand`, and each gets its whole distance
      // after it.
      unsigned pend = 0, cand = 0;
      auto test_query = [&](int qq) {
        const uint4* qs = reinterpret_cast<const uint4*>(sh.qsig[qq]);
        uint32_t x[W];
#pragma unroll
        for (int w = 0; w < (P + 3) / 4; ++w) {
          const uint4 v = qs[w];
          x[4 * w] = e[4 * w] ^ v.x;
          if (4 * w + 1 < P) x[4 * w + 1] = e[4 * w + 1] ^ v.y;
          if (4 * w + 2 < P) x[4 * w + 2] = e[4 * w + 2] ^ v.z;
          if (4 * w + 3 < P) x[4 * w + 3] = e[4 * w + 3] ^ v.w;
        }
        const unsigned bit = (prefix_count<P, W>(x) <= l.radius ? 1u : 0u) << qq;
        if constexpr (P == W) pend |= bit; else cand |= bit;
      };
      const int whole = qn & ~7;
      for (int g = 0; g < whole; g += 8) {
#pragma unroll
        for (int u = 0; u < 8; ++u) test_query(g + u);
      }
      for (int qq = whole; qq < qn; ++qq) test_query(qq);
      if constexpr (P < W) {
        while (cand) {   // this thread's few candidates, each with its whole distance
          const int qq = __ffs(cand) - 1;
          cand &= cand - 1;
          const uint4* qs = reinterpret_cast<const uint4*>(sh.qsig[qq]);
          uint32_t x[W];
#pragma unroll
          for (int w = 0; w < W / 4; ++w) {
            const uint4 v = qs[w];
            x[4 * w] = e[4 * w] ^ v.x;
            x[4 * w + 1] = e[4 * w + 1] ^ v.y;
            x[4 * w + 2] = e[4 * w + 2] ^ v.z;
            x[4 * w + 3] = e[4 * w + 3] ^ v.w;
          }
          pend |= (hamming<W, W>(x) <= l.radius ? 1u : 0u) << qq;
        }
      }
      pend = ok && j < j_end ? pend & qmask : 0u;
      // Queue the admitted pairs; flush while the queue is past kFlushAt or a pair found it full. Every round of
      // this loop either queues all pending pairs or fills the queue, so it ends.
      int top = -1;   // the highest queue slot this thread took in this round
      for (;;) {
        unsigned full = 0;
        while (pend) {
          const int qq = __ffs(pend) - 1;
          pend &= pend - 1;
          const int slot = atomicAdd(&sh.count, 1);
          if (slot < G::kCap) {
            sh.items[slot] = Item{(int32_t)j, qq};
            top = slot;
          } else {
            full |= 1u << qq;
          }
        }
        pend = full;
        // the barrier's OR gives every thread the same answer (a read of the count after a plain barrier
        // could already see the next tile's items in some threads)
        if (!__syncthreads_or(pend != 0 || top >= G::kFlushAt)) break;
        flush<W, Bulk>(sh, a, q0, qn);
        top = -1;
      }
      if constexpr (Bulk) {
        // every thread has read stage st (the barrier above): thread 0 refills it with the tile S ahead
        if (threadIdx.x == 0 && live && ti + S < tiles) {
          fetch_tile<W>(sh, l.sig, j_begin, j_end, ti + S, st);
          ++issued;
        }
      }
    }
    u0 += (uint32_t)tiles;
    flush<W, Bulk>(sh, a, q0, qn);
    // the lists' candidates (a sorted list holds them in its first slots, then zeros) and each list's record
    for (int i = threadIdx.x; i < qn * C; i += kThreads) {
      const int qq = i / C;
      const uint64_t x = sh.list[qq][i - qq * C];
      if (x) a.part_cand[((int64_t)s * a.B + q0 + qq) * C + (i - qq * C)] = x;
    }
    if (threadIdx.x < qn) {
      uint32_t count = 0;
      while ((int)count < C && sh.list[threadIdx.x][count]) ++count;
      a.part_meta[(int64_t)s * a.B + q0 + threadIdx.x] = PartMeta{score_of_order(sh.best[threadIdx.x]), count};
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    // each pending copy gets its own bounded wait: one that never arrives does not cut short the wait for the
    // others, which may still be writing this CTA's shared memory
    for (int64_t k = 0; k < drain_count; ++k) {
      const uint32_t u = drain_first + (uint32_t)k;
      mbar_wait(smem_u32(&sh.bar[u % S]), (u / S) & 1u, nullptr);
    }
  }
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Query signatures of a small batch on the CUDA cores. The tensor-core GEMM that signs entries at insert runs only
// bits / 128 CTAs with a dozen dependent k-steps each, about 11.5 us whatever the batch; here one CTA per (query,
// 32-hyperplane word) takes one memory round trip. Warp i computes hyperplanes 32w + 4i .. 32w + 4i + 3: lane l reads
// the rows' 16-byte chunks l, l + 32, ... (coalesced), accumulates in fp32 (each lane's chunks in order), and a
// butterfly reduce-scatter of the four sums leaves hyperplane 4i + l / 8's dot in lanes l. Bit h of word w is set
// iff <hyperplane 32w + h, query> >= 0, as for the entries' signatures.
__global__ void __launch_bounds__(256) sign_queries_kernel(const __nv_bfloat16* __restrict__ q, int d,
                                                           const __nv_bfloat16* __restrict__ hyper, int words,
                                                           uint32_t* __restrict__ qsig, int wait_first) {
  __shared__ uint32_t part[8];
  if (wait_first) asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int w = blockIdx.x % words, qi = blockIdx.x / words;
  const int dc = d / 8;
  const uint4* qrow = reinterpret_cast<const uint4*>(q + (int64_t)qi * d);
  const uint4* hrow = reinterpret_cast<const uint4*>(hyper + (int64_t)(32 * w + 4 * warp) * d);
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
  for (int c = lane; c < dc; c += 32) {
    const uint4 qv = __ldg(qrow + c);
    uint4 hv[4];
#pragma unroll
    for (int h = 0; h < 4; ++h) hv[h] = __ldg(hrow + (int64_t)h * dc + c);
#pragma unroll
    for (int h = 0; h < 4; ++h) acc[h] = dot8(hv[h], qv, acc[h]);
  }
  // reduce-scatter of four values: after two halving steps lane l holds value l / 8's sum over 4 lanes, and three
  // more steps add across the lanes that share it
  const bool hi16 = (lane & 16) != 0, hi8 = (lane & 8) != 0;
  float x0 = (hi16 ? acc[2] : acc[0]) + __shfl_xor_sync(kFull, hi16 ? acc[0] : acc[2], 16);
  float x1 = (hi16 ? acc[3] : acc[1]) + __shfl_xor_sync(kFull, hi16 ? acc[1] : acc[3], 16);
  float v = (hi8 ? x1 : x0) + __shfl_xor_sync(kFull, hi8 ? x0 : x1, 8);
#pragma unroll
  for (int o = 4; o >= 1; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  const unsigned ballot = __ballot_sync(kFull, (lane & 7) == 0 && v >= 0.f);
  if (lane == 0) {
    uint32_t b = 0;
#pragma unroll
    for (int h = 0; h < 4; ++h) b |= ((ballot >> (8 * h)) & 1u) << h;
    part[warp] = b << (4 * warp);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t word = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) word |= part[i];
    asm volatile("griddepcontrol.wait;" ::: "memory");   // the previous lookup's scan has read qsig
    qsig[(int64_t)qi * words + w] = word;
  }
}

// The scan is a programmatic dependent launch of the query-signature kernel: its CTAs may be scheduled while the
// signatures are computed and wait in griddepcontrol.wait, which hides the launch gap.
template <int W, bool Bulk, int P>
cudaError_t launch_w(const Stage1Args& a, const LshArgs& l, int splits, cudaStream_t st) {
  using Sh = Shared<W, Bulk>;
  static_assert(offsetof(Sh, ring) % 16 == 0 && offsetof(Sh, qsig) % 16 == 0 &&
                    (sizeof(uint32_t) * Geo<W, Bulk>::kRingWords) % 16 == 0 && offsetof(Sh, bar) % 8 == 0,
                "16-byte vector reads and bulk copies need 16-byte aligned rows; mbarriers 8 bytes");
  static_assert(2 * (sizeof(Sh) + 1024) <= 228 * 1024, "two CTAs per SM");
  const size_t smem = sizeof(Sh);
  cudaError_t e = cudaFuncSetAttribute(lsh_scan_kernel<W, Bulk, P>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(splits);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, lsh_scan_kernel<W, Bulk, P>, a, l, splits);
}

// The ring form for scans bound by memory, the register form for those bound by the distance arithmetic. Measured
// per lookup step, both forms forced, mid-1m (1M entries) from a flushed L2 and large-16m (16.7M entries):
//  - 512-bit signatures: the ring is faster at every batch tried (1 to 32 queries; 177 against 223 us at one query
//    on large-16m), its 16 free registers counting as much as the bytes in flight;
//  - 128 and 256 bits: the ring is faster only for one query on a store of at least 16 tiles per split (86 against
//    101 us at 256 bits on large-16m, 82 against 90 at 128); at two or more queries, or on mid-1m's 7 tiles per
//    split, the register form is as fast or faster (up to 10 %).
bool bulk_ring(int words, int B, int64_t n, int splits) {
  return words == 16 || (B == 1 && n / splits >= 16 * (int64_t)kTile);
}

// Probability that two independent uniformly random n-bit strings differ in at most r positions.
double random_pair_within(int n, int r) {
  if (r >= n) return 1.0;
  double p = 0.0;
  for (int i = 0; i <= r; ++i) p += std::exp(std::lgamma(n + 1.0) - std::lgamma(i + 1.0) - std::lgamma(n - i + 1.0));
  return p * std::exp(-n * std::log(2.0));
}

// The distance test's prefix: 3, 5 or 8 words at W = 4, 8 or 16 (96, 160 or 256 bits) when at most 2 % of
// unrelated pairs (whose distance is about that of random strings) stay within the radius on it, else the whole
// signature. At the radii the thresholds give (35, 60 and 106 bits at tau_c = 0.9) the prefix keeps 0.5 %, 0.1 %
// and 0.4 % of them.
template <int W>
constexpr int kPrefixWords = W == 4 ? 3 : W == 8 ? 5 : 8;
template <int W>
bool use_prefix(int radius) {
  return random_pair_within(32 * kPrefixWords<W>, radius) <= 0.02;
}

template <int W>
cudaError_t launch_form(bool bulk, const Stage1Args& a, const LshArgs& l, int splits, cudaStream_t st) {
  constexpr int P = kPrefixWords<W>;
  const bool prefix = use_prefix<W>(l.radius);
  if constexpr (W == 16) {   // 512-bit signatures always take the ring form
    return prefix ? launch_w<W, true, P>(a, l, splits, st) : launch_w<W, true, W>(a, l, splits, st);
  } else {
    if (prefix) return bulk ? launch_w<W, true, P>(a, l, splits, st) : launch_w<W, false, P>(a, l, splits, st);
    return bulk ? launch_w<W, true, W>(a, l, splits, st) : launch_w<W, false, W>(a, l, splits, st);
  }
}

}  // namespace

cudaError_t launch_sign_queries(const __nv_bfloat16* q, int B, int d, const __nv_bfloat16* hyperplanes, int bits,
                                uint32_t* qsig, cudaStream_t st, bool q_from_previous) {
  const int words = bits / 32;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(B * words));
  cfg.blockDim = dim3(256);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, sign_queries_kernel, q, d, hyperplanes, words, qsig, q_from_previous ? 1 : 0);
}

cudaError_t launch_stage1_lsh(const Stage1Args& a, const LshArgs& l, int num_sms, int max_splits, cudaStream_t st,
                              int* splits, bool* ring) {
  const int64_t tiles = (a.n + kTile - 1) / kTile;
  int s = (int)(tiles < 2 * (int64_t)num_sms ? tiles : 2 * (int64_t)num_sms);
  if (s > max_splits) s = max_splits;
  if (s < 1) s = 1;
  *splits = s;
  const bool bulk = bulk_ring(l.words, a.B, a.n, s);
  *ring = bulk;
  switch (l.words) {   // 128, 256 or 512-bit signatures (16-byte loads)
    case 4: return launch_form<4>(bulk, a, l, s, st);
    case 8: return launch_form<8>(bulk, a, l, s, st);
    case 16: return launch_form<16>(bulk, a, l, s, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace lc

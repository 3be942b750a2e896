// Stage 1 through the SimHash index (Eq. 1; Algorithm 1's "search semantic cache with key h(x)"): the key check
// sim(x, x') >= tau_c applied only to the entries whose signature is within `radius` bits of the query's.
//
// One CTA per contiguous split of the entries (two per SM); one entry per thread per tile of 512. A thread loads
// its entry's signature (16-byte loads, one tile ahead, into registers) and counts the differing bits against each
// of up to 32 query signatures held in shared memory. Admitted (query, entry) pairs are queued in shared memory.
// When the queue passes three quarters of its capacity, and at the end of the split, all warps take queue items two
// at a time and compute the exact fp32 score over the gathered key row (each lane's 8-element chunks in order,
// then a butterfly sum). The warp of each query then folds the scores that clear tau_c into that query's top-c
// list. A tile can admit more pairs than the queue has room for (up to 512 x 32, e.g. with radius = bits): a pair
// that finds the queue full stays in its thread's pending mask and is queued again after the next flush. The
// partial lists have the format of the other stage-1 kernels, so stage 2 is shared.
#include "internal.cuh"

namespace lc {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kTile = kThreads;     // entries per tile, one per thread
constexpr int kQC = 32;             // queries per pass over the entries (one bit each in a thread's masks)
constexpr int kCap = 8192;          // queue capacity
constexpr int kFlushAt = kCap - kCap / 4;   // a tile that leaves more items than this is followed by a flush
constexpr unsigned kFull = 0xffffffffu;

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

struct Shared {
  uint32_t qsig[kQC][16];
  uint64_t list[kQC][kMaxTopC];   // per query: sorted packed candidates of this split, 0 = empty
  unsigned int best[kQC];         // score_order of the best admitted score
  int count;                      // queued items
  Item items[kCap];
  float score[kCap];
};

// Exact scores of the queued items, then each query's warp folds its items into the query's list.
__device__ void flush(Shared& sh, const Stage1Args& a, int q0, int qn) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int total = min(sh.count, kCap);   // pairs that found the queue full were not stored
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

// Number of set bits in x[0..W). Population count runs at 16 per clock per SM, the logic operations at 64, so
// carry-save adders first fold words into sum and carry words, each group of 8 words into 5 popcounts (3 adders):
//   x0 + x1 + x2 = sa + 2 ca,  x3 + x4 + x5 = sb + 2 cb,  sa + sb + x6 = sc + 2 cc,
//   |x0..x7| = |sc| + |x7| + 2 (|ca| + |cb| + |cc|);
// a group of 4 words into 3 (one adder). The count is exact.
template <int W>
__device__ __forceinline__ int hamming(const uint32_t (&x)[W]) {
  int h = 0;
  if constexpr (W % 8 == 0) {
#pragma unroll
    for (int g = 0; g < W; g += 8) {
      uint32_t ca, sa, cb, sb, cc, sc;
      csa(ca, sa, x[g], x[g + 1], x[g + 2]);
      csa(cb, sb, x[g + 3], x[g + 4], x[g + 5]);
      csa(cc, sc, sa, sb, x[g + 6]);
      h += __popc(sc) + __popc(x[g + 7]) + 2 * (__popc(ca) + __popc(cb) + __popc(cc));
    }
  } else {
    static_assert(W % 4 == 0, "signature words come in groups of 4");
#pragma unroll
    for (int g = 0; g < W; g += 4) {
      uint32_t c, s;
      csa(c, s, x[g], x[g + 1], x[g + 2]);
      h += __popc(s) + __popc(x[g + 3]) + 2 * __popc(c);
    }
  }
  return h;
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

template <int W>
__global__ void __launch_bounds__(kThreads, 2) lsh_scan_kernel(Stage1Args a, LshArgs l, int splits) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  Shared& sh = *reinterpret_cast<Shared*>(smem_raw);
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int s = blockIdx.x;
  const int64_t j_begin = a.n * s / splits, j_end = a.n * (s + 1) / splits;
  const int C = a.top_c;
  for (int q0 = 0; q0 < a.B; q0 += kQC) {
    const int qn = min(kQC, a.B - q0);
    for (int i = threadIdx.x; i < kQC * W; i += kThreads) {
      const int qq = i / W;
      sh.qsig[qq][i % W] = qq < qn ? l.qsig[(int64_t)(q0 + qq) * W + i % W] : 0u;
    }
    for (int i = threadIdx.x; i < kQC * kMaxTopC; i += kThreads) sh.list[i / kMaxTopC][i % kMaxTopC] = 0;
    if (threadIdx.x < kQC) sh.best[threadIdx.x] = score_order(-INFINITY);
    if (threadIdx.x == 0) sh.count = 0;
    __syncthreads();
    // The next tile's signatures are loaded before the current tile is counted, so the load latency is hidden
    // behind the popcounts.
    uint32_t nxt[W];
    load_sig<W>(l.sig, j_begin + threadIdx.x, j_end, nxt);
    const unsigned qmask = qn >= 32 ? kFull : (1u << qn) - 1u;
    for (int64_t t0 = j_begin; t0 < j_end; t0 += kTile) {
      const int64_t j = t0 + threadIdx.x;
      uint32_t e[W];
#pragma unroll
      for (int w = 0; w < W; ++w) e[w] = nxt[w];
      load_sig<W>(l.sig, j + kTile, j_end, nxt);
      // every query's distance first, as a mask of the admitted queries (the queue stores below could alias the
      // query signatures for the compiler): whole groups of 8 queries unrolled, then the pass's remaining queries
      // (a uniform count), so a pass of one query computes one distance
      unsigned pend = 0;
      auto test_query = [&](int qq) {
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
        pend |= (hamming<W>(x) <= l.radius ? 1u : 0u) << qq;
      };
      const int whole = qn & ~7;
      for (int g = 0; g < whole; g += 8) {
#pragma unroll
        for (int u = 0; u < 8; ++u) test_query(g + u);
      }
      for (int qq = whole; qq < qn; ++qq) test_query(qq);
      pend = j < j_end ? pend & qmask : 0u;
      // Queue the admitted pairs; flush while the queue is past kFlushAt or a pair found it full. Every round of
      // this loop either queues all pending pairs or fills the queue, so it ends.
      int top = -1;   // the highest queue slot this thread took in this round
      for (;;) {
        unsigned full = 0;
        while (pend) {
          const int qq = __ffs(pend) - 1;
          pend &= pend - 1;
          const int slot = atomicAdd(&sh.count, 1);
          if (slot < kCap) {
            sh.items[slot] = Item{(int32_t)j, qq};
            top = slot;
          } else {
            full |= 1u << qq;
          }
        }
        pend = full;
        // the barrier's OR gives every thread the same answer (a read of the count after a plain barrier
        // could already see the next tile's items in some threads)
        if (!__syncthreads_or(pend != 0 || top >= kFlushAt)) break;
        flush(sh, a, q0, qn);
        top = -1;
      }
    }
    flush(sh, a, q0, qn);
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
template <int W>
cudaError_t launch_w(const Stage1Args& a, const LshArgs& l, int splits, cudaStream_t st) {
  const size_t smem = sizeof(Shared);
  cudaError_t e = cudaFuncSetAttribute(lsh_scan_kernel<W>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
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
  return cudaLaunchKernelEx(&cfg, lsh_scan_kernel<W>, a, l, splits);
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
                              int* splits) {
  const int64_t tiles = (a.n + kTile - 1) / kTile;
  int s = (int)(tiles < 2 * (int64_t)num_sms ? tiles : 2 * (int64_t)num_sms);
  if (s > max_splits) s = max_splits;
  if (s < 1) s = 1;
  *splits = s;
  switch (l.words) {   // 128, 256 or 512-bit signatures (16-byte loads)
    case 4: return launch_w<4>(a, l, s, st);
    case 8: return launch_w<8>(a, l, s, st);
    case 16: return launch_w<16>(a, l, s, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace lc

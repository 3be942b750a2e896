// The SimHash-indexed key check of larger batches on the tensor cores (Eq. 1; Algorithm 1's cache search): the
// Hamming test of every (query, entry) pair as one e4m3 GEMM over a pre-expanded index, then the exact key check
// of the admitted pairs. Same contract and outputs as the popcount scan in lsh.cu, which serves small batches.
//
// With signature bit 1 read as +1 and bit 0 as -1, the dot product of two b-bit signatures is
// (agreements - disagreements) = b - 2 hd, so hd <= radius iff dot >= b - 2 radius. Each term is +-1 and each sum
// an integer of at most 512 in magnitude, so an fp32 accumulation of e4m3 +-1 operands is exact.
//
// The index: every entry's signature as b e4m3 bytes (0x38 = +1, 0xB8 = -1), in blocks of 128 entries, each block
// already in the 128-byte swizzle layout the MMA reads ([128 rows x 128 B] per 128-bit atom of the signature;
// 16-byte chunk c of row r at (c ^ (r & 7)) * 16). expand_signatures_kernel writes it from the packed signatures
// whenever entries are signed, so one bulk copy moves a block from HBM into an operand stage.
//
// One CTA per contiguous range of blocks, warp-specialised:
//   warp 17 (loader): cp.async.bulk of one block per stage into a kS-deep ring;
//   warp 16 (MMA): allocates TMEM; per block issues tcgen05.mma.kind::f8f6f4 (M = 128 entries, N = the pass's
//     queries rounded up to 16, K = 32) over the resident query operand, into one of kNbuf accumulators;
//   warps 0-7 (mask warps; warp w reads TMEM lane quadrant w % 4 and the 32-query column chunks c with
//     c % 2 = w / 4): per block read each entry's dot products, and only where their maximum reaches the
//     threshold turn them into a mask of the admitted queries; release the accumulator; after every kRound blocks
//     queue the admitted (query, entry) pairs in shared memory, each slot stamped with the queue's epoch;
//   warps 8-15 (checker warps): claim queued pairs kItems at a time as they arrive, compute their exact fp32 key
//     scores over the gathered key rows (each lane's 8-element chunks in order, then a butterfly sum) while the
//     scan goes on, and fold each score into its query's best score and, if it clears tau_c, into the query's
//     top-c list (under a per-query lock).
// When the queue passes three quarters of its capacity, and at the end of the range, the mask warps close it: the
// checkers finish what was queued below the close, then the queue is emptied and reopened in a new epoch. A pair
// that finds the queue full stays in its thread's pending mask and is queued after the reopening. All sixteen
// epilogue warps expand the pass's query signatures into the query operand and write the lists out. The checker
// warps leave their loop only at a reopening, which the mask warps always run at the end of a pass, also after a
// timeout, so every named barrier sees all its warps.
// Queries are taken kQC at a time (one pass over the range each). Every mbarrier wait is bounded: on a timeout the
// CTA records LACACHE_ERR_DEVICE_TIMEOUT in the status word, the roles stop at the next pass boundary, in-flight
// copies and MMAs are drained, TMEM is freed and the CTA exits.
#include "internal.cuh"
#include "tcgen05.cuh"

namespace lc {
namespace {

constexpr int kMaskGroups = 2;                           // mask warps per TMEM lane quadrant
constexpr int kMaskWarps = 4 * kMaskGroups;              // warps 0-7: lane quadrant w % 4, group w / 4
constexpr int kCheckWarps = 8;                           // warps 8-15: exact checks of the queued pairs
constexpr int kEpiWarps = kMaskWarps + kCheckWarps;      // warps 0-15
constexpr int kMmaWarp = kEpiWarps;                      // warp 16
constexpr int kLoadWarp = kEpiWarps + 1;                 // warp 17
constexpr int kThreads = (kEpiWarps + 2) * 32;
constexpr int kCap = 1024;                               // queue capacity
constexpr int kFlushAt = kCap - kCap / 4;                // a round that leaves more items than this closes the queue
constexpr int kRound = 4;                                // blocks the mask warps take between their barriers
constexpr int kItems = 4;                                // queue items a checker warp claims at a time
constexpr int kBlockRows = 128;                          // entries per block and MMA (TMEM lanes)
constexpr int kAtomBytes = 128;                          // K bytes per swizzle atom (128 e4m3 values)
constexpr unsigned kFull = 0xffffffffu;

// Geometry per signature width: W = b / 32 words. A block is 128 entries x b bytes; kS blocks in flight; kQC
// queries per pass (the resident query operand is kQC * b bytes); kNbuf accumulators of kQC columns fill TMEM.
template <int W>
struct TcGeo {
  static constexpr int kBits = 32 * W;
  static constexpr int kAtoms = kBits / kAtomBytes;            // 1, 2 or 4
  static constexpr int kBlockBytes = kBlockRows * kBits;       // 16, 32 or 64 KB
  static constexpr int kS = W == 4 ? 6 : (W == 8 ? 4 : 2);
  static constexpr int kQC = W <= 8 ? 128 : 64;
  static constexpr int kQueryBytes = kQC * kBits;
  static constexpr int kNbuf = 512 / kQC;                      // 4 or 8
  static_assert(kNbuf * kQC == 512, "TMEM columns");
};
constexpr int kPer = (128 / 32 + kMaskGroups - 1) / kMaskGroups;   // column chunks per mask warp (at most)
static_assert(kEpiWarps * 32 >= 128, "the epilogue threads cover a pass's queries when they set up the lists");

struct Item {
  int32_t j;      // entry id
  int32_t q;      // query within the pass
};

// Shared memory after the operands: the queue, the per-query best scores and locks, flags and barriers; the
// per-query lists follow it.
struct Tail {
  Item items[kCap];
  uint32_t ready[kCap];        // the epoch (reopenings so far) whose item the slot holds, written after the item
  unsigned int best[128];      // score_order of the best admitted score, per query of the pass
  int lock[128];               // per query of the pass: its list is being updated
  int count;                   // queued items (may run past kCap: those pairs stay pending)
  int claim;                   // queue positions claimed by the checker warps
  int closed_at;               // while closing: min(count, kCap) when the queue was closed
  uint32_t closing;            // the mask warps closed the queue
  uint32_t pass_end;           // ... for the last time in the pass
  uint32_t abort_flag;
  uint32_t tmem_slot;
  uint32_t pad;
  uint64_t bars[32];           // full[kS], empty[kS], tfull[kNbuf], tempty[kNbuf], drain
};

template <int W>
constexpr size_t tc_smem_bytes(int top_c) {
  using G = TcGeo<W>;
  return 1024 + (size_t)G::kS * G::kBlockBytes + G::kQueryBytes + sizeof(Tail) + (size_t)G::kQC * top_c * 8;
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

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

// The mask warps' OR barrier (named barrier 1), and the barrier of all epilogue warps (named barrier 2).
__device__ __forceinline__ bool mask_any(bool p) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\t"
      "setp.ne.u32 pi, %1, 0;\n\t"
      "bar.red.or.pred po, 1, %2, pi;\n\t"
      "selp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)p), "n"(kMaskWarps * 32)
      : "memory");
  return r != 0;
}
__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync 2, %0;" ::"n"(kEpiWarps * 32) : "memory"); }

__device__ __forceinline__ uint32_t ld_volatile(const uint32_t* p) { return *reinterpret_cast<const volatile uint32_t*>(p); }
__device__ __forceinline__ void st_volatile(uint32_t* p, uint32_t v) { *reinterpret_cast<volatile uint32_t*>(p) = v; }

// Four signature bits (bit i = K index i) as four e4m3 bytes: +1 (0x38) for a set bit, -1 (0xB8) for a clear one.
// The complement's bit i lands on bit 8i + 7, the sign of byte i: 0x10204080 = 2^7 + 2^14 + 2^21 + 2^28, whose
// shifted copies of a 4-bit value do not overlap, so the product has no carries.
__device__ __forceinline__ uint32_t e4m3_signs(uint32_t nibble) {
  return (((~nibble & 0xFu) * 0x10204080u) & 0x80808080u) | 0x38383838u;
}

// The 16 e4m3 bytes of 16-byte chunk c of a signature: bits 16 (c & 1) .. 16 (c & 1) + 15 of word c / 2.
__device__ __forceinline__ uint4 e4m3_chunk(const uint32_t* words, int c) {
  const uint32_t half = (words[c / 2] >> (16 * (c & 1))) & 0xFFFFu;
  return make_uint4(e4m3_signs(half), e4m3_signs(half >> 4), e4m3_signs(half >> 8), e4m3_signs(half >> 12));
}

// Byte offset of chunk c of row r in a [rows x b] operand in the 128-byte swizzle layout: atom c / 8 is its own
// [rows x 128 B] block, and chunk c % 8 of row r sits at ((c % 8) ^ (r & 7)) * 16 within the row's 128-byte line.
__host__ __device__ __forceinline__ uint32_t swizzled_chunk(int rows, int r, int c) {
  return (uint32_t)(c / 8) * rows * kAtomBytes + (uint32_t)r * kAtomBytes + (uint32_t)(((c % 8) ^ (r & 7)) << 4);
}

// One thread per (entry, 16-byte chunk) of entries [first, first + n).
__global__ void expand_signatures_kernel(const uint32_t* __restrict__ sig, int64_t first, int64_t n, int words,
                                         uint8_t* __restrict__ index) {
  const int chunks = 2 * words;
  const int64_t total = n * chunks;
  const int64_t block_bytes = (int64_t)kBlockRows * 32 * words;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t j = first + i / chunks;
    const int c = (int)(i % chunks);
    const uint4 v = e4m3_chunk(sig + j * words, c);
    const int r = (int)(j % kBlockRows);
    *reinterpret_cast<uint4*>(index + (j / kBlockRows) * block_bytes + swizzled_chunk(kBlockRows, r, c)) = v;
  }
}

__device__ __forceinline__ void mma_e4m3(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}"
      ::"r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// A checker lane's wait for queue position `slot` of epoch ep: true once the item is there; false once the mask
// warps closed the queue at or below the slot (that position holds nothing to check in this epoch), or after about
// a second (the timeout is recorded; the mask warps then see the abort flag and close the queue).
__device__ __forceinline__ bool wait_slot(Tail& t, int slot, uint32_t ep, unsigned int* dev_status) {
  const long long t0 = clock64();
  for (;;) {
    if (slot < kCap && ld_volatile(&t.ready[slot]) == ep) {
      __threadfence_block();   // the item was written before its ready stamp
      return true;
    }
    if (ld_volatile(&t.closing)) {
      __threadfence_block();   // closed_at was written before closing
      if (slot >= (int)ld_volatile(reinterpret_cast<uint32_t*>(&t.closed_at))) return false;
      // below closed_at: the item was queued before the close and its stamp is on the way
    }
    if (clock64() - t0 > kWaitCycles) {
      st_volatile(&t.abort_flag, 1u);
      atomicOr(dev_status, kDevTimeout);
      return false;
    }
    __nanosleep(32);
  }
}

// A checker warp's exact key scores of the queue items at base + u for the set bits u of `ready`: kItems key rows
// in flight together, each lane's 8-element chunks in order, then a butterfly sum (every lane ends with every
// score).
__device__ __forceinline__ void check_items(const Tail& t, unsigned ready, int base, float (&acc)[kItems],
                                            const __nv_bfloat16* __restrict__ keys,
                                            const __nv_bfloat16* __restrict__ q, int d, int q0, int lane) {
  const int v = d / 8;
  const int first = base + __ffs(ready) - 1;
  const uint4* kp[kItems];
  const uint4* xp[kItems];
#pragma unroll
  for (int u = 0; u < kItems; ++u) {
    const Item it = t.items[(ready >> u) & 1u ? base + u : first];
    kp[u] = reinterpret_cast<const uint4*>(keys + (int64_t)it.j * d);
    xp[u] = reinterpret_cast<const uint4*>(q + (int64_t)(q0 + it.q) * d);
    acc[u] = 0.f;
  }
#pragma unroll 1
  for (int c = lane; c < v; c += 32) {
    uint4 kv[kItems], xv[kItems];
#pragma unroll
    for (int u = 0; u < kItems; ++u) {
      kv[u] = __ldg(kp[u] + c);
      xv[u] = __ldg(xp[u] + c);
    }
#pragma unroll
    for (int u = 0; u < kItems; ++u) acc[u] = dot8(xv[u], kv[u], acc[u]);
  }
#pragma unroll
  for (int u = 0; u < kItems; ++u) acc[u] = warp_sum(acc[u]);
}

// Fold one exact score into query qq's best score and, if it clears tau_c, into its top-c list (under the
// query's lock: several checker warps fold concurrently). False after a lock timeout (recorded).
__device__ __forceinline__ bool fold_one(Tail& t, uint64_t* lists, int C, float tau_c, int qq, int32_t j, float sc,
                                         unsigned int* dev_status) {
  atomicMax(&t.best[qq], score_order(sc));
  if (!(sc >= tau_c)) return true;
  const uint64_t x = pack_cand(sc, (uint32_t)j);
  const long long t0 = clock64();
  while (atomicCAS(&t.lock[qq], 0, 1) != 0) {
    if (clock64() - t0 > kWaitCycles || ld_volatile(&t.abort_flag)) {
      st_volatile(&t.abort_flag, 1u);
      atomicOr(dev_status, kDevTimeout);
      return false;
    }
    __nanosleep(32);
  }
  __threadfence_block();
  volatile uint64_t* L = lists + (size_t)qq * C;
  if (x > L[C - 1]) {
    int p = C - 1;
    while (p > 0 && L[p - 1] < x) {
      L[p] = L[p - 1];
      --p;
    }
    L[p] = x;
  }
  __threadfence_block();
  atomicExch(&t.lock[qq], 0);
  return true;
}

// Run by all epilogue warps after the mask warps closed the queue: once every checker has arrived, every queued
// pair has been checked and folded into its query's list; then the queue is emptied and reopened.
__device__ __forceinline__ void reopen(Tail& t, int ew, int lane) {
  epi_sync();
  if (ew == 0 && lane == 0) {
    t.count = 0;
    t.claim = 0;
    t.closing = 0;
  }
  epi_sync();
}

template <int W>
__global__ void __launch_bounds__(kThreads, 1) lsh_tc_kernel(Stage1Args a, LshArgs l, int splits) {
  using G = TcGeo<W>;
  extern __shared__ unsigned char smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  unsigned char* gbase = smem_raw + (base - raw);
  const uint32_t a_smem = base;                                      // kS index blocks
  const uint32_t q_smem = a_smem + G::kS * G::kBlockBytes;           // kQC query rows
  Tail& t = *reinterpret_cast<Tail*>(gbase + (size_t)G::kS * G::kBlockBytes + G::kQueryBytes);
  uint64_t* lists = reinterpret_cast<uint64_t*>(&t + 1);            // [kQC][top_c]
  volatile uint32_t* abort_flag = &t.abort_flag;
  const uint32_t bar0 = smem_u32(t.bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (G::kS + s); };
  auto tfull_bar = [&](int b) { return bar0 + 8u * (2 * G::kS + b); };
  auto tempty_bar = [&](int b) { return bar0 + 8u * (2 * G::kS + G::kNbuf + b); };
  const uint32_t drain_bar = bar0 + 8u * (2 * G::kS + 2 * G::kNbuf);
  static_assert(2 * G::kS + 2 * G::kNbuf + 1 <= 32, "barrier slots");

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < G::kS; ++s) {
      mbar_init(full_bar(s), 1);     // the loader's arrive, with the copy's bytes
      mbar_init(empty_bar(s), 1);    // the MMA commit
    }
    for (int b = 0; b < G::kNbuf; ++b) {
      mbar_init(tfull_bar(b), 1);
      mbar_init(tempty_bar(b), kMaskWarps);
    }
    mbar_init(drain_bar, 1);
    t.abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  for (int i = threadIdx.x; i < kCap; i += kThreads) t.ready[i] = ~0u;   // no epoch
  if (warp == kMmaWarp) {
    tmem_alloc<false>(smem_u32(&t.tmem_slot), 512);
    tmem_relinquish<false>();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = t.tmem_slot;
  // the query signatures are the previous kernel's output
  asm volatile("griddepcontrol.wait;" ::: "memory");

  auto fail = [&]() {
    *abort_flag = 1u;
    atomicOr(a.dev_status, kDevTimeout);
  };

  const int s = blockIdx.x;
  const int64_t nblocks = (a.n + kBlockRows - 1) / kBlockRows;
  const int64_t g_begin = nblocks * s / splits, g_end = nblocks * (s + 1) / splits;
  const int64_t j_end = min(a.n, g_end * kBlockRows);
  const int64_t nb = g_end - g_begin;
  const int C = a.top_c;
  const float thr = (float)(G::kBits - 2 * l.radius);   // admitted iff dot >= b - 2 radius
  uint32_t it = 0;        // blocks so far, over all passes (every role counts the same blocks)
  uint32_t tb = 0;        // accumulator uses so far
  uint32_t issued = 0;    // loader: copies issued, blocks 0 .. issued - 1
  uint32_t ep = 0;        // epilogue: reopenings so far (the epoch of the queue's ready stamps)

  for (int q0 = 0; q0 < a.B; q0 += G::kQC) {
    const int qn = min(G::kQC, a.B - q0);
    const int npad = max(16, (qn + 15) / 16 * 16);
    // ---- pass set-up (epilogue warps): the resident query operand, the lists and counters ----
    if (warp < kEpiWarps) {
      const int et = threadIdx.x;
      for (int r = et; r < G::kQC; r += kEpiWarps * 32) {
        uint32_t w[W];
        const bool valid = r < qn;
#pragma unroll
        for (int i = 0; i < W; ++i) w[i] = valid ? l.qsig[(int64_t)(q0 + r) * W + i] : 0u;
#pragma unroll
        for (int c = 0; c < 2 * W; ++c) {
          const uint4 v = valid ? e4m3_chunk(w, c) : make_uint4(0, 0, 0, 0);
          const uint32_t addr = q_smem + swizzled_chunk(G::kQC, r, c);
          asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z),
                       "r"(v.w)
                       : "memory");
        }
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      for (int i = et; i < G::kQC * C; i += kEpiWarps * 32) lists[i] = 0;
      for (int i = et; i < G::kQC; i += kEpiWarps * 32) {
        t.best[i] = score_order(-INFINITY);
        t.lock[i] = 0;
      }
      if (et == 0) {
        t.count = 0;
        t.claim = 0;
        t.closing = 0;
        t.pass_end = 0;
      }
    }
    __syncthreads();

    if (warp == kLoadWarp) {
      // ---------------- loader ----------------
      if (lane == 0) {
        for (int64_t ti = 0; ti < nb; ++ti) {
          const uint32_t k = it + (uint32_t)ti;
          const int st = k % G::kS;
          if (!mbar_wait(empty_bar(st), ((k / G::kS) & 1u) ^ 1u, abort_flag)) {
            fail();
            break;
          }
          mbar_expect_tx(full_bar(st), G::kBlockBytes);
          asm volatile(
              "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
              ::"r"(a_smem + (uint32_t)st * G::kBlockBytes),
              "l"(l.index + (g_begin + ti) * (int64_t)G::kBlockBytes), "r"((uint32_t)G::kBlockBytes),
              "r"(full_bar(st))
              : "memory");
          issued = k + 1;
        }
      }
      __syncwarp();
      it += (uint32_t)nb;
    } else if (warp == kMmaWarp) {
      // ---------------- MMA issue ----------------
      if (lane == 0) {
        // kind::f8f6f4: D f32 (bits 4-5 = 1), A and B e4m3 (bits 7-9, 10-12 = 0), both K-major, N >> 3 in bits
        // 17-22, M >> 4 in bits 24-28
        const uint32_t idesc = (1u << 4) | ((uint32_t)(npad >> 3) << 17) | ((uint32_t)(kBlockRows >> 4) << 24);
        for (int64_t ti = 0; ti < nb; ++ti) {
          const uint32_t k = it + (uint32_t)ti;
          const int st = k % G::kS;
          const int b = tb % G::kNbuf;
          const uint32_t tph = (tb / G::kNbuf) & 1u;
          ++tb;
          if (!mbar_wait(tempty_bar(b), tph ^ 1u, abort_flag) || !mbar_wait(full_bar(st), (k / G::kS) & 1u,
                                                                             abort_flag)) {
            fail();
            break;
          }
          tc_fence_after();
          const uint32_t blk = a_smem + (uint32_t)st * G::kBlockBytes;
          const uint32_t d = tmem + (uint32_t)(b * G::kQC);
#pragma unroll
          for (int at = 0; at < G::kAtoms; ++at)
#pragma unroll
            for (int ks = 0; ks < kAtomBytes / 32; ++ks)
              mma_e4m3(d, smem_desc(blk + (uint32_t)at * kBlockRows * kAtomBytes + 32u * ks),
                       smem_desc(q_smem + (uint32_t)at * G::kQC * kAtomBytes + 32u * ks), idesc,
                       (at | ks) != 0 ? 1u : 0u);
          mma_commit<false>(empty_bar(st), 0);
          mma_commit<false>(tfull_bar(b), 0);
        }
      }
      __syncwarp();
      tb = __shfl_sync(kFull, tb, 0);
      it += (uint32_t)nb;
    } else if (warp < kMaskWarps) {
      // ---------------- mask warps ----------------
      const int mw = warp;                                 // mask warp
      const int quad = mw % 4, group = mw / 4;             // TMEM lane quadrant; column chunks c % kMaskGroups == group
      const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
      // close the queue (every mask warp has queued its pairs); reopen it once the checkers are done with it
      auto close_and_reopen = [&](bool last) {
        if (mw == 0 && lane == 0) {
          t.closed_at = min(t.count, kCap);
          if (last) t.pass_end = 1;
          __threadfence_block();
          st_volatile(&t.closing, 1u);
        }
        reopen(t, mw, lane);
        ++ep;
      };
      bool stop = false;
      for (int64_t t0 = 0; t0 < nb && !stop; t0 += kRound) {
        // the admitted queries of this thread's entry in each block of the round, as bit masks over the warp's
        // column chunks (chunk group + kMaskGroups u)
        uint32_t pend[kRound][kPer];
        bool got = true;
#pragma unroll
        for (int r = 0; r < kRound; ++r) {
#pragma unroll
          for (int u = 0; u < kPer; ++u) pend[r][u] = 0;
          if (t0 + r >= nb || !got) continue;              // the same for every mask warp
          const int b = tb % G::kNbuf;
          const uint32_t tph = (tb / G::kNbuf) & 1u;
          ++tb;
          got = __all_sync(kFull, mbar_wait(tfull_bar(b), tph, abort_flag));
          if (!got) continue;   // the warp-collective loads below need the whole warp
          tc_fence_after();
#pragma unroll
          for (int u = 0; u < kPer; ++u) {
            const int c = group + kMaskGroups * u;
            if (c < G::kQC / 32 && 32 * c < npad) {   // the same for the whole warp
              float v[32];
              tmem_ld32(tmem + lane_addr + (uint32_t)(b * G::kQC) + 32u * c, v);
              // admitted pairs are rare: a max over the 32 scores decides whether the mask is built at all
              float m[16];
#pragma unroll
              for (int i = 0; i < 16; ++i) m[i] = fmaxf(v[i], v[i + 16]);
#pragma unroll
              for (int w = 8; w > 0; w >>= 1)
#pragma unroll
                for (int i = 0; i < w; ++i) m[i] = fmaxf(m[i], m[i + w]);
              if (m[0] >= thr) {
                uint32_t mask = 0;
#pragma unroll
                for (int i = 0; i < 32; ++i) mask |= (v[i] >= thr ? 1u : 0u) << i;
                const int left = qn - 32 * c;
                pend[r][u] = left >= 32 ? mask : (left > 0 ? mask & ((1u << left) - 1u) : 0u);
              }
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(tempty_bar(b));
        }
        // queue the admitted pairs, each with its epoch stamp, for the checker warps; close while the queue is
        // past kFlushAt or a pair found it full (every round either queues all pending pairs or fills the queue,
        // so this ends). All mask warps leave together.
        int top = -1;
        for (;;) {
          bool left = false;
#pragma unroll
          for (int r = 0; r < kRound; ++r) {
            const int64_t j = (g_begin + t0 + r) * kBlockRows + quad * 32 + lane;
            const bool valid = got && j < j_end;
#pragma unroll
            for (int u = 0; u < kPer; ++u) {
              uint32_t p = valid ? pend[r][u] : 0u;
              uint32_t full = 0;
              while (p) {
                const int bit = __ffs(p) - 1;
                p &= p - 1;
                const int slot = atomicAdd(&t.count, 1);
                if (slot < kCap) {
                  t.items[slot] = Item{(int32_t)j, 32 * (group + kMaskGroups * u) + bit};
                  __threadfence_block();
                  st_volatile(&t.ready[slot], ep);
                  top = slot;
                } else {
                  full |= 1u << bit;
                }
              }
              pend[r][u] = full;
              left |= full != 0;
            }
          }
          if (!mask_any(!got || *abort_flag || left || top >= kFlushAt)) break;
          if (mask_any(!got || *abort_flag)) {
            if (!got) fail();
            stop = true;
            break;
          }
          close_and_reopen(false);
          top = -1;
        }
      }
      // the pass's last close, also after a timeout: the checker warps leave only at a reopening
      close_and_reopen(true);
      it += (uint32_t)nb;
    } else {
      // ---------------- checker warps ----------------
      // claim kItems queue positions at a time, check and fold their pairs while the scan goes on; at a close,
      // finish what was queued below it, then take part in the reopening
      for (;;) {
        for (;;) {
          int base = 0;
          if (lane == 0) base = atomicAdd(&t.claim, kItems);
          base = __shfl_sync(kFull, base, 0);
          const bool mine = lane < kItems && wait_slot(t, base + lane, ep, a.dev_status);
          const unsigned ready = __ballot_sync(kFull, mine);
          if (ready) {
            float acc[kItems];
            check_items(t, ready, base, acc, a.keys, a.q, a.d, q0, lane);
            if (lane == 0) {
#pragma unroll
              for (int u = 0; u < kItems; ++u)
                if ((ready >> u) & 1u)
                  fold_one(t, lists, C, a.tau_c, t.items[base + u].q, t.items[base + u].j, acc[u], a.dev_status);
            }
            __syncwarp();
          }
          if (ready != (1u << kItems) - 1u) break;   // a position past the close (or a timeout)
        }
        reopen(t, warp, lane);
        ++ep;
        if (ld_volatile(&t.pass_end)) break;
      }
      it += (uint32_t)nb;
    }

    // ---- pass end: every role is here; a timeout anywhere stops them all together ----
    if (__syncthreads_or(*abort_flag != 0)) break;
    if (warp < kEpiWarps) {
      const int et = threadIdx.x;
      // the lists' candidates (a sorted list holds them in its first slots, then zeros) and each list's record
      for (int i = et; i < qn * C; i += kEpiWarps * 32) {
        const int qq = i / C;
        if (lists[i]) a.part_cand[((int64_t)s * a.B + q0 + qq) * C + (i - qq * C)] = lists[i];
      }
      for (int i = et; i < qn; i += kEpiWarps * 32) {
        uint32_t count = 0;
        while ((int)count < C && lists[(size_t)i * C + count]) ++count;
        a.part_meta[(int64_t)s * a.B + q0 + i] = PartMeta{score_of_order(t.best[i]), count};
      }
    }
    __syncthreads();
  }

  // nothing in flight when the CTA exits: the loader waits for its last kS copies (a consumed one passes at
  // once), the MMA issuer for every MMA; then TMEM is freed
  if (warp == kLoadWarp && lane == 0) {
    for (uint32_t k = issued >= (uint32_t)G::kS ? issued - G::kS : 0u; k < issued; ++k)
      mbar_wait(full_bar(k % G::kS), (k / G::kS) & 1u, nullptr);
  }
  if (warp == kMmaWarp && lane == 0) {
    mma_commit<false>(drain_bar, 0);
    mbar_wait(drain_bar, 0, nullptr);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kMmaWarp) tmem_dealloc<false>(tmem, 512);
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// A programmatic dependent launch of the query-signature GEMM: the CTAs may be scheduled while the signatures are
// computed and wait in griddepcontrol.wait.
template <int W>
cudaError_t launch_w(const Stage1Args& a, const LshArgs& l, int splits, cudaStream_t st) {
  const size_t smem = tc_smem_bytes<W>(a.top_c);
  cudaError_t e = cudaFuncSetAttribute(lsh_tc_kernel<W>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
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
  return cudaLaunchKernelEx(&cfg, lsh_tc_kernel<W>, a, l, splits);
}

static_assert(tc_smem_bytes<4>(kMaxTopC) <= 227 * 1024 && tc_smem_bytes<8>(kMaxTopC) <= 227 * 1024 &&
                  tc_smem_bytes<16>(kMaxTopC) <= 227 * 1024,
              "shared memory budget");

}  // namespace

size_t lsh_index_bytes(int64_t capacity, int bits) {
  return (size_t)((capacity + kBlockRows - 1) / kBlockRows) * kBlockRows * bits;
}

cudaError_t launch_expand_signatures(const uint32_t* sig, int64_t first, int64_t n, int bits, uint8_t* index,
                                     int num_sms, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  const int64_t total = n * (bits / 16);
  const int64_t want = (total + 255) / 256;
  const int blocks = (int)(want < (int64_t)num_sms * 8 ? want : (int64_t)num_sms * 8);
  expand_signatures_kernel<<<blocks, 256, 0, st>>>(sig, first, n, bits / 32, index);
  return cudaGetLastError();
}

cudaError_t launch_stage1_lsh_tc(const Stage1Args& a, const LshArgs& l, int num_sms, int max_splits,
                                 cudaStream_t st, int* splits) {
  const int64_t blocks = (a.n + kBlockRows - 1) / kBlockRows;
  int s = (int)(blocks < (int64_t)num_sms ? blocks : (int64_t)num_sms);
  if (s > max_splits) s = max_splits;
  if (s < 1) s = 1;
  *splits = s;
  switch (l.words) {   // 128, 256 or 512-bit signatures
    case 4: return launch_w<4>(a, l, s, st);
    case 8: return launch_w<8>(a, l, s, st);
    case 16: return launch_w<16>(a, l, s, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace lc

// Stage 1 on the tensor cores: the key check sim(x, x') >= tau_c (Algorithm 1's cache search; section 4.1) as a
// tcgen05 GEMM of the query tile against the key store, fused with the threshold and a per-query running
// top_c. The B x N score matrix never leaves the SM.
//
//   D[m][n] = sum_k Q[qt*128 + m][k] * K[t*256 + n][k]      (bf16 operands, fp32 accumulation in TMEM)
//
// Layout of the work. One query tile (B <= 128): a dynamic schedule, in which CTAs claim 256-key tiles from a
// global counter (one split per CTA), which balances the tail. Several query tiles: units are (query tile of
// 128, split of the key tiles), walked by a persistent grid with the query tile varying fastest, so the CTAs that
// run at the same time stream the same key range and share it through L2; more than one query tile runs on CTA
// pairs (below). Each CTA:
//   warp 0      TMA producer: per k-step, one 128x64 query box and one 256x64 key box (128-byte swizzle) into a
//               4-stage shared-memory ring (mbarrier full/empty pairs);
//   warp 1      MMA issuer: allocates 512 TMEM columns (two 128x256 fp32 accumulators) and issues
//               tcgen05.mma kind::f16 (M=128, N=256, K=16) from one thread; tcgen05.commit frees ring stages
//               and hands a finished accumulator to the epilogue;
//   warps 2..5  epilogue: thread = query row (TMEM lane); reads its 256 scores with tcgen05.ld, keeps a sorted
//               top_c of (score, id) in registers with the threshold max(tau_c, current c-th best), and finally
//               writes the unit's partial list. Double-buffered accumulators overlap it with the next tile's MMAs.
// Batches of more than one query tile run as CTA pairs (a two-CTA cluster on the two SMs of a TPC): one
// tcgen05.mma.cta_group::2 of M=256 (two query tiles, one per SM), N=256, K=16 per step. Each SM loads its own
// 128x64 query box and HALF of the key box (128 keys); the pair's tensor cores exchange the key halves, and each
// SM's TMEM receives its own 128 query rows x 256 keys. Per SM and k-step that is 32 KB of TMA writes and of MMA
// operand reads instead of 48 KB, and each key tile is read once per pair of query tiles. The leader CTA (rank 0)
// issues the MMAs; both CTAs' loads complete on the leader's full barrier, its commits arrive on both CTAs'
// empty and tmem_full barriers, and both CTAs' epilogues release an accumulator on the leader's tmem_empty.
// Every mbarrier wait is bounded: on a timeout the CTA records LACACHE_ERR_DEVICE_TIMEOUT in the status word, the
// other roles see an abort flag and stop, in-flight copies and MMAs are drained, TMEM is freed and the CTA exits.
#include <cuda.h>
#include <string.h>

#include <atomic>

#include "internal.cuh"
#include "tcgen05.cuh"

namespace lc {
namespace {

constexpr int BM = 128;                     // queries per tile (TMEM lanes)
constexpr int BN = 256;                     // keys per tile (accumulator columns)
constexpr int BK = 64;                      // bf16 per k-step = one 128-byte swizzled row
constexpr int A_BYTES = BM * BK * 2;        // 16 KB
constexpr int TMEM_COLS = 2 * BN;           // two accumulators
constexpr int kThreads = 192;
constexpr int kEpiWarps = 4;
constexpr int RING = 4;                             // tile-index ring of the dynamic schedule
constexpr size_t kStashBytes = 32 * 129 * 4;          // epilogue's rare-path chunk stash
constexpr int kMaxDeviceSlots = 64;                   // devices whose CTA-pair capacity is cached
constexpr int64_t kPairSplitBytes = (int64_t)11 << 20;  // keys per split of the CTA-pair schedule (L2 reuse)

// Per-CTA geometry. Single CTA: the whole 256-key box per stage, 4 stages. CTA pair: half the key box, so 6
// stages fit in the same shared memory.
template <bool PAIR>
struct Geo {
  static constexpr int kStages = PAIR ? 6 : 4;
  static constexpr int kBRows = PAIR ? BN / 2 : BN;        // key rows this CTA loads per tile
  static constexpr int kBBytes = kBRows * BK * 2;
  static constexpr int kStageBytes = A_BYTES + kBBytes;
  // full, empty, tmem_full x2, tmem_empty x2, drain, ring full/empty
  static constexpr int kBarriers = 2 * kStages + 5 + 2 * RING;
  static constexpr size_t kSmem = 1024 + (size_t)kStages * kStageBytes + kBarriers * 8 + 16 + RING * 4 + kStashBytes;
  // tcgen05 instruction descriptor, kind::f16: D f32 (bits 4-5 = 1), A bf16 (bits 7-9 = 1), B bf16 (bits 10-12
  // = 1), A and B K-major (bits 15, 16 = 0), N >> 3 in bits 17-22, M >> 4 in bits 24-28 (M = 256 for the pair).
  static constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                                     ((uint32_t)((PAIR ? 2 * BM : BM) >> 4) << 24);
};
static_assert(Geo<false>::kSmem <= 227 * 1024 && Geo<true>::kSmem <= 227 * 1024, "shared memory budget");

struct TcParams {
  int64_t n;
  int d;
  int B;
  float tau_c;
  int top_c;
  int q_tiles;
  int pairs;      // CTA-pair schedule: query-tile pairs (ceil(q_tiles / 2)); units are (pair, split)
  int splits;
  int units;
  int64_t n_tiles;
  int k_steps;
  int a_rows;     // rows of the query box: B rounded up to 8 when B <= 128, else 128
  int inject_stall;  // test support: CTA 0 withholds its second load, so its MMA issuer's bounded wait runs out
  int* tile_ctr;      // dynamic schedule: [next tile, CTAs done], zero at launch and left zero (nullptr: static)
  int wait_first;     // wait for the preceding grids before reading anything (they write the queries)
  uint32_t* sig;     // signature mode: [n x sig_words] output words
  int sig_words;
  uint64_t* part_cand;
  PartMeta* part_meta;
  unsigned int* dev_status;
};

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
// CTA-pair form: the destination is this CTA's shared memory, the mbarrier may be the peer's (the leader's).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3}], [%4];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_id_x() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_count_x() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
  return r;
}
// Address of the same shared-memory variable in the cluster CTA of the given rank.
__device__ __forceinline__ uint32_t map_to_rank(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
}
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

template <bool PAIR>
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t accumulate) {
  if constexpr (PAIR)
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(Geo<true>::kIdesc), "r"(accumulate)
        : "memory");
  else
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(Geo<false>::kIdesc), "r"(accumulate)
        : "memory");
}
// Running top_c of one query: scores descending; among equal scores the earlier (lower) id first, which holds
// because ids arrive in increasing order. Slots past top_c are kept but never read.
template <int CPAD>
struct TopC {
  float s[CPAD];
  uint32_t j[CPAD];
  int count;
  float thr;  // a new candidate enters iff score >= thr

  __device__ __forceinline__ void init(float tau_c) {
#pragma unroll
    for (int i = 0; i < CPAD; ++i) {
      s[i] = -INFINITY;
      j[i] = 0xFFFFFFFFu;
    }
    count = 0;
    thr = tau_c;
  }
  __device__ __forceinline__ void insert(float v, uint32_t id, int c) {
#pragma unroll
    for (int i = 0; i < CPAD; ++i) {
      if (v > s[i]) {
        const float ts = s[i];
        const uint32_t tj = j[i];
        s[i] = v;
        j[i] = id;
        v = ts;
        id = tj;
      }
    }
    if (count < c) ++count;
    if (count >= c) {
      // the c-th best is the minimum of the first c (sorted) slots; written as a masked min so that it stays a
      // register computation rather than a dynamically indexed (local-memory) read of s[c - 1]
      float w = INFINITY;
#pragma unroll
      for (int i = 0; i < CPAD; ++i) w = fminf(w, i < c ? s[i] : INFINITY);
      thr = fmaxf(thr, nextafterf(w, INFINITY));   // equal scores arrive with larger ids: they lose
    }
  }
};

// SIGN = false: the key check (threshold + top-c partial lists). SIGN = true: the same GEMM with random hyperplanes
// in place of the queries, and an epilogue that writes SimHash signatures: bit h of row j's signature is set iff
// <r_h, row_j> >= 0; each warp's 32 hyperplanes form one 32-bit word, packed with a ballot per key column.
// PAIR = true: launched as two-CTA clusters, static schedule over (query-tile pair, split) units.
template <int CPAD, bool SIGN, bool PAIR>
__global__ void __launch_bounds__(kThreads, 1)
    stage1_tensor_kernel(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
                         const TcParams p) {
  using G = Geo<PAIR>;
  constexpr int S = G::kStages;
  extern __shared__ unsigned char smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  unsigned char* gbase = smem_raw + (base - raw);
  const uint32_t a_smem = base;
  const uint32_t b_smem = base + S * A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(gbase + (size_t)S * G::kStageBytes);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + G::kBarriers);
  volatile int* tid_ring = reinterpret_cast<volatile int*>(tmem_slot + 4);
  float* stash = reinterpret_cast<float*>(tmem_slot + 4 + RING);
  volatile uint32_t* abort_flag = tmem_slot + 1;
  const uint32_t bar0 = smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (S + s); };
  auto tfull_bar = [&](int b) { return bar0 + 8u * (2 * S + b); };
  auto tempty_bar = [&](int b) { return bar0 + 8u * (2 * S + 2 + b); };
  const uint32_t drain_bar = bar0 + 8u * (2 * S + 4);
  auto tid_full_bar = [&](int r) { return bar0 + 8u * (2 * S + 5 + r); };
  auto tid_empty_bar = [&](int r) { return bar0 + 8u * (2 * S + 5 + RING + r); };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = PAIR ? cluster_rank() : 0u;   // 0: leader (issues the MMAs)

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full_bar(s), 1);    // the (leader's) producer's arrive; both CTAs' bytes complete it
      mbar_init(empty_bar(s), 1);   // the (leader's) MMA commit
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull_bar(b), 1);
      mbar_init(tempty_bar(b), (PAIR ? 2 : 1) * kEpiWarps);   // the epilogue warps of both CTAs of a pair
    }
    mbar_init(drain_bar, 1);
    for (int r = 0; r < RING; ++r) {
      mbar_init(tid_full_bar(r), 1);
      mbar_init(tid_empty_bar(r), 1 + kEpiWarps);   // the MMA issuer and the four epilogue warps
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmap_q);
    tma_prefetch_desc(&tmap_k);
  }
  // A pair: both CTAs' barriers are initialised, and both CTAs are running, before either touches the other's
  // shared memory or allocates the pair's TMEM.
  if constexpr (PAIR) cluster_sync();
  if (warp == 1) {
    tmem_alloc<PAIR>(smem_u32(tmem_slot), TMEM_COLS);
    tmem_relinquish<PAIR>();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // Launched as a programmatic dependent of the previous lookup's stage 2. That grid reads the partial lists
  // this one writes, and writes nothing this one reads, so the scan runs alongside it: each epilogue thread waits
  // for the preceding grids (griddepcontrol.wait) only before its first global write. Inputs written by earlier
  // work on the stream are complete, because those kernels let their dependents start only when they finish. The
  // one exception, the host-input gather, writes the queries and starts its dependent early: then every thread
  // waits here, before reading anything. This lookup's stage 2 may be scheduled now; it waits for this grid's
  // completion before reading anything.
  if (p.wait_first) asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  auto fail = [&]() {
    *abort_flag = 1u;
    if constexpr (PAIR) {   // the peer stops too
      const uint32_t peer = map_to_rank(smem_u32((const void*)abort_flag), rank ^ 1u);
      asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(peer), "r"(1u) : "memory");
    }
    atomicOr(p.dev_status, kDevTimeout);
  };

  // Dynamic schedule (one query tile): the producer claims key tiles from a global counter and hands their
  // indices to the MMA issuer and the epilogue through a small ring; a CTA's claims increase, so ids still arrive
  // in increasing order. Static schedule: units (query tile, split of the key tiles) in a fixed order; for a
  // pair, units (pair of query tiles, split) and this CTA takes the pair's tile of its rank.
  const bool dyn = !PAIR && p.tile_ctr != nullptr;
  const int unit0 = PAIR ? (int)cluster_id_x() : (int)blockIdx.x;
  const int ustep = PAIR ? (int)cluster_count_x() : (int)gridDim.x;
  const int per_split = PAIR ? p.pairs : p.q_tiles;
  auto unit_qt = [&](int u) { return PAIR ? 2 * (u % p.pairs) + (int)rank : u % p.q_tiles; };

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      uint32_t it = 0;
      bool ok = true;
      const uint32_t withheld = (p.inject_stall && blockIdx.x == 0) ? 1u : 0xFFFFFFFFu;
      auto load_tile = [&](int qt, int64_t t) -> bool {
        for (int ks = 0; ks < p.k_steps; ++ks, ++it) {
          const int s = it % S;
          const uint32_t ph = (it / S) & 1u;
          if (!mbar_wait(empty_bar(s), ph ^ 1u, abort_flag)) {
            fail();
            return false;
          }
          if (it == withheld) continue;   // nothing arrives on this stage: its consumer's wait runs out
          if constexpr (PAIR) {
            // both CTAs' boxes complete the leader's full barrier, which expects the bytes of all four. A box
            // that would lie wholly out of bounds (the odd query tile's partner, the upper half of a last key
            // tile of at most 128 keys) is replaced by the leader's box: the epilogue never reads those rows
            // (queries >= B) or columns (ids >= n).
            const uint32_t lead_full = map_to_rank(full_bar(s), 0);
            if (rank == 0) mbar_expect_tx(full_bar(s), (uint32_t)(2 * G::kStageBytes));
            const int qy = (qt < p.q_tiles ? qt : qt - 1) * BM;
            const int64_t ky = t * BN + (int64_t)rank * G::kBRows;
            tma_load_2d_pair(a_smem + s * A_BYTES, &tmap_q, lead_full, ks * BK, qy);
            tma_load_2d_pair(b_smem + s * G::kBBytes, &tmap_k, lead_full, ks * BK, (int)(ky < p.n ? ky : t * BN));
          } else {
            mbar_expect_tx(full_bar(s), (uint32_t)(p.a_rows * BK * 2 + G::kBBytes));
            tma_load_2d(a_smem + s * A_BYTES, &tmap_q, full_bar(s), ks * BK, qt * BM);
            tma_load_2d(b_smem + s * G::kBBytes, &tmap_k, full_bar(s), ks * BK, (int)(t * BN));
          }
        }
        return true;
      };
      if (dyn) {
        int64_t next = atomicAdd(p.tile_ctr, 1);
        for (uint32_t r = 0; ok; ++r) {
          const int64_t t = next;
          const bool done = t >= p.n_tiles;
          if (!done) next = atomicAdd(p.tile_ctr, 1);   // claim one ahead: hides the atomic's latency
          const int slot = r % RING;
          if (!mbar_wait(tid_empty_bar(slot), ((r / RING) & 1u) ^ 1u, abort_flag)) {
            fail();
            break;
          }
          tid_ring[slot] = done ? -1 : (int)t;
          mbar_arrive(tid_full_bar(slot));               // release: the index is visible to its readers
          if (done) break;
          ok = load_tile(0, t);
        }
        // This CTA has made its last claim. The last CTA of the launch to get here zeroes both counters, so the
        // next launch (which reads them only after this grid has completed) starts from zero: the schedule keeps
        // no state on the host, and a lookup captured in a CUDA graph replays correctly.
        __threadfence();
        if (atomicAdd(p.tile_ctr + 1, 1) == (int)gridDim.x - 1) {
          p.tile_ctr[0] = 0;
          p.tile_ctr[1] = 0;
        }
      } else {
        for (int u = unit0; ok && u < p.units; u += ustep) {
          const int qt = unit_qt(u), sp = u / per_split;
          const int64_t t_begin = p.n_tiles * sp / p.splits, t_end = p.n_tiles * (sp + 1) / p.splits;
          for (int64_t t = t_begin; ok && t < t_end; ++t) ok = load_tile(qt, t);
        }
      }
      // drain: the last load issued into each stage has landed before the CTA may exit. A pair's loads complete
      // on the leader's barrier, so the peer waits instead for the MMA commits that free its stages (each
      // follows the MMAs that read them, which waited for the data).
      const uint32_t first = it > (uint32_t)S ? it - S : 0u;
      for (uint32_t i = first; i < it; ++i) {
        if (i == withheld) continue;
        const bool landed = (PAIR && rank != 0) ? mbar_wait(empty_bar(i % S), (i / S) & 1u, nullptr)
                                                : mbar_wait(full_bar(i % S), (i / S) & 1u, nullptr);
        if (!landed) {
          fail();
          break;
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // ---------------- MMA issuer ----------------
      uint32_t it = 0, tile_i = 0;
      bool ok = true;
      auto mma_tile = [&]() -> bool {
        const int b = tile_i & 1u;
        if (!mbar_wait(tempty_bar(b), ((tile_i >> 1) & 1u) ^ 1u, abort_flag)) {
          fail();
          return false;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem + (uint32_t)(b * BN);
        for (int ks = 0; ks < p.k_steps; ++ks, ++it) {
          const int s = it % S;
          if (!mbar_wait(full_bar(s), (it / S) & 1u, abort_flag)) {
            fail();
            return false;
          }
          tc_fence_after();
          const uint64_t ad = smem_desc(a_smem + s * A_BYTES);
          const uint64_t bd = smem_desc(b_smem + s * G::kBBytes);
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            mma_bf16<PAIR>(d_tmem, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), (ks | kk) != 0 ? 1u : 0u);
          mma_commit<PAIR>(empty_bar(s), 3);
        }
        mma_commit<PAIR>(tfull_bar(b), 3);
        ++tile_i;
        return true;
      };
      if (dyn) {
        for (uint32_t r = 0; ok; ++r) {
          const int slot = r % RING;
          if (!mbar_wait(tid_full_bar(slot), (r / RING) & 1u, abort_flag)) {
            fail();
            break;
          }
          const int t = tid_ring[slot];
          mbar_arrive(tid_empty_bar(slot));
          if (t < 0) break;
          ok = mma_tile();
        }
      } else {
        for (int u = unit0; ok && u < p.units; u += ustep) {
          const int sp = u / per_split;
          const int64_t t_begin = p.n_tiles * sp / p.splits, t_end = p.n_tiles * (sp + 1) / p.splits;
          for (int64_t t = t_begin; ok && t < t_end; ++t) ok = mma_tile();
        }
      }
      // drain: every MMA issued by this thread has completed before TMEM is freed
      mma_commit<PAIR>(drain_bar, 1);
      if (!mbar_wait(drain_bar, 0, nullptr)) fail();
      // a pair: the peer's epilogue releases of the last accumulators (remote arrivals on this CTA's barriers)
      // have landed before the leader may exit
      if (PAIR && ok) {
        for (uint32_t i = tile_i > 2u ? tile_i - 2u : 0u; i < tile_i; ++i)
          if (!mbar_wait(tempty_bar(i & 1u), (i >> 1) & 1u, abort_flag)) {
            fail();
            break;
          }
      }
    }
  } else {
    // ---------------- epilogue ----------------
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    float* my_stash = stash + row;   // column-major [32][129]: conflict-free across a warp
    const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
    uint32_t tile_i = 0;
    bool ok = true;
    const unsigned full = 0xffffffffu;
    TopC<CPAD> top;
    float best = -INFINITY;
    // One finished accumulator: the 256 scores of key tile t for this thread's query row.
    bool waited = p.wait_first != 0;   // this thread has waited for the preceding grids
    auto dep_wait = [&]() {
      if (!waited) {
        asm volatile("griddepcontrol.wait;" ::: "memory");
        waited = true;
      }
    };
    auto epi_tile = [&](int64_t t, bool active, int word) -> bool {
      const int b = tile_i & 1u;
      const uint32_t par = (tile_i >> 1) & 1u;
      // every lane waits (each needs the barrier's acquire); the warp proceeds only if all lanes saw the phase
      // complete, so the warp-collective tcgen05.ld below is never reached by part of a warp
      const bool got = mbar_wait(tfull_bar(b), par, abort_flag);
      if (!__all_sync(full, got)) {
        if (lane == 0) fail();
        return false;
      }
      tc_fence_after();
      const int64_t j0 = t * BN;
      const bool ragged = j0 + BN > p.n;
#pragma unroll 1
      for (int ch = 0; ch < BN / 32; ++ch) {
        float v[32];
        tmem_ld32(tmem + lane_addr + (uint32_t)(b * BN + ch * 32), v);
        if constexpr (SIGN) {
          // lane e keeps the word of key column jc + e: bit `lane` of it is this thread's hyperplane's sign
          const int64_t jc = j0 + ch * 32;
          uint32_t mine = 0;
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const uint32_t w = __ballot_sync(full, v[e] >= 0.f);
            if (lane == e) mine = w;
          }
          dep_wait();
          if (word < p.sig_words && jc + lane < p.n) p.sig[(jc + lane) * p.sig_words + word] = mine;
        } else if (active) {
          const int64_t jc = j0 + ch * 32;
          if (ragged) {
#pragma unroll
            for (int e = 0; e < 32; ++e)
              if (jc + e >= p.n) v[e] = -INFINITY;
          }
          float m = v[0];
#pragma unroll
          for (int e = 1; e < 32; ++e) m = fmaxf(m, v[e]);
          best = fmaxf(best, m);
          if (m >= top.thr) {
            // rare path: stash the chunk in shared memory and insert the entries that clear the threshold
            uint32_t mask = 0;
#pragma unroll
            for (int e = 0; e < 32; ++e) {
              mask |= (v[e] >= top.thr ? 1u : 0u) << e;
              my_stash[e * 129] = v[e];
            }
            while (mask) {
              const int e = __ffs(mask) - 1;
              mask &= mask - 1;
              const float x = my_stash[e * 129];
              if (x >= top.thr && jc + e < p.n) top.insert(x, (uint32_t)(jc + e), p.top_c);
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if constexpr (PAIR)
          mbar_arrive_cluster(map_to_rank(tempty_bar(b), 0));
        else
          mbar_arrive(tempty_bar(b));
      }
      ++tile_i;
      return true;
    };
    auto write_partial = [&](int sp, int q) {
      dep_wait();
      uint64_t* dst = p.part_cand + ((int64_t)sp * p.B + q) * p.top_c;
#pragma unroll
      for (int i = 0; i < CPAD; ++i)
        if (i < top.count) dst[i] = pack_cand(top.s[i], top.j[i]);
      p.part_meta[(int64_t)sp * p.B + q] = PartMeta{best, (uint32_t)top.count};
    };
    if (dyn) {
      const bool active = row < p.B;
      top.init(p.tau_c);
      best = -INFINITY;
      for (uint32_t r = 0; ok; ++r) {
        const int slot = r % RING;
        const bool got = mbar_wait(tid_full_bar(slot), (r / RING) & 1u, abort_flag);
        if (!__all_sync(full, got)) {
          if (lane == 0) fail();
          ok = false;
          break;
        }
        const int t = tid_ring[slot];
        __syncwarp();
        if (lane == 0) mbar_arrive(tid_empty_bar(slot));
        if (t < 0) break;
        ok = epi_tile(t, active, 0);
      }
      if (ok && active && !SIGN) write_partial(blockIdx.x, row);
    } else {
      for (int u = unit0; ok && u < p.units; u += ustep) {
        const int qt = unit_qt(u), sp = u / per_split;
        const int q = qt * BM + row;
        const bool active = q < p.B;
        const int64_t t_begin = p.n_tiles * sp / p.splits, t_end = p.n_tiles * (sp + 1) / p.splits;
        const int word = (qt * BM + quad * 32) / 32;   // signature mode: this warp's word of every signature
        top.init(p.tau_c);
        best = -INFINITY;
        for (int64_t t = t_begin; ok && t < t_end; ++t) ok = epi_tile(t, active, word);
        if (ok && active && !SIGN) write_partial(sp, q);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  // a pair: neither CTA frees the pair's TMEM or exits while the other may still read its accumulators or
  // receive the other's barrier arrivals
  if constexpr (PAIR) cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc<PAIR>(tmem, TMEM_COLS);
  }
}

int gcd_int(int a, int b) {
  while (b) {
    const int t = a % b;
    a = b;
    b = t;
  }
  return a;
}

template <int CPAD, bool SIGN, bool PAIR>
cudaLaunchConfig_t launch_config(cudaLaunchAttribute (&attr)[2], int grid, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = Geo<PAIR>::kSmem;
  cfg.stream = st;
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = PAIR ? 2 : 1;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = PAIR ? 2 : 1;
  return cfg;
}

template <int CPAD, bool SIGN, bool PAIR>
cudaError_t launch_cpad(const CUtensorMap* tq, const CUtensorMap* tk, const TcParams& p, int grid, cudaStream_t st) {
  cudaError_t e = cudaFuncSetAttribute(stage1_tensor_kernel<CPAD, SIGN, PAIR>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Geo<PAIR>::kSmem);
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = launch_config<CPAD, SIGN, PAIR>(attr, grid, st);
  e = cudaLaunchKernelEx(&cfg, stage1_tensor_kernel<CPAD, SIGN, PAIR>, *tq, *tk, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// CTA pairs of this kernel that can be resident at once on the current device (0: none, or not supported).
template <int CPAD>
int max_pair_clusters(cudaStream_t st) {
  if (cudaFuncSetAttribute(stage1_tensor_kernel<CPAD, false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)Geo<true>::kSmem) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = launch_config<CPAD, false, true>(attr, 2, st);
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, stage1_tensor_kernel<CPAD, false, true>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return clusters;
}

bool encode_rows(EncodeTiledFn encode, CUtensorMap* m, const void* base, int64_t d, int64_t rows,
                 uint32_t box_rows) {
  const cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)d * 2};
  const cuuint32_t box[2] = {(cuuint32_t)BK, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Key check of a batch of at least two query tiles on CTA pairs; false if no pair can be resident (the caller
// then uses single CTAs).
template <int CPAD>
bool launch_pairs(TcParams p, const Stage1Args& a, EncodeTiledFn encode, int max_splits, cudaStream_t st,
                  int* splits, cudaError_t* err) {
  // per device and kernel instance, asked once (an idempotent query: concurrent first calls store the same value)
  static std::atomic<int> cache[kMaxDeviceSlots];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDeviceSlots) {
    cudaGetLastError();
    return false;
  }
  int clusters = cache[dev].load(std::memory_order_relaxed);
  if (clusters == 0) {
    clusters = max_pair_clusters<CPAD>(st);
    cache[dev].store(clusters < 1 ? -1 : clusters, std::memory_order_relaxed);
  }
  if (clusters < 1) return false;
  p.pairs = (p.q_tiles + 1) / 2;
  p.a_rows = BM;
  CUtensorMap tq, tk;
  if (!encode_rows(encode, &tq, a.q, a.d, a.B, (uint32_t)BM) ||
      !encode_rows(encode, &tk, a.keys, a.d, a.n, (uint32_t)Geo<true>::kBRows)) {
    *err = cudaErrorInvalidValue;
    return true;
  }
  // Whole waves of units over the resident pairs: a multiple of s0 splits. With several pairs of query tiles every
  // key tile is read by each pair, and the pairs that share a split run at the same time, so a split's keys should
  // stay in L2 until the last of them has read it: splits of at most kPairSplitBytes of keys (as many as the
  // scratch allows). Larger splits were fetched from DRAM again by the pairs of the next wave (1.34x the
  // algorithmic bytes at 21 MB per split, 1.00-1.01x at 10.6 MB and below, at the same kernel time).
  const int s0 = clusters / gcd_int(clusters, p.pairs);
  int s = s0;
  if (p.pairs > 1) {
    const int64_t per = (int64_t)s0 * kPairSplitBytes;
    const int64_t want = (p.n * p.d * 2 + per - 1) / per;
    s = (int)(want * s0 <= max_splits ? want * s0 : (max_splits >= s0 ? max_splits / s0 * s0 : max_splits));
  }
  if ((int64_t)s > p.n_tiles) s = (int)p.n_tiles;
  if (s > max_splits) s = max_splits;
  if (s < 1) s = 1;
  p.splits = s;
  p.units = p.pairs * s;
  *splits = s;
  const int grid = 2 * (p.units < clusters ? p.units : clusters);
  *err = launch_cpad<CPAD, false, true>(&tq, &tk, p, grid, st);
  return true;
}

template <int CPAD>
cudaError_t launch_key_check(TcParams p, const Stage1Args& a, EncodeTiledFn encode, int num_sms, int max_splits,
                             cudaStream_t st, int* splits, bool* paired) {
  cudaError_t err = cudaSuccess;
  if (p.q_tiles >= 2 && launch_pairs<CPAD>(p, a, encode, max_splits, st, splits, &err)) {
    if (paired) *paired = true;
    return err;
  }
  // A batch of at most 128 queries is loaded as a box of B rows (rounded up to 8) rather than 128: boxes that
  // are mostly out of bounds stream measurably slower. The MMA still computes 128 rows; rows past B hold stale
  // shared memory and their TMEM lanes are never read.
  p.a_rows = a.B >= BM ? BM : ((a.B + 7) / 8) * 8;
  CUtensorMap tq, tk;
  if (!encode_rows(encode, &tq, a.q, a.d, a.B, (uint32_t)p.a_rows) ||
      !encode_rows(encode, &tk, a.keys, a.d, a.n, (uint32_t)BN))
    return cudaErrorInvalidValue;
  // splits such that q_tiles * splits is a multiple of the SM count (whole waves of units); one query tile with
  // a tile counter: a dynamic schedule with one split per CTA
  int s = num_sms / gcd_int(num_sms, p.q_tiles);
  if ((int64_t)s > p.n_tiles) s = (int)p.n_tiles;
  if (s > max_splits) s = max_splits;
  if (s < 1) s = 1;
  p.splits = s;
  p.units = p.q_tiles * s;
  if (p.q_tiles == 1 && a.tile_ctr) p.tile_ctr = a.tile_ctr;
  *splits = s;
  const int grid = p.units < num_sms ? p.units : num_sms;
  return launch_cpad<CPAD, false, false>(&tq, &tk, p, grid, st);
}

}  // namespace

cudaError_t launch_signatures(const __nv_bfloat16* rows, int64_t n, int d, const __nv_bfloat16* hyperplanes,
                              int bits, uint32_t* sig, unsigned int* dev_status, EncodeTiledFn encode, int num_sms,
                              cudaStream_t st, bool rows_from_previous) {
  if (n <= 0) return cudaSuccess;
  TcParams p{};
  p.wait_first = rows_from_previous ? 1 : 0;
  p.n = n;
  p.d = d;
  p.B = bits;
  p.tau_c = 0.f;
  p.top_c = 1;
  p.q_tiles = (bits + BM - 1) / BM;
  p.n_tiles = (n + BN - 1) / BN;
  p.k_steps = (d + BK - 1) / BK;
  p.a_rows = bits >= BM ? BM : ((bits + 7) / 8) * 8;
  int s = num_sms / gcd_int(num_sms, p.q_tiles);
  if ((int64_t)s > p.n_tiles) s = (int)p.n_tiles;
  if (s < 1) s = 1;
  p.splits = s;
  p.units = p.q_tiles * s;
  p.sig = sig;
  p.sig_words = bits / 32;
  p.dev_status = dev_status;
  CUtensorMap tq, tk;
  if (!encode_rows(encode, &tq, hyperplanes, d, bits, (uint32_t)p.a_rows) ||
      !encode_rows(encode, &tk, rows, d, n, (uint32_t)BN))
    return cudaErrorInvalidValue;
  const int grid = p.units < num_sms ? p.units : num_sms;
  return launch_cpad<4, true, false>(&tq, &tk, p, grid, st);
}

cudaError_t launch_stage1_tensor(const Stage1Args& a, EncodeTiledFn encode, int num_sms, int max_splits,
                                 cudaStream_t st, int* splits, bool* paired) {
  if (paired) *paired = false;
  TcParams p{};
  p.n = a.n;
  p.d = a.d;
  p.B = a.B;
  p.tau_c = a.tau_c;
  p.top_c = a.top_c;
  p.q_tiles = (a.B + BM - 1) / BM;
  p.n_tiles = (a.n + BN - 1) / BN;
  p.k_steps = (a.d + BK - 1) / BK;
  p.part_cand = a.part_cand;
  p.part_meta = a.part_meta;
  p.dev_status = a.dev_status;
  p.inject_stall = a.inject_stall;
  p.wait_first = a.inputs_from_previous;
  if (a.top_c <= 4) return launch_key_check<4>(p, a, encode, num_sms, max_splits, st, splits, paired);
  if (a.top_c <= 8) return launch_key_check<8>(p, a, encode, num_sms, max_splits, st, splits, paired);
  if (a.top_c <= 16) return launch_key_check<16>(p, a, encode, num_sms, max_splits, st, splits, paired);
  return launch_key_check<32>(p, a, encode, num_sms, max_splits, st, splits, paired);
}

}  // namespace lc

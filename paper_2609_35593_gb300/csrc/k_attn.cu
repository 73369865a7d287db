// Block-sparse attention forward over the kept 64x64 blocks (Sec. 3 step (3)) on sm_103a.
//
// Work item = (head h, pair of query blocks): their 128 query rows form the M = 128 operand
// of tcgen05.mma, and the CTA walks the union of the two kept lists (built by k_pairs, or
// by a forward's CSR kernel: the blocks kept by one query block only, alternating between
// the two, then the rest ascending).  The pair is the adjacent blocks 2p, 2p+1, or, in a
// forward on the 64-token grid, the two candidate blocks that the pairing table names
// (paired by the overlap of their kept lists, so fewer union entries are kept by one block
// only).  Each union entry carries a 2-bit mask saying which of the two query blocks keeps
// it; rows of a block that does not keep the tile get P = 0, so every row sees exactly its
// own kept blocks (softmax renormalised among them).  A one-sided tile keeps only two of the
// four softmax warps busy (rows 0-63 or 64-127); alternating the sides lets the next tile's
// two warps start while the current tile's finish, since S is double-buffered.
//
// Warp roles (192 threads, 2 CTAs per SM):
//   warp 0     TMA producer: Q tile (two 64 x 64 halves, one per query block) per item,
//              K/V tiles (64 x 64) per entry into a 5-stage ring, 128-byte swizzled (UMMA
//              canonical layouts).
//   warp 1     TMEM owner and single-thread MMA issuer:
//                S[g % 2] = Q K_g^T              (M128 N64 K64, Q from TMEM, K from shared memory)
//                O       += P_{g-1} [V_{g-1} | 1]  (M128 N80 K64, P from TMEM, V MN-major)
//              The second 64-column atom of that B operand is a constant shared tile whose
//              first column is 1, so O's column 64 accumulates the row sum of exactly the bf16
//              P values the MMA multiplies, in fp32, and follows every rescale of O for free.
//              Q is copied once per item from its TMA staging buffer into TMEM (tcgen05.cp),
//              so that neither A operand is read from shared memory, whose bandwidth the
//              N = 64 MMAs would otherwise saturate together with the TMA writes.
//              S is double-buffered in TMEM so that S_{g+1} runs while softmax works on S_g;
//              P_g (bf16) is written over the first half of S_g's columns and read from
//              there as the A operand, which keeps it off the shared-memory bus.  MMAs
//              issued by one thread run in issue order, so S_{g+2} overwrites P_g only after
//              P_g V_g has read it.
//   warps 2-5  one query row per thread: tcgen05.ld of S, online softmax in the exp2 domain
//              with lazy rescaling of the TMEM accumulator (only when the running max grows
//              by more than 2^20, done after P is written so that the exponentials overlap
//              the previous P V), tcgen05.st of P, epilogue O / l.  The exponentials are
//              taken against the row's current reference maximum while the tile's maximum
//              is formed (they use different pipes), and redone in the rare case that the
//              maximum grew past the threshold.  The producer announces each item through a
//              small ring of item slots and the softmax warps read its union list from
//              global memory themselves, so that their per-tile work waits only for S.
// Every mbarrier wait is bounded; a wait that gives up records RESS_ETIMEOUT in the status
// word, makes the whole CTA leave its loops, drains in-flight copies and MMAs, frees TMEM
// and returns.

#include <climits>

#include <cudaTypedefs.h>

#include "ress_internal.cuh"
#include "sm100_ptx.cuh"

namespace ress {
using namespace ptx;

constexpr int kAttnThreads = 192;
constexpr int kStages = 5;
constexpr int kRows = 128;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kColS0 = 0, kColO = 128, kColQ = 208;  // TMEM columns: S/P x2, O (80), Q
constexpr int kNO = 80;  // O columns: 64 output channels, the row sum, 15 unused
constexpr uint64_t kWaitNs = 2000000000ull;  // 2 s per wait
constexpr uint64_t kDrainNs = 200000000ull;  // 0.2 s to drain after an abort
constexpr int kFirst = 1, kLast = 2, kTerm = 4;
constexpr int kItemSlots = 4;  // items announced to the softmax warps ahead of their tiles
constexpr uint32_t kTileBytes = 64 * 128;    // one 64 x 64 bf16 tile
// log2 units: rescale only when the running max grows by more than 2^20.  P is bf16 and O
// and its row sum accumulate in fp32, so p <= 2^20 over at most 2^18 keys stays far from
// overflow; a stale max changes no result, the scale cancels in O / l.
constexpr float kLazyThreshold = 20.0f;

struct TileInfo {
  int j, mask, flags, item;
};

struct __align__(1024) AttnSmem {
  uint8_t Q[kRows * 128];
  uint8_t K[kStages][kTileBytes];
  uint8_t V[kStages][kTileBytes];
  uint8_t ONES[kTileBytes];  // B operand columns 64..127 of P V: column 64 all ones
  uint64_t kv_full[kStages], kv_empty[kStages];
  uint64_t q_full, q_empty;
  uint64_t s_full[2], p_full[2];
  uint64_t drain;
  uint64_t it_full[kItemSlots], it_empty[kItemSlots];
  int item_q[kItemSlots];  // item index, or -1: no more items
  TileInfo info[kStages];
  uint32_t tmem_base;
  int abort;
};

struct AttnParams {
  int N, H, nb, npairs, nitems;
  int p0, p1;                   // pairs [p0, p1) of every head are this launch's items
  int rows_per_head, row_step;  // CSR row of item (h, p): h * rows_per_head + row_step * p
  int nsparse;           // pairs 0..nsparse-1 of a head hold only candidate query blocks
  const int32_t* row_ptr;
  const int32_t* plist;  // union lists: entry = j | mask << 16, at row_ptr[h*nb + 2p]
  const int32_t* plen;   // [H * npairs]
  const int32_t* prow;   // items p < npaired: query blocks a | b << 16 (64-token grid), or NULL
  int npaired;
  void* O;               // bf16 or float32 [N, H, 64]
  uint32_t* status;
  uint32_t* counter;
};

// Work order within the launch's pairs [p0, p1): those that hold special (dense) query
// blocks, of every head, first (they are the longest), then the others head by head, so
// that the CTAs running at the same time share one head's K and V in L2.
__device__ __forceinline__ void item_pair(const AttnParams& a, int item, int& h, int& p) {
  const int dlo = max(a.p0, a.nsparse);  // first pair of the range with a dense block
  const int ndense = max(0, a.p1 - dlo);
  const int nsp = max(0, min(a.p1, a.nsparse) - a.p0);
  const int first = a.H * ndense;
  if (item < first) {
    h = item / ndense;
    p = dlo + item % ndense;
  } else {
    h = (item - first) / nsp;
    p = a.p0 + (item - first) % nsp;
  }
}

// Bounded wait for a whole warp.  Fast path: every lane tests the barrier (one shared-memory
// access for the warp, each lane acquiring for itself) and the warp leaves together if all
// saw the phase complete.  Otherwise lane 0 polls (one poller per warp keeps the barrier
// traffic low) and the verdict is broadcast, so that no lane leaves a loop its neighbours
// stay in (the warp runs .sync.aligned code); __syncwarp orders the other lanes' later reads
// after lane 0's acquire.
// First tokens of the two 64-row halves of item (h, p): the query blocks of its table entry
// when the forward paired them, else rows 128 p .. 128 p + 127 (adjacent 64-token blocks,
// or one 128-token block).  A half past the sequence starts at or past N.
__device__ __forceinline__ void item_tokens(const AttnParams& a, int h, int p, int& t0, int& t1) {
  if (p < a.npaired) {
    const int32_t pr = a.prow[(int64_t)h * a.npairs + p];
    t0 = 64 * (pr & 0xffff);
    t1 = 64 * (pr >> 16);
  } else {
    t0 = kRows * p;
    t1 = kRows * p + 64;
  }
}

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, abort, kWaitNs) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  __syncwarp();
  return ok != 0;
}

__device__ __forceinline__ void give_up(AttnSmem& S, uint32_t* status) {
  flag_status(status, kStatusTimeout);
  *reinterpret_cast<volatile int*>(&S.abort) = 1;
}

// ------------------------------------------------------------------------------------
// Union of the two kept lists of every query-block pair, via per-warp bitmaps.  With
// 128-token query blocks (one block per 128-row item) the list is the block's own, every
// entry kept by both halves.  One warp per item; grid ceil(H * npairs / 8) x 256 threads.
// ------------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_pairs(const int32_t* __restrict__ row_ptr,
                                               const int32_t* __restrict__ col_idx,
                                               int64_t cap, int64_t scratch_cap, int nb,
                                               int npairs, int H, bool qb128,
                                               int32_t* __restrict__ plist,
                                               int32_t* __restrict__ plen, uint32_t* status) {
  __shared__ uint32_t bits[8][2][RESS_MAX_BLOCKS / 32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int pair = blockIdx.x * 8 + warp;
  if (pair >= H * npairs) return;
  const int h = pair / npairs, p = pair % npairs;
  const int words = (nb + 31) / 32;
  uint32_t* bA = bits[warp][0];
  uint32_t* bB = bits[warp][1];
  for (int w = lane; w < words; w += 32) bA[w] = bB[w] = 0u;
  const int64_t ra = qb128 ? (int64_t)h * npairs + p : (int64_t)h * nb + 2 * p;
  const bool has_b = !qb128 && 2 * p + 1 < nb;
  const int64_t sa = row_ptr[ra], ea = row_ptr[ra + 1];
  const int64_t eb = has_b ? row_ptr[ra + 2] : ea;
  const bool ok = sa >= 0 && sa <= ea && ea <= eb && eb <= cap && eb <= scratch_cap &&
                  ea - sa <= nb && eb - ea <= nb;
  __syncwarp();
  if (!ok) {
    if (lane == 0) {
      flag_status(status, kStatusBadRow);
      plen[pair] = 0;
    }
    return;
  }
#pragma unroll 4
  for (int64_t x = sa + lane; x < eb; x += 32) {
    const int j = col_idx[x];
    if (j < 0 || j >= nb) {
      flag_status(status, kStatusBadIndex);
      continue;
    }
    atomicOr((x < ea ? bA : bB) + (j >> 5), 1u << (j & 31));
  }
  __syncwarp();
  // Entry order: the k-th block kept by the first query block only and the k-th kept by the
  // second only (k < P, the smaller of the two counts, both ascending) alternate at list
  // positions 2k, 2k + 1, so that the two halves' softmax work of consecutive one-sided
  // tiles overlaps; then the rest of the union in ascending order.  Lane l looks at block
  // 32 w + l.
  int nA = 0, nB = 0;
  for (int w = lane; w < words; w += 32) {
    const uint32_t a = bA[w], b = qb128 ? a : bB[w];
    nA += __popc(a & ~b);
    nB += __popc(b & ~a);
  }
  const int P = min(__reduce_add_sync(0xffffffffu, nA), __reduce_add_sync(0xffffffffu, nB));
  const uint32_t below = (1u << lane) - 1u;
  int cA = 0, cB = 0, cR = 0;  // first-only, second-only and other entries before word w
  for (int w = 0; w < words; ++w) {
    const uint32_t a = bA[w], b = qb128 ? a : bB[w];
    const uint32_t oa = a & ~b, ob = b & ~a;
    const int rA = cA + __popc(oa & below), rB = cB + __popc(ob & below);
    const bool pa = ((oa >> lane) & 1u) && rA < P, pb = ((ob >> lane) & 1u) && rB < P;
    const bool rest = (((a | b) >> lane) & 1u) && !pa && !pb;
    const uint32_t restw = __ballot_sync(0xffffffffu, rest);
    const int j = w * 32 + lane;
    if (pa) plist[sa + 2 * rA] = j | (1 << 16);
    if (pb) plist[sa + 2 * rB + 1] = j | (2 << 16);
    if (rest) {
      const int m = (int)((a >> lane) & 1u) | (int)(((b >> lane) & 1u) << 1);
      plist[sa + 2 * P + cR + __popc(restw & below)] = j | (m << 16);
    }
    cA += __popc(oa);
    cB += __popc(ob);
    cR += __popc(restw);
  }
  if (lane == 0) plen[pair] = 2 * P + cR;
}

// ------------------------------------------------------------------------------------
// main kernel
// ------------------------------------------------------------------------------------
template <bool kOutF32>
__global__ void __launch_bounds__(kAttnThreads, 2)
    k_attn(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
           const __grid_constant__ CUtensorMap tmV, const AttnParams a) {
  extern __shared__ uint8_t smem_raw[];
  AttnSmem& S = *reinterpret_cast<AttnSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &S.abort;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&S.kv_full[s], 1);
      mbar_init(&S.kv_empty[s], 1);
    }
    mbar_init(&S.q_full, 1);
    mbar_init(&S.q_empty, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&S.s_full[b], 1);
      mbar_init(&S.p_full[b], 4);
    }
    mbar_init(&S.drain, 1);
    for (int q = 0; q < kItemSlots; ++q) {
      mbar_init(&S.it_full[q], 1);
      mbar_init(&S.it_empty[q], 4);
    }
    S.abort = 0;
    fence_barrier_init();
    prefetch_tensormap(&tmQ);
    prefetch_tensormap(&tmK);
    prefetch_tensormap(&tmV);
  }
  for (int f = threadIdx.x; f < kTileBytes / 16; f += blockDim.x)
    reinterpret_cast<uint4*>(S.ONES)[f] = make_uint4(0u, 0u, 0u, 0u);
  __syncthreads();
  if (threadIdx.x < 64)  // key row k: element 0 of its 128-byte swizzled row = bf16 1.0
    *reinterpret_cast<uint16_t*>(S.ONES + threadIdx.x * 128 + ((threadIdx.x & 7) << 4)) = 0x3F80;
  fence_proxy_async_smem();
  if (warp == 1) tmem_alloc(&S.tmem_base, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = S.tmem_base;

  if (warp == 0) {
    // =============================== producer ====================================
    // All lanes walk the list together (32 entries per coalesced load, broadcast by
    // shuffle); lane 0 issues the barrier operations and the TMA copies.
    int g = 0, it = 0, pub = 0;
    bool failed = false, q_loaded = false;
    // announce an item (or -1: none left) to the softmax warps, which walk its list themselves
    auto publish = [&](int item) -> bool {
      const int slot = pub % kItemSlots, u = pub / kItemSlots;
      if (u > 0 && !warp_wait(&S.it_empty[slot], (u - 1) & 1, abort)) return false;
      if (lane == 0) {
        S.item_q[slot] = item;
        mbar_arrive(&S.it_full[slot]);
      }
      __syncwarp();
      ++pub;
      return true;
    };
    for (;;) {
      int item = 0;
      if (lane == 0) item = (int)atomicAdd(a.counter, 1u);
      item = __shfl_sync(0xffffffffu, item, 0);
      if (item >= a.nitems) break;
      int h, p;
      item_pair(a, item, h, p);
      const int n = a.plen[h * a.npairs + p];
      if (n <= 0) continue;
      const int32_t* lst = a.plist + a.row_ptr[(int64_t)h * a.rows_per_head + a.row_step * p];
      if (!publish(item)) {
        failed = true;
        break;
      }
      if (it > 0 && !warp_wait(&S.q_empty, (it - 1) & 1, abort)) {
        failed = true;
        break;
      }
      if (lane == 0) {
        int t0, t1;
        item_tokens(a, h, p, t0, t1);
        mbar_arrive_expect_tx(&S.q_full, kRows * 128);
        tma_load_3d(S.Q, &tmQ, &S.q_full, 0, h, t0);               // rows 0..63
        tma_load_3d(S.Q + 64 * 128, &tmQ, &S.q_full, 0, h, t1);    // rows 64..127
      }
      q_loaded = true;
      for (int e0 = 0; e0 < n && !failed; e0 += 32) {
        const int mine = (e0 + lane < n) ? lst[e0 + lane] : 0;
        const int cnt = min(32, n - e0);
        for (int k = 0; k < cnt; ++k) {
          const int ent = __shfl_sync(0xffffffffu, mine, k);
          const int s = g % kStages, u = g / kStages;
          if (u > 0 && !warp_wait(&S.kv_empty[s], (u - 1) & 1, abort)) {
            failed = true;
            break;
          }
          if (lane == 0) {
            const int j = ent & 0xffff;
            int fl = 0;
            if (e0 + k == 0) fl |= kFirst;
            if (e0 + k == n - 1) fl |= kLast;
            S.info[s] = TileInfo{j, ent >> 16, fl, item};
            mbar_arrive_expect_tx(&S.kv_full[s], 2 * kTileBytes);
            tma_load_3d(S.K[s], &tmK, &S.kv_full[s], 0, h, 64 * j);
            tma_load_3d(S.V[s], &tmV, &S.kv_full[s], 0, h, 64 * j);
          }
          ++g;
        }
      }
      if (failed) break;
      ++it;
      q_loaded = false;
    }
    if (!failed) {
      const int s = g % kStages, u = g / kStages;
      if (u > 0 && !warp_wait(&S.kv_empty[s], (u - 1) & 1, abort)) {
        failed = true;
      } else if (lane == 0) {
        S.info[s] = TileInfo{0, 0, kTerm, -1};
        mbar_arrive(&S.kv_full[s]);
      }
      if (!failed && !publish(-1)) failed = true;
    }
    if (failed && lane == 0) {
      give_up(S, a.status);
      // let every copy already issued land before the CTA's shared memory goes away
      for (int back = 1; back <= kStages && g - back >= 0; ++back) {
        const int gg = g - back;
        volatile int no_abort = 0;
        mbar_wait(&S.kv_full[gg % kStages], (gg / kStages) & 1, &no_abort, kDrainNs);
      }
      if (q_loaded) {
        volatile int no_abort = 0;
        mbar_wait(&S.q_full, it & 1, &no_abort, kDrainNs);
      }
    }
  } else if (warp == 1) {
    // ================================ MMA issuer ===================================
    // The whole warp walks the pipeline (lane 0 polls each barrier and broadcasts the
    // verdict) and one lane, chosen by elect.sync, issues every tcgen05 operation: issued
    // from converged code the MMAs go out several times faster than from a lone thread.
    const bool leader = elect_one();
    bool failed = false;
    if (__popc(__ballot_sync(0xffffffffu, leader)) != 1) {  // exactly one issuing lane
      if (lane == 0) flag_status(a.status, kStatusBadRow);
      failed = true;
    }
    const uint32_t idesc_qk = idesc_bf16_f32(kRows, 64, false);
    const uint32_t idesc_pv = idesc_bf16_f32(kRows, kNO, true);
    const uint32_t ones_addr = smem_u32(S.ONES);
    const uint32_t q_addr = smem_u32(S.Q);
    // Descriptors of stage 0's K and V tiles (V with the ONES atom LBO bytes after it).  A
    // descriptor's start address (bits 0-13, in 16-byte units) is below 2^14 for every
    // shared-memory address here, so stage s and K16 slice k are plain adds: the stages
    // lie kTileBytes apart, a K slice 32 bytes on and a V slice 2048 bytes on, and V's
    // leading byte offset (bits 16-29, to ONES) shrinks by the same stage stride.
    constexpr uint64_t kStageUnits = kTileBytes >> 4;
    const uint64_t kdesc0 = sdesc_sw128(smem_u32(S.K[0]));
    const uint32_t v0 = smem_u32(S.V[0]);
    const uint64_t vdesc0 = (sdesc_sw128(v0) & ~(0x3FFFull << 16)) |
                            ((uint64_t)(((ones_addr - v0) >> 4) & 0x3FFFu) << 16);
    bool prev_first = false;
    int it = 0;
    auto issue_pv = [&](int pg, bool first) -> bool {
      const int pb = pg & 1, ps = pg % kStages;
      // the N = 80 B operand: atom 0 = V (channels), atom 1 = ONES, LBO bytes after it
      const uint64_t vd = vdesc0 + (uint64_t)ps * kStageUnits - (((uint64_t)ps * kStageUnits) << 16);
      if (!warp_wait(&S.p_full[pb], (pg >> 1) & 1, abort)) return false;
      tc_fence_after();
      if (leader) {
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mma_bf16_ts(tmem + kColO, tmem + kColS0 + 64 * pb + 8 * k, vd + 128 * k, idesc_pv,
                      (k > 0 || !first) ? 1u : 0u);
        mma_commit(&S.kv_empty[ps]);  // also tells the softmax warps that P V has landed
      }
      __syncwarp();
      return true;
    };
    // the info of tile t once its K/V stage has landed
    auto fetch = [&](int t, TileInfo& info) -> bool {
      if (!warp_wait(&S.kv_full[t % kStages], (t / kStages) & 1, abort)) return false;
      info = S.info[t % kStages];
      return true;
    };
    // Order per tile g: S_g, then (with tile g+1 already landed and its info read, so that
    // none of that sits between P_{g-1} and the next S) P_{g-1} V_{g-1}.  S_{g+1} overwrites
    // the buffer of P_{g-1}, which P_{g-1} V_{g-1}, issued before it, has read by then.
    TileInfo info;
    if (!failed && !fetch(0, info)) failed = true;
    for (int g = 0; !failed && !(info.flags & kTerm); ++g) {
      if (info.flags & kFirst) {
        if (!warp_wait(&S.q_full, it & 1, abort)) {
          failed = true;
          break;
        }
        tc_fence_after();
        // Q (128 x 64) into TMEM, one K16 slice (8 columns) per copy; the staging buffer
        // is free again once the copies have completed.  Copies and MMAs issued by this
        // lane run in order, so earlier S MMAs have read the previous Q by then.
        if (leader) {
#pragma unroll
          for (int k = 0; k < 4; ++k) tmem_cp_128x256b(tmem + kColQ + 8 * k, sdesc_sw128(q_addr + 32 * k));
          mma_commit(&S.q_empty);
        }
        __syncwarp();
        ++it;
      }
      // no thread-sync fence here: S_g overwrites what softmax read for tile g-2, and the
      // fence after waiting for P_{g-2} already orders every later tcgen05 operation
      const int s = g % kStages, b = g & 1;
      const uint64_t kd = kdesc0 + (uint64_t)s * kStageUnits;
      if (leader) {
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mma_bf16_ts(tmem + kColS0 + 64 * b, tmem + kColQ + 8 * k, kd + 2 * k, idesc_qk,
                      k > 0 ? 1u : 0u);
        mma_commit(&S.s_full[b]);
      }
      __syncwarp();
      const bool first = (info.flags & kFirst) != 0;
      if (!fetch(g + 1, info)) {
        failed = true;
        break;
      }
      if (g > 0 && !issue_pv(g - 1, prev_first)) {
        failed = true;
        break;
      }
      prev_first = first;
      if ((info.flags & kTerm) && !issue_pv(g, first)) {  // the CTA's last tile
        failed = true;
        break;
      }
    }
    if (failed && lane == 0) give_up(S, a.status);
    // wait for every MMA issued so far before TMEM is released
    if (leader) {
      mma_commit(&S.drain);
      volatile int no_abort = 0;
      mbar_wait(&S.drain, 0, &no_abort, kDrainNs);
    }
    __syncwarp();
  } else {
    // ================================ softmax =====================================
    // Each warp walks the announced items' union lists itself (32 entries per coalesced
    // load, the next 32 loaded while the current ones are used), so a tile costs it only
    // the wait for S.
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;  // query row within the 128-row tile
    const int half = r >> 6;
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    const float kScale = 1.4426950408889634f * 0.125f;  // log2(e) / sqrt(64)
    // p = 2^(s * log2(e)/8 - m) of this row's 64 columns, two columns per packed FMA
    auto exps = [&](const float (&x)[64], float m, uint32_t (&w)[32]) {
      const float nm = -m;
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        float t0, t1;
        fma2(t0, t1, x[2 * e], x[2 * e + 1], kScale, kScale, nm, nm);
        w[e] = pack_bf16x2(ex2(t0), ex2(t1));
      }
    };
    // the row maximum of the raw scores (the scale is positive) as a tree of 3-input maxima
    auto row_max = [&](const float (&x)[64]) -> float {
      float m1[22];
#pragma unroll
      for (int k = 0; k < 21; ++k) m1[k] = fmax3(x[3 * k], x[3 * k + 1], x[3 * k + 2]);
      m1[21] = x[63];
      float m2[8];
#pragma unroll
      for (int k = 0; k < 7; ++k) m2[k] = fmax3(m1[3 * k], m1[3 * k + 1], m1[3 * k + 2]);
      m2[7] = m1[21];
      return fmax3(fmax3(m2[0], m2[1], m2[2]), fmax3(m2[3], m2[4], m2[5]), fmaxf(m2[6], m2[7]));
    };
    int g = 0;
    bool stop = false;
    for (int pub = 0; !stop; ++pub) {
      const int slot = pub % kItemSlots;
      if (!warp_wait(&S.it_full[slot], (pub / kItemSlots) & 1, abort)) {
        give_up(S, a.status);
        break;
      }
      const int item = S.item_q[slot];
      __syncwarp();
      if (lane == 0) mbar_arrive(&S.it_empty[slot]);
      if (item < 0) break;
      int h, p, t0, t1;
      item_pair(a, item, h, p);
      item_tokens(a, h, p, t0, t1);
      const int n = a.plen[h * a.npairs + p];
      const int32_t* lst = a.plist + a.row_ptr[(int64_t)h * a.rows_per_head + a.row_step * p];
      float m_use = -INFINITY;  // this row's reference maximum (log2 units); warp-uniform -inf
      int mine = lane < n ? lst[lane] : 0;
      for (int e0 = 0; e0 < n && !stop; e0 += 32) {
        const int nxt = (e0 + 32 + lane < n) ? lst[e0 + 32 + lane] : 0;
        const int cnt = min(32, n - e0);
        for (int k = 0; k < cnt; ++k) {
          const int ent = __shfl_sync(0xffffffffu, mine, k);
          const int j = ent & 0xffff;
          const bool active = (ent >> (16 + half)) & 1;  // warp-uniform
          const int b = g & 1;
          // S_g complete implies every earlier MMA complete, P_{g-2} V_{g-2} included
          if (!warp_wait(&S.s_full[b], (g >> 1) & 1, abort)) {
            give_up(S, a.status);
            stop = true;
            break;
          }
          tc_fence_after();
          const uint32_t tS = tmem + lane_base + kColS0 + 64 * b;
          if (active) {
            float x[64];
            {
              uint32_t v[64];
              RESS_TMEM_LD64(tS, v);
#pragma unroll
              for (int c = 0; c < 64; ++c) x[c] = __uint_as_float(v[c]);
            }
            if (j == a.nb - 1) {  // ragged last key block: keys past N do not exist
              const int valid = a.N - 64 * j;
#pragma unroll
              for (int c = 0; c < 64; ++c)
                if (c >= valid) x[c] = -INFINITY;
            }
            uint32_t w[32];
            float alpha = 1.f;
            bool rescale = false;
            if (m_use == -INFINITY) {
              // first kept tile of this row: O row is still zero
              m_use = row_max(x) * kScale;
              exps(x, m_use, w);
            } else {
              // the exponentials against the current reference run alongside the maximum;
              // a row whose maximum grew by more than 2^20 (rare) takes the new maximum
              // and the warp recomputes, so P is the same as with the maximum taken first
              exps(x, m_use, w);
              const float mt = row_max(x) * kScale;
              const bool grow = mt > m_use + kLazyThreshold;
              if (__any_sync(0xffffffffu, grow)) {
                if (grow) {
                  alpha = ex2(m_use - mt);
                  m_use = mt;
                  rescale = true;
                }
                exps(x, m_use, w);
              }
            }
            RESS_TMEM_ST32(tS, w);  // P_g over the first 32 columns of S_g
            if (__any_sync(0xffffffffu, rescale)) {
              // the previous P V must have landed before the accumulator row is rescaled;
              // the exponentials above ran while it was in flight
              if (!warp_wait(&S.kv_empty[(g - 1) % kStages], ((g - 1) / kStages) & 1, abort)) {
                give_up(S, a.status);
                stop = true;
                break;
              }
              tc_fence_after();
#pragma unroll
              for (int hc = 0; hc < 2; ++hc) {
                uint32_t v[32];
                RESS_TMEM_LD32(tmem + lane_base + kColO + 32 * hc, v);
#pragma unroll
                for (int c = 0; c < 32; ++c) v[c] = __float_as_uint(__uint_as_float(v[c]) * alpha);
                RESS_TMEM_ST32(tmem + lane_base + kColO + 32 * hc, v);
              }
              {  // the row sum (column 64) and the unused columns after it
                uint32_t v[16];
                RESS_TMEM_LD16(tmem + lane_base + kColO + 64, v);
#pragma unroll
                for (int c = 0; c < 16; ++c) v[c] = __float_as_uint(__uint_as_float(v[c]) * alpha);
                RESS_TMEM_ST16(tmem + lane_base + kColO + 64, v);
              }
            }
          } else {
            uint32_t w[32];
#pragma unroll
            for (int e = 0; e < 32; ++e) w[e] = 0u;
            RESS_TMEM_ST32(tS, w);
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&S.p_full[b]);

          if (e0 + k == n - 1) {
            // epilogue: O / l for this row once the last P V has landed
            if (!warp_wait(&S.kv_empty[g % kStages], (g / kStages) & 1, abort)) {
              give_up(S, a.status);
              stop = true;
              break;
            }
            tc_fence_after();
            const int token = (half ? t1 : t0) + (r & 63);
            const bool row_exists = token < a.N;
            uint32_t o[2][32], ls[16];
            RESS_TMEM_LD32(tmem + lane_base + kColO, o[0]);
            RESS_TMEM_LD32(tmem + lane_base + kColO + 32, o[1]);
            RESS_TMEM_LD16(tmem + lane_base + kColO + 64, ls);
            const float l = __uint_as_float(ls[0]);  // row sum of the bf16 probabilities
            if (row_exists) {
              if (!(l > 0.f)) flag_status(a.status, kStatusBadRow);
              const float inv = l > 0.f ? 1.0f / l : 0.f;
              const int64_t off = ((int64_t)token * a.H + h) * 64;
              if (kOutF32) {
                float4* dst = reinterpret_cast<float4*>(static_cast<float*>(a.O) + off);
#pragma unroll
                for (int ch = 0; ch < 16; ++ch) {
                  const int c = ch * 4;
                  dst[ch] = make_float4(__uint_as_float(o[c >> 5][c & 31]) * inv,
                                        __uint_as_float(o[(c + 1) >> 5][(c + 1) & 31]) * inv,
                                        __uint_as_float(o[(c + 2) >> 5][(c + 2) & 31]) * inv,
                                        __uint_as_float(o[(c + 3) >> 5][(c + 3) & 31]) * inv);
                }
              } else {
                uint4* dst = reinterpret_cast<uint4*>(static_cast<uint16_t*>(a.O) + off);
#pragma unroll
                for (int ch = 0; ch < 8; ++ch) {
                  uint32_t wo[4];
#pragma unroll
                  for (int e = 0; e < 4; ++e) {
                    const int c = ch * 8 + 2 * e;
                    wo[e] = pack_bf16x2(__uint_as_float(o[c >> 5][c & 31]) * inv,
                                        __uint_as_float(o[(c + 1) >> 5][(c + 1) & 31]) * inv);
                  }
                  dst[ch] = make_uint4(wo[0], wo[1], wo[2], wo[3]);
                }
              }
            }
            tc_fence_before();
          }
          ++g;
        }
        mine = nxt;
      }
    }
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------------------------
// host side
// ------------------------------------------------------------------------------------
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// [N, H, 64] bf16 viewed as a 3-D tensor {64, H, N}; box {64, 1, rows}, 128-byte swizzle.
static bool make_map(CUtensorMap* m, const void* base, int N, int H, int rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {64, (cuuint64_t)H, (cuuint64_t)N};
  cuuint64_t strides[2] = {128, (cuuint64_t)H * 128};
  cuuint32_t box[3] = {64, 1, (cuuint32_t)rows};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

static int sm_count() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
}

int attn_num_pairs(const Shape& s) { return (s.nb + 1) / 2; }

cudaError_t launch_attn_pairs(const AttnArgs& x, cudaStream_t st) {
  const Shape& s = x.s;
  const int npairs = attn_num_pairs(s);
  const int pairs = s.H * npairs;
  k_pairs<<<(pairs + 7) / 8, 256, 0, st>>>(x.row_ptr, x.col_idx, x.col_capacity, x.scratch_cap,
                                           s.nb, npairs, s.H, s.qb == 128, x.plist, x.plen,
                                           x.status);
  note_launch();
  return cudaGetLastError();
}

cudaError_t launch_attn_range(const AttnArgs& x, int p0, int p1, int slot, cudaStream_t st) {
  const Shape& s = x.s;
  const int npairs = attn_num_pairs(s);
  if (p0 < 0 || p1 > npairs || p0 >= p1 || slot < 0 || slot >= kAttnCounterSlots)
    return cudaErrorInvalidValue;
  CUtensorMap tq, tk, tv;
  if (!make_map(&tq, x.Q, s.N, s.H, 64) || !make_map(&tk, x.K, s.N, s.H, 64) ||
      !make_map(&tv, x.V, s.N, s.H, 64))
    return cudaErrorInvalidValue;
  const int items = s.H * (p1 - p0);
  const bool qb128 = s.qb == 128;
  AttnParams p;
  p.N = s.N;
  p.H = s.H;
  p.nb = s.nb;
  p.npairs = npairs;
  p.p0 = p0;
  p.p1 = p1;
  // items whose rows are all candidate query rows come first in each head's order
  p.nsparse = qb128 ? s.nqc : s.ncand / 2;
  p.rows_per_head = qb128 ? s.nq : s.nb;
  p.row_step = qb128 ? 1 : 2;
  p.nitems = items;
  p.row_ptr = x.row_ptr;
  p.plist = x.plist;
  p.plen = x.plen;
  p.prow = x.prow;
  p.npaired = x.prow ? x.npaired : 0;
  p.O = x.O;
  p.status = x.status;
  p.counter = x.counter + slot;
  const size_t smem = sizeof(AttnSmem) + 1024;
  auto kern = x.out_f32 ? k_attn<true> : k_attn<false>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int grid = min(items, 2 * sm_count());
  kern<<<grid, kAttnThreads, smem, st>>>(tq, tk, tv, p);
  note_launch();
  return cudaGetLastError();
}

cudaError_t launch_sparse_attn(const AttnArgs& x, cudaStream_t st) {
  cudaError_t e = launch_attn_pairs(x, st);
  if (e != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(x.counter, 0, sizeof(uint32_t), st)) != cudaSuccess) return e;
  return launch_attn_range(x, 0, attn_num_pairs(x.s), 0, st);
}

}  // namespace ress

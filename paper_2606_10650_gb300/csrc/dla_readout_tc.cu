// dla_readout_tc.cu -- K2, the read-out of Eq. (capacity_bounded_output), on
// the 5th-generation tensor cores (tcgen05 + TMEM + TMA) for bf16 inputs,
// d = 128:
//   o_t = sum_{x < m0} lambda_{t, L_t(x)} (S_x q_t)                  snapshot part
//       + sum_{s <= t in interval} lambda_{t, L_t(e(s))} (q_t . k_s) v_s   intra part
// The cache seen by token t is the snapshot taken by K1 at the start of t's
// 128-token interval (m0 states, logical order) regrouped by the merges decided
// inside the interval: merges only add states, so snapshot entry x contributes
// with the lambda of its logical slot L_t(x) after the interval's events up to
// t.  The tokens of the interval itself belong to the entry opened by the last
// boundary event at or before them (event 0: the snapshot's open entry).
//
// One CTA per (pair of consecutive intervals A, B, stream).  Consecutive
// snapshot lists share most of their states (only entries that changed get new
// pool entries), so the CTA loads the union of the two lists once and applies
// each state to the tokens of both intervals: D_x^A = Q_A S_x^T and
// D_x^B = Q_B S_x^T (M = 128 tokens each, N = 128, K = 128) in fp16: K1 stores
// each snapshot as S_x / s_x in fp16 (s_x a power of two from a bound of
// |S_x|_F, so that no element overflows and every element keeps 2^-12
// relative rounding), and Q is converted in place to fp16 with a power-of-two
// scale per row once the intra part has used it (exact: bf16 values fit fp16's
// significand); the epilogue multiplies D_x by s_x and the row's inverse scale
// together with lambda.  An interval's MMAs are skipped for a state that is
// not in its list.  Before
// the states, the intra part of each interval: P = Q K^T, Pt = P o W
// (W_ts = lambda_{t, L_t(e(s))} for s <= t, else 0) written as bf16 over the K
// tile, O = Pt V with V as loaded (an MN-major operand), which o starts from.
// Roles: warp 0 issues TMA loads (the two Q, K and V tiles, then each union
// state, 32 KB in fp16, through four 32 KB stages), warp 1
// issues tcgen05.mma (one thread) into two TMEM buffers of two 128-column
// accumulators (A, B), warps 2..17 read TMEM, weight by lambda and accumulate o
// in registers (one token row, one interval and one 64-column half per thread;
// warp w reads TMEM lane quadrant w % 4).  All waits are bounded (~2 s, then
// an abort flag and status 5).
#include "dla_common.cuh"
#include "dla_sm100.cuh"
#include "dla_tmap.h"

namespace dla {

namespace {

using namespace sm100;

constexpr int L = 128;   // tokens per interval
constexpr int D = 128;   // head dimension
constexpr int NT = 576;   // 18 warps
constexpr int NEPI = 16;  // epilogue warps
constexpr int NHS = 4;   // shared-memory stages (32 KB: an fp16 state, a K / Pt tile or a V tile)
constexpr int NBUF = 2;  // TMEM buffers (each: accumulator A, accumulator B)
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kTile = L * 128;  // one K-major 128B-swizzled tile: 128 rows x 64 bf16
constexpr int kRows = L + 1;         // events 0 .. L of an interval
// Slot tables of one interval, in one region: first the intra part's tab[e][i]
// for the entry opened at event i <= e (row e at e (e + 1) / 2), later the
// snapshot entries' slots tab[e][x] (row stride kMaxC).
constexpr int kSnapTab = kRows * kMaxC;
constexpr int kIntraTab = kRows * (kRows + 1) / 2;
constexpr int kTabBytes = kSnapTab > kIntraTab ? kSnapTab : kIntraTab;

struct Side {      // per interval of the pair
  int evt[L];      // events (boundaries) at or before token t
  int mlog[L];     // merge indices
  uint8_t bnd[L];  // boundary flags
};

// CAPB: the largest capacity of the instance.  CAPB > kMaxC is the DLA(I)
// instance: no merges, so an entry's logical slot is its list index and the
// entry opened at the interval's e-th boundary sits at slot m0 - 1 + e; it
// keeps no slot tables.
template <int CAPB>
struct TcSmem {
  static constexpr bool kBig = CAPB > kMaxC;
  static constexpr int MAXU = 2 * CAPB;  // union of two lists
  uint8_t Q[2][2][kTile];      // [interval][k-half]: Q, the A operand                 64 KB
  uint8_t hs[NHS][2][kTile];   // [stage][half]: K then Pt, V, then state parts         128 KB
  unsigned char tab[2][kBig ? 16 : kTabBytes];
  Side side[2];
  int ids[2][CAPB];            // pool ids of the two lists
  int uid[MAXU];               // union: pool id
  int uxa[MAXU], uxb[MAXU];    // union: index in list A / list B, or -1
  float uscale[MAXU];          // union: scale s_x of the fp16 entry (S_x / s_x is stored)
  float qmax[2][2][L];         // [interval][k-half][row]: max |q| of the half row (Q's fp16 scales)
  int logi[2][kRows];          // table-build scratch, per interval
  int nu;                      // union size
  uint64_t bar_q, bar_pt, bar_done;
  uint64_t full[NHS], empty[NHS], acc_full[NBUF], acc_empty[NBUF];
  uint32_t tmem_base;
  int abort_flag;
  int skip;                    // the call has failed before this CTA's work: do none of it
};

// Snapshot entries' slot table of one interval (one warp): row e holds L(x) of
// snapshot entry x after the interval's first e boundary events.
__device__ __forceinline__ void build_snap_table(const Side& sd, unsigned char* tab, int* logi, int m0, int lane) {
  for (int x = lane; x < m0; x += 32) {
    logi[x] = x;
    tab[x] = (unsigned char)x;
  }
  __syncwarp();
  unsigned long long lo64 = 0, hi64 = 0;
#pragma unroll
  for (int w4 = 0; w4 < 4; ++w4) {
    const unsigned m = __ballot_sync(0xffffffffu, sd.bnd[32 * w4 + lane] != 0);
    if (w4 < 2) lo64 |= (unsigned long long)m << (32 * w4);
    else hi64 |= (unsigned long long)m << (32 * (w4 - 2));
  }
  int ev = 0;
  while (lo64 | hi64) {
    const int tt = lo64 ? (__ffsll((long long)lo64) - 1) : (64 + __ffsll((long long)hi64) - 1);
    if (lo64) lo64 &= lo64 - 1; else hi64 &= hi64 - 1;
    const int j = sd.mlog[tt];
    ev += 1;
    for (int x = lane; x < m0; x += 32) {
      int li = logi[x];
      if (j >= 0 && li > j) logi[x] = --li;
      tab[ev * kMaxC + x] = (unsigned char)li;
    }
  }
}

// Intra part's slot table of one interval (one warp): row e (at e (e + 1) / 2)
// holds the slot, after event e, of the entry opened at event i <= e (event 0:
// the snapshot's open entry, slot m0 - 1).  Lane x owns the entries opened at
// events x, x + 32, ...; a merge at index j moves every slot above j down by one.
__device__ __forceinline__ void build_intra_table(const Side& sd, unsigned char* tab, int* logi, int m0, int lane) {
  if (lane == 0) {
    logi[0] = m0 - 1;  // unused when m0 = 0 (the interval then opens with a boundary)
    tab[0] = (unsigned char)(m0 - 1);
  }
  unsigned long long lo64 = 0, hi64 = 0;
#pragma unroll
  for (int w4 = 0; w4 < 4; ++w4) {
    const unsigned m = __ballot_sync(0xffffffffu, sd.bnd[32 * w4 + lane] != 0);
    if (w4 < 2) lo64 |= (unsigned long long)m << (32 * w4);
    else hi64 |= (unsigned long long)m << (32 * (w4 - 2));
  }
  int cnt = m0, ev = 0;
  while (lo64 | hi64) {
    const int tt = lo64 ? (__ffsll((long long)lo64) - 1) : (64 + __ffsll((long long)hi64) - 1);
    if (lo64) lo64 &= lo64 - 1; else hi64 &= hi64 - 1;
    const int j = sd.mlog[tt];
    if (j >= 0) cnt -= 1;
    ev += 1;
    if ((ev & 31) == lane) logi[ev] = cnt;
    cnt += 1;
    unsigned char* row = tab + ev * (ev + 1) / 2;
    for (int i = lane; i <= ev; i += 32) {
      int li = logi[i];
      if (j >= 0 && i < ev && li > j) logi[i] = --li;
      row[i] = (unsigned char)li;
    }
  }
}

// Events at or before token tt of an interval (one warp, one token per lane).
__device__ __forceinline__ int events_before(const Side& sd, int tt, int lane) {
  int e = 0;
#pragma unroll
  for (int w4 = 0; w4 < 4; ++w4) {
    const unsigned m = __ballot_sync(0xffffffffu, sd.bnd[32 * w4 + lane] != 0);
    if (32 * w4 + 31 <= tt) e += __popc(m);
    else if (32 * w4 <= tt) e += __popc(m & (0xffffffffu >> (31 - (tt - 32 * w4))));
  }
  return e;
}

}  // namespace

// 18 warps: the sub-partitions holding five of them bound a thread to 96 registers.
// kStream: inputs streamed in by the host while the kernel runs (lambda read
// through L2) and the output copied back piece by piece (per-piece CTA counts).
// kRagged: per-row lengths (padding after them).  Separate instances, so the
// common one keeps its code unchanged.
template <bool kStream, bool kRagged, int CAPB = kMaxC>
__global__ void __launch_bounds__(NT, 1)
    readout_tc_kernel(ReadoutArgs a, const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmS,
                      const __grid_constant__ CUtensorMap tmO, int32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  using Smem = TcSmem<CAPB>;
  constexpr bool kBig = Smem::kBig;
  Smem& sm = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int bh = blockIdx.x, pair = blockIdx.y;  // streams fastest: CTAs dispatched interval pair by pair
  const int b = bh / a.H, h = bh % a.H;
  const int C = a.C;
  const int sA = 2 * pair;
  // token row of the row's token 0, and the TMA coordinates of it: (token, batch)
  // = (t, b) in the padded layout, (row_start[b] + t, 0) in the packed one (the
  // per-row-length instance only)
  const long long tok0 = kRagged ? row_tok0(a.row_start, b, a.T) : (long long)b * a.T;
  const bool packed = kRagged && a.row_start != nullptr;
  const int tma_t = packed ? (int)tok0 : 0, tma_b = packed ? 0 : b;
  // this row's end (padding after it)
  const int t_end = kRagged ? row_t_end(a.seq_lens, b, a.t_begin, a.t_end) : a.t_end;
  if constexpr (kRagged) {
    if (a.t_begin + sA * L >= t_end) {  // the pair lies past the row's length: o not written
      if constexpr (kStream) {
        if (a.out_done && tid == 0) atomicAdd(a.out_done + pair / a.out_piece_pairs, 1);
      }
      return;
    }
  }
  const bool hasB = (sA + 1) < a.nsnap && (!kRagged || a.t_begin + (sA + 1) * L < t_end);
  // with a scan running concurrently: both intervals of the pair must be complete
  wait_progress(a.progress, a.progress_ctas, bh, a.snap_base + sA + (hasB ? 2 : 1), a.status);
  if (tid == 0) {
    // thread 0 issues the TMA loads: they read what the scan wrote (pool entries)
    // and the inputs streamed in before its progress
    if (a.progress) asm volatile("fence.proxy.async.global;" ::: "memory");
    // A failed call (a bounded wait that gave up, here or in another kernel, or a
    // device check): the scan may not have written this pair's lists, so the
    // CTA does none of the work and leaves o unwritten.
    sm.skip = (*(volatile int32_t*)a.status != 0);
  }
  __syncthreads();
  if (sm.skip) {
    if constexpr (kStream) {
      if (a.out_done && tid == 0) atomicAdd(a.out_done + pair / a.out_piece_pairs, 1);
    }
    return;
  }
  // interval A (side 0) and B (side 1) of the pair
  const int c0A = a.t_begin + sA * L, c0B = c0A + L;
  const int LcA = min(L, t_end - c0A), LcB = hasB ? min(L, t_end - c0B) : 0;
  const long long lrowA = (long long)bh * a.snap_stride + a.snap_base + sA, lrowB = lrowA + 1;
  // lists and trace come from the scan: read past L1 (__ldcg)
  // live entries of the two lists, checked against the capacity (a violation is
  // a device-check failure and is clamped, so that nothing indexes out of bounds)
  int m0A = __ldcg(a.snap_m0 + lrowA), m0B = hasB ? __ldcg(a.snap_m0 + lrowB) : 0;
  if (m0A < 0 || m0A > C || m0B < 0 || m0B > C) {
    if (tid == 0) atomicCAS(a.status, 0, 6);
    m0A = min(max(m0A, 0), C);
    m0B = min(max(m0B, 0), C);
  }
  auto c0_of = [&](int side) { return side ? c0B : c0A; };
  auto Lc_of = [&](int side) { return side ? LcB : LcA; };
  volatile int* abort = &sm.abort_flag;

  if (tid == 0) {
    mbar_init(&sm.bar_q, 1);
    mbar_init(&sm.bar_pt, NEPI);
    mbar_init(&sm.bar_done, 1);
    for (int i = 0; i < NHS; ++i) {
      mbar_init(&sm.full[i], 1);
      mbar_init(&sm.empty[i], 1);
    }
    for (int i = 0; i < NBUF; ++i) {
      mbar_init(&sm.acc_full[i], 1);
      mbar_init(&sm.acc_empty[i], NEPI);
    }
    sm.abort_flag = 0;
    fence_mbar_init();
    // the Q tiles go out first; they depend on nothing
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
    prefetch_tmap(&tmS);
    mbar_expect_tx(&sm.bar_q, (hasB ? 4 : 2) * kTile);
    tma_load_4d(sm.Q[0][0], &tmQ, &sm.bar_q, 0, h, tma_t + c0A, tma_b);
    tma_load_4d(sm.Q[0][1], &tmQ, &sm.bar_q, 64, h, tma_t + c0A, tma_b);
    if (hasB) {
      tma_load_4d(sm.Q[1][0], &tmQ, &sm.bar_q, 0, h, tma_t + c0B, tma_b);
      tma_load_4d(sm.Q[1][1], &tmQ, &sm.bar_q, 64, h, tma_t + c0B, tma_b);
    }
  }
  for (int i = tid; i < 2 * CAPB; i += NT) {
    const int side = i / CAPB, x = i % CAPB;
    int id = (x < (side ? m0B : m0A)) ? __ldcg(a.snap_ids + (side ? lrowB : lrowA) * C + x) : -1;
    if (x < (side ? m0B : m0A) && (id < 0 || id >= a.pool_cap)) {  // a pool id outside the pool
      atomicCAS(a.status, 0, 6);
      id = 0;
    }
    sm.ids[side][x] = id;
  }
  if (warp == 1) tmem_alloc(&sm.tmem_base, kTmemCols);
  __syncthreads();
  if (warp == 0) {
    // union of the two lists: list A in order, then the entries of list B not in A
    for (int x = lane; x < CAPB; x += 32) {
      if (x < m0A) {
        sm.uid[x] = sm.ids[0][x];
        sm.uxa[x] = x;
        sm.uxb[x] = -1;
      }
    }
    __syncwarp();
    int nb_only = 0;
    for (int base = 0; base < m0B; base += 32) {
      const int x = base + lane;
      int match = -1;
      if (x < m0B) {
        const int id = sm.ids[1][x];
        for (int y = 0; y < m0A; ++y)
          if (sm.ids[0][y] == id) match = y;
      }
      const unsigned only = __ballot_sync(0xffffffffu, x < m0B && match < 0);
      if (x < m0B) {
        if (match >= 0) {
          sm.uxb[match] = x;
        } else {
          const int u = m0A + nb_only + __popc(only & ((1u << lane) - 1u));
          sm.uid[u] = sm.ids[1][x];
          sm.uxa[u] = -1;
          sm.uxb[u] = x;
        }
      }
      nb_only += __popc(only);
    }
    if (lane == 0) sm.nu = m0A + nb_only;
    __syncwarp();
    const int nu_w = m0A + nb_only;
    for (int u = lane; u < nu_w; u += 32) sm.uscale[u] = __ldcg(a.pool_scale + (long long)bh * a.pool_cap + sm.uid[u]);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  const int nu = sm.nu;
  // Ring units: g = 0, 1 the K tiles of intervals A and B (then Pt over them),
  // g = 2, 3 their V tiles (the MN-major B operand of O), g = 4 + x union state
  // x (fp16).  Unit g uses stage g % NHS for the (g / NHS)-th time.
  // Accumulators (TMEM buffer n % NBUF): n = 0 P = Q K^T, n = 1 O = Pt V,
  // n = 2 + x union state x.

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int issued[NHS];  // uses of each stage so far
      mbar_expect_tx(&sm.full[0], 2 * kTile);
      tma_load_4d(sm.hs[0][0], &tmK, &sm.full[0], 0, h, tma_t + c0A, tma_b);
      tma_load_4d(sm.hs[0][1], &tmK, &sm.full[0], 64, h, tma_t + c0A, tma_b);
      mbar_expect_tx(&sm.full[2], 2 * kTile);
      tma_load_4d(sm.hs[2][0], &tmV, &sm.full[2], 0, h, tma_t + c0A, tma_b);
      tma_load_4d(sm.hs[2][1], &tmV, &sm.full[2], 64, h, tma_t + c0A, tma_b);
      if (hasB) {
        mbar_expect_tx(&sm.full[1], 2 * kTile);
        tma_load_4d(sm.hs[1][0], &tmK, &sm.full[1], 0, h, tma_t + c0B, tma_b);
        tma_load_4d(sm.hs[1][1], &tmK, &sm.full[1], 64, h, tma_t + c0B, tma_b);
        mbar_expect_tx(&sm.full[3], 2 * kTile);
        tma_load_4d(sm.hs[3][0], &tmV, &sm.full[3], 0, h, tma_t + c0B, tma_b);
        tma_load_4d(sm.hs[3][1], &tmV, &sm.full[3], 64, h, tma_t + c0B, tma_b);
      } else {  // first phase complete without data: the stages' later uses keep their parity
        mbar_arrive(&sm.full[1]);
        mbar_arrive(&sm.full[3]);
      }
      for (int i = 0; i < NHS; ++i) issued[i] = 1;
      for (int u = 0; u < nu; ++u) {
        const int g = 4 + u, hsi = g % NHS, k = g / NHS;
        if (!mbar_wait(&sm.empty[hsi], (uint32_t)((k & 1) ^ 1), abort, status)) break;
        mbar_expect_tx(&sm.full[hsi], 2 * kTile);
        const int row = (int)(((long long)bh * a.pool_cap + sm.uid[u]) * D);
        tma_load_2d(sm.hs[hsi][0], &tmS, &sm.full[hsi], 0, row);
        tma_load_2d(sm.hs[hsi][1], &tmS, &sm.full[hsi], 64, row);
        issued[hsi] = k + 1;
      }
      if (*abort) {  // let copies in flight land before the CTA exits
        for (int i = 0; i < NHS; ++i)
          if (issued[i] > 0) mbar_wait_drain(&sm.full[i], (uint32_t)((issued[i] - 1) & 1));
        mbar_wait_drain(&sm.bar_q, 0);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(L, D);
      auto acc_acquire = [&](int n) -> bool {
        const int buf = n % NBUF, kb = n / NBUF;
        if (!mbar_wait(&sm.acc_empty[buf], (uint32_t)((kb & 1) ^ 1), abort, status)) return false;
        tc_fence_after();
        return true;
      };
      auto unit_wait = [&](int g) -> bool {
        if (!mbar_wait(&sm.full[g % NHS], (uint32_t)((g / NHS) & 1), abort, status)) return false;
        tc_fence_after();
        return true;
      };
      // Descriptors: a tile's descriptor plus (byte offset >> 4) addresses a
      // later part of it (shared-memory addresses stay below 2^18).  K step kk
      // of a K-major 128-row tile pair: k-half kk / 4, 32 bytes per step.
      const uint64_t qd0 = desc_kmajor_sw128(smem_u32(sm.Q[0][0]));
      const uint64_t qd1 = desc_kmajor_sw128(smem_u32(sm.Q[1][0]));
      const uint64_t hd0 = desc_kmajor_sw128(smem_u32(sm.hs[0][0]));
      constexpr uint64_t kStage = (2 * kTile) >> 4;
      auto kstep = [](int kk) -> uint64_t { return (uint64_t)((kk >> 2) * (kTile >> 4) + (kk & 3) * 2); };
      bool ok = mbar_wait(&sm.bar_q, 0, abort, status) && unit_wait(0) && (!hasB || unit_wait(1));
      if (ok) {  // P = Q K^T (accumulator 0; buffer 0 is fresh)
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          mma_bf16(tmem, qd0 + kstep(kk), hd0 + kstep(kk), idesc, kk > 0);
          if (hasB) mma_bf16(tmem + 128u, qd1 + kstep(kk), hd0 + kStage + kstep(kk), idesc, kk > 0);
        }
        mma_commit(&sm.acc_full[0]);
      }
      // O = Pt V (accumulator 1; buffer 1 is fresh): Pt over the K tiles
      // (stages 0, 1, written by the epilogue), V in stages 2, 3 as loaded:
      // [s][j], the MN-major B operand (K step: 16 rows of 128 bytes)
      if (ok && (ok = mbar_wait(&sm.bar_pt, 0, abort, status)) && (ok = unit_wait(2)) && (!hasB || (ok = unit_wait(3)))) {
        constexpr uint32_t idesc_v = idesc_bf16_f32_bmn(L, D);
        const uint64_t vd0 = desc_mnmajor_sw128(smem_u32(sm.hs[2][0]), kTile);
        const uint64_t vd1 = desc_mnmajor_sw128(smem_u32(sm.hs[3][0]), kTile);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          mma_bf16(tmem + 256u, hd0 + kstep(kk), vd0 + (uint64_t)(kk * (2048 >> 4)), idesc_v, kk > 0);
          if (hasB) mma_bf16(tmem + 384u, hd0 + kStage + kstep(kk), vd1 + (uint64_t)(kk * (2048 >> 4)), idesc_v, kk > 0);
        }
        mma_commit(&sm.acc_full[1]);
      }
      for (int i = 0; i < NHS; ++i) mma_commit(&sm.empty[i]);  // every stage is free once O is done
      // the state products, fp16 Q (converted by the epilogue before bar_pt) and fp16 states
      constexpr uint32_t idesc_h = idesc_f16_f32(L, D);
      for (int x = 0; ok && x < nu; ++x) {
        const int buf = x % NBUF;
        const bool inA = sm.uxa[x] >= 0, inB = hasB && sm.uxb[x] >= 0;
        if (!(ok = acc_acquire(x + 2))) break;
        const uint32_t dA = tmem + 256u * buf, dB = dA + 128u;
        const int g = 4 + x, hsi = g % NHS;
        if (!(ok = unit_wait(g))) break;
        const uint64_t bd = hd0 + (uint64_t)hsi * kStage;
        if (inA && inB) {
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            mma_bf16(dA, qd0 + kstep(kk), bd + kstep(kk), idesc_h, kk > 0);
            mma_bf16(dB, qd1 + kstep(kk), bd + kstep(kk), idesc_h, kk > 0);
          }
        } else if (inA || inB) {
          const uint32_t dd = inA ? dA : dB;
          const uint64_t qd = inA ? qd0 : qd1;
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) mma_bf16(dd, qd + kstep(kk), bd + kstep(kk), idesc_h, kk > 0);
        }
        mma_commit(&sm.empty[hsi]);
        mma_commit(&sm.acc_full[buf]);
      }
      mma_commit(&sm.bar_done);  // every MMA issued above has completed once this fires
      mbar_wait_drain(&sm.bar_done, 0);
    }
  } else {
    // ------------------------------------------------------------ epilogue warps
    // 16 warps: warp w reads TMEM lane quadrant w % 4; epilogue warp ew = w - 2
    // owns interval (ew / 4) % 2 and the 64-column half ew / 8 of its rows.
    const int ew = warp - 2;              // 0..15
    const int quad = warp & 3;            // TMEM lane quadrant of this warp
    const int side = (ew >> 2) & 1;       // interval A (0) or B (1)
    const int ch = ew >> 3;               // column half
    const int t = quad * 32 + lane;       // token row of this thread
    const uint32_t lane_addr = tmem + ((uint32_t)(quad * 32) << 16);
    const int etid = ew * 32 + lane;      // 0..511
    const int c0s = c0_of(side), Lcs = Lc_of(side);
    const bool side_in = (side == 0 || hasB);  // warp-uniform
    const long long rowbase = (tok0 + c0s) * a.H + h;

    if (etid < 2 * L) {  // both intervals' boundary flags and merge indices
      const int sd = etid / L, tt = etid % L;
      const bool in = tt < Lc_of(sd);
      const long long tr = (long long)bh * a.T + c0_of(sd) + tt;
      sm.side[sd].bnd[tt] = in ? __ldcg(a.boundary + tr) : (uint8_t)0;
      sm.side[sd].mlog[tt] = in ? __ldcg(a.merge_log + tr) : -1;
    }
    asm volatile("bar.sync 1, 512;" ::: "memory");
    if constexpr (!kBig) {
      if (ew == 0) build_intra_table(sm.side[0], sm.tab[0], sm.logi[0], m0A, lane);
      if (ew == 4 && hasB) build_intra_table(sm.side[1], sm.tab[1], sm.logi[1], m0B, lane);
    }
    if (etid < 2 * L) {
      const int sd = etid / L, tt = etid % L;
      sm.side[sd].evt[tt] = events_before(sm.side[sd], tt, lane);
    }
    asm volatile("bar.sync 1, 512;" ::: "memory");
    const float* lam_t = (a.lam && t < Lcs) ? a.lam + (rowbase + (long long)t * a.H) * C : nullptr;
    // lambda is read-only while the kernel runs (the read-only path), except when
    // the host streams it in beside the work (then through L2)
    auto lam_at = [&](int i) -> float {
      if constexpr (kStream) return __ldcg(lam_t + i);
      else return __ldg(lam_t + i);
    };
    const int evt_t = sm.side[side].evt[t];
    // an interval without boundary events (the common case) weights every
    // column s <= t of row t by lambda of the open entry: loaded ahead of P
    const bool no_ev = sm.side[side].evt[L - 1] == 0;  // warp-uniform
    const int m0s = side ? m0B : m0A;
    // slot, after this row's events, of the entry opened at event e (0: the open entry)
    auto intra_slot = [&](const unsigned char* trow_, int e) -> int {
      if constexpr (kBig) return min(m0s - 1 + e, C - 1);  // a consistent trace stays below C
      else return trow_[e];
    };
    const float w_open = (no_ev && t < Lcs) ? (lam_t ? lam_at(intra_slot(sm.tab[side], 0)) : 1.f) : 0.f;
    bool ok;
    {  // P (accumulator 0) -> Pt over this interval's K tile (its MMAs are complete)
      ok = __all_sync(0xffffffffu, mbar_wait(&sm.acc_full[0], 0, abort, status));
      if (ok && side_in) {
        tc_fence_after();
        const uint32_t base = lane_addr + 128u * side + 64 * ch;
        // the weight of column s depends on s only through evt[s], which changes
        // at the interval's boundaries: it is looked up again only then
        const unsigned char* trow = kBig ? sm.tab[side] : sm.tab[side] + evt_t * (evt_t + 1) / 2;
        const int* evs = sm.side[side].evt;
        int last_e = -1;
        float last_w = 0.f;
        uint8_t* ptile = sm.hs[side][ch];
#pragma unroll
        for (int c = 0; c < 64; c += 16) {
          float p[16];
          tmem_ld16(base + c, p);
#pragma unroll
          for (int h8 = 0; h8 < 2; ++h8) {
            uint32_t packed[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              float w2[2];
#pragma unroll
              for (int u = 0; u < 2; ++u) {
                const int ss = 64 * ch + c + 8 * h8 + 2 * i + u;
                float wt = 0.f;
                if (no_ev) {
                  wt = (ss <= t) ? w_open : 0.f;
                } else if (ss <= t && t < Lcs) {
                  const int e = evs[ss];
                  if (e != last_e) {
                    last_e = e;
                    last_w = lam_t ? lam_at(intra_slot(trow, e)) : 1.f;
                  }
                  wt = last_w;
                }
                w2[u] = p[8 * h8 + 2 * i + u] * wt;
              }
              const __nv_bfloat162 pr = __floats2bfloat162_rn(w2[0], w2[1]);
              packed[i] = *reinterpret_cast<const uint32_t*>(&pr);
            }
            const int c8 = (c >> 3) + h8;  // 16-byte chunk of the row
            *reinterpret_cast<uint4*>(ptile + t * 128 + ((c8 ^ (t & 7)) << 4)) =
                make_uint4(packed[0], packed[1], packed[2], packed[3]);
          }
        }
      }
    }
    // This row's half of Q into fp16 in place (the P MMAs, the only bf16 use of Q,
    // are complete): a power-of-two scale per row, agreed on by the two k-halves
    // through qmax, keeps every element below 2^14 and in fp16's normal range
    // (bf16 values fit fp16's significand, so only values below 2^-14 of the
    // row's scale round); the epilogue multiplies D by its inverse, qinv.
    float qinv = 1.f;
    {
      uint8_t* qtile = sm.Q[side][ch];
      const bool conv = ok && side_in;  // warp-uniform
      float mx = 0.f;
      if (conv) {
#pragma unroll
        for (int c8 = 0; c8 < 8; ++c8) {
          const uint4 w = *reinterpret_cast<const uint4*>(qtile + t * 128 + ((c8 ^ (t & 7)) << 4));
          const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&ws[i]));
            mx = fmaxf(mx, fmaxf(fabsf(f.x), fabsf(f.y)));
          }
        }
      }
      sm.qmax[side][ch][t] = mx;
      asm volatile("bar.sync 1, 512;" ::: "memory");
      if (conv) {
        const float rm = fmaxf(sm.qmax[side][0][t], sm.qmax[side][1][t]);
        int ex = 0;
        if (rm > 0.f) frexpf(rm, &ex);  // rm < 2^ex
        const float sc = ldexpf(1.f, 14 - ex);
        qinv = ldexpf(1.f, ex - 14);
#pragma unroll
        for (int c8 = 0; c8 < 8; ++c8) {
          uint4* ptr = reinterpret_cast<uint4*>(qtile + t * 128 + ((c8 ^ (t & 7)) << 4));
          const uint4 w = *ptr;
          uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&ws[i]));
            const __half2 hh = __floats2half2_rn(f.x * sc, f.y * sc);
            ws[i] = *reinterpret_cast<const uint32_t*>(&hh);
          }
          *ptr = make_uint4(ws[0], ws[1], ws[2], ws[3]);
        }
      }
      fence_proxy_async();  // the generic-proxy writes (Pt, fp16 Q) feed the tensor core
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&sm.acc_empty[0]);
        mbar_arrive(&sm.bar_pt);
      }
    }
    asm volatile("bar.sync 1, 512;" ::: "memory");  // every warp is past the intra tables
    if constexpr (!kBig) {
      if (ew == 0) build_snap_table(sm.side[0], sm.tab[0], sm.logi[0], m0A, lane);
      if (ew == 4) build_snap_table(sm.side[1], sm.tab[1], sm.logi[1], m0B, lane);
    }
    asm volatile("bar.sync 1, 512;" ::: "memory");
    float o[64];
    {  // o starts from O (accumulator 1)
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&sm.acc_full[1], 0, abort, status));
      if (ok && side_in) {
        tc_fence_after();
        const uint32_t base = lane_addr + 256u + 128u * side + 64 * ch;
#pragma unroll
        for (int c = 0; c < 64; c += 16) tmem_ld16(base + c, o + c);
      } else {
#pragma unroll
        for (int i = 0; i < 64; ++i) o[i] = 0.f;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.acc_empty[1]);
    }
    const int* ux = side ? sm.uxb : sm.uxa;
    {  // snapshot part
      const unsigned char* tab_t = sm.tab[side] + (kBig ? 0 : evt_t * kMaxC);
      // weight of union state x for this token (0 when not in its interval's list):
      // lambda times the entry's scale s_x and the row's inverse Q scale
      auto weight = [&](int x) -> float {
        if (x >= nu || t >= Lcs) return 0.f;
        const int xi = ux[x];
        if (xi < 0) return 0.f;
        return (lam_t ? lam_at(kBig ? xi : (int)tab_t[xi]) : 1.f) * sm.uscale[x] * qinv;
      };
      float wn = weight(0);
      for (int x = 0; ok && x < nu; ++x) {
        const int n = x + 2, buf = n % NBUF, kb = n / NBUF;
        const bool in = side_in && ux[x] >= 0;  // warp-uniform
        const float wx = wn;
        wn = weight(x + 1);
        // tcgen05.ld below is warp-wide: the warp takes one decision
        if (!(ok = __all_sync(0xffffffffu, mbar_wait(&sm.acc_full[buf], (uint32_t)(kb & 1), abort, status)))) break;
        tc_fence_after();
        if (in) {
          float dv[16];
          const uint32_t base = lane_addr + 256u * buf + 128u * side + 64 * ch;
#pragma unroll
          for (int c = 0; c < 64; c += 16) {
            tmem_ld16(base + c, dv);
#pragma unroll
            for (int i = 0; i < 16; ++i) o[c + i] += wx * dv[i];
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.acc_empty[buf]);
      }
    }
    // fp32 output of the common instance: staged in the ring stages (free once
    // every state product is complete, which this warp has seen) in the
    // 128-byte swizzle and stored by TMA, eight 128-row x 32-column tiles per
    // CTA (rows past T are clipped); otherwise per-row stores
    bool tma_out = false;
    if constexpr (!kStream && !kRagged) tma_out = (a.out_bf16 == 0);
    if (tma_out) {
      if (ok && side_in) {
#pragma unroll
        for (int cbl = 0; cbl < 2; ++cbl) {
          const int box = side * 4 + 2 * ch + cbl;
          uint8_t* tile = sm.hs[box >> 1][box & 1];
#pragma unroll
          for (int c = 0; c < 8; ++c)
            *reinterpret_cast<float4*>(tile + t * 128 + ((c ^ (t & 7)) << 4)) =
                make_float4(o[32 * cbl + 4 * c], o[32 * cbl + 4 * c + 1], o[32 * cbl + 4 * c + 2], o[32 * cbl + 4 * c + 3]);
        }
      }
      fence_proxy_async();  // the staged output feeds the TMA engine
      asm volatile("bar.sync 1, 512;" ::: "memory");
      if (ew == 0 && lane == 0 && !*abort) {
        for (int box = 0; box < (hasB ? 8 : 4); ++box)
          tma_store_4d(&tmO, sm.hs[box >> 1][box & 1], 32 * (box & 3), h, tma_t + c0_of(box >> 2), tma_b);
        bulk_commit();
        bulk_wait0();  // the CTA's shared memory stays valid until the stores are done
      }
    } else if (ok && !*abort && side_in && t < Lcs) {
      const long long orow = (rowbase + (long long)t * a.H) * D + 64 * ch;
      if (a.out_bf16) {
        __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(a.o) + orow;
#pragma unroll
        for (int i = 0; i < 64; i += 4) store4(out + i, make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]));
      } else {
        float* out = reinterpret_cast<float*>(a.o) + orow;
#pragma unroll
        for (int i = 0; i < 64; i += 4) store4(out + i, make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]));
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
  // every CTA reaches this point, also after a failed wait: the host's copy of
  // the output piece waits for the count of its CTAs
  if constexpr (kStream) {
    if (a.out_done && tid == 0) {
      __threadfence();
      atomicAdd(a.out_done + pair / a.out_piece_pairs, 1);
    }
  }
}

// ---------------------------------------------------------------- host side
cudaError_t launch_readout_tc(const ReadoutArgs& a, int32_t* status, cudaStream_t st) {
  CUtensorMap mq, mk, mv, ms, mo;
  const long long rows = (long long)a.B * a.H * a.pool_cap * D;  // fp16 entries of D rows
  // packed layout: one batch coordinate over all token rows
  const int mb = a.row_start ? 1 : a.B;
  const long long mt = a.row_start ? (a.total_rows > 0 ? a.total_rows : 1) : a.T;
  if (mt >= (1LL << 31)) return cudaErrorInvalidValue;
  if (!tmap_tokens(&mq, a.q, mb, (int)mt, a.H) || !tmap_tokens(&mk, a.k, mb, (int)mt, a.H) ||
      !tmap_tokens(&mv, a.v, mb, (int)mt, a.H) || !tmap_pool(&ms, a.pool, rows, true))
    return cudaErrorInvalidValue;
  if (a.row_start && !a.seq_lens) return cudaErrorInvalidValue;  // the packed layout needs per-row lengths
  const bool big = a.C > kMaxC;  // DLA(I): device-resident whole rows only
  const size_t smem = big ? sizeof(TcSmem<kMaxCBig>) + 1024 : sizeof(TcSmem<kMaxC>) + 1024;
  const bool stream = a.lam_l2 || a.out_done, ragged = a.seq_lens != nullptr;
  if (big && (stream || ragged || a.C > kMaxCBig)) return cudaErrorInvalidValue;
  auto kern = big ? readout_tc_kernel<false, false, kMaxCBig>
                  : stream ? (ragged ? readout_tc_kernel<true, true> : readout_tc_kernel<true, false>)
                           : (ragged ? readout_tc_kernel<false, true> : readout_tc_kernel<false, false>);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  if ((a.nsnap + 1) / 2 > 65535) return cudaErrorInvalidConfiguration;
  dim3 grid(a.B * a.H, (a.nsnap + 1) / 2);  // streams x pairs of intervals
  // the common instance stores an fp32 output by TMA (the map is unused otherwise)
  if (!stream && !ragged && !a.out_bf16) {
    if (!tmap_out_f32(&mo, a.o, a.B, a.T, a.H)) return cudaErrorInvalidValue;
  } else {
    mo = mq;
  }
  kern<<<grid, NT, smem, st>>>(a, mq, mk, mv, ms, mo, status);
  return cudaGetLastError();
}

size_t readout_tc_smem_bytes() { return sizeof(TcSmem<kMaxCBig>) + 1024; }

cudaError_t preload_readout_kernels() {
  cudaFuncAttributes fa;
  cudaError_t e;
  if ((e = cudaFuncGetAttributes(&fa, readout_tc_kernel<false, false>)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, readout_tc_kernel<true, false>)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, readout_tc_kernel<false, true>)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, readout_tc_kernel<true, true>)) != cudaSuccess) return e;
  return cudaFuncGetAttributes(&fa, readout_tc_kernel<false, false, kMaxCBig>);
}

}  // namespace dla

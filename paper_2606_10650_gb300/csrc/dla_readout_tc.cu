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
// One CTA per (interval, stream), sized so that two CTAs share an SM (about
// 110 KB of shared memory and 256 TMEM columns each): one CTA's fixed phases
// (tables, the intra part, the output) run while the other's state products
// keep the tensor core busy.  K1 stores each snapshot as S_x / s_x in fp16 (s_x
// a power of two from a bound of |S_x|_F, so that no element overflows and
// every element keeps 2^-12 relative rounding).  The weights are folded into
// the A operand, so that the interval keeps one accumulator over all its
// states: with q~_t = q_t 2^(14 - e_t) the row's fp16 image (exact: bf16 values
// fit fp16's significand) and s_ref the largest s_x of the list,
//   o_t = qinv_t s_ref sum_x A_x[t] . (S_x / s_x)[:, :],
//   A_x[t] = fp16(lambda_{t, L_t(x)} (s_x / s_ref) q~_t),   qinv_t = 2^(e_t - 14),
// one fp16 MMA chain (M = 128 tokens, N = 128, K = 128 per state) with A in
// tensor memory.  A_x is formed in fp16 arithmetic (the weight rounded to fp16,
// then the product): at most two roundings of 2^-11 relative each (plus fp16's
// absolute spacing of 2^-24 for weights far below s_ref, i.e. states far
// smaller than the largest), beside the entry's 2^-12.  The intra part comes
// first and starts the same accumulator: P = Q K^T, Pt = P o W (W_ts =
// lambda_{t, L_t(e(s))} for s <= t, else 0) scaled by 1 / (qinv_t s_ref) (a
// power of two) and written as bf16 over the K tile, O = Pt V with V as loaded
// (an MN-major operand).
// Roles: warp 0 issues TMA loads (Q, K and V, then each state of the list, 32
// KB in fp16, through three 32 KB stages); one thread of warp 1 issues
// tcgen05.mma; warps 2..9 (one token row and one 64-wide half of q per thread;
// warp w reads TMEM lane quadrant w % 4) form Pt and, per state, the A operand
// in TMEM slot x % 2, and finally read the accumulator out.  An issuing thread
// that waits on an mbarrier starves the tensor core, so the issuer takes one
// wait (`ready`: the A operand written and the state's tile landed, signalled
// by the epilogue warps) and one commit (the tile's stage, which also frees
// the TMEM slot for the state two later) per state.  All waits are bounded
// (~2 s, then an abort flag and status 5).
#include "dla_common.cuh"
#include "dla_sm100.cuh"
#include "dla_tmap.h"

namespace dla {

namespace {

using namespace sm100;

constexpr int L = 128;   // tokens per interval
constexpr int D = 128;   // head dimension
constexpr int NT = 320;  // 10 warps
constexpr int NEPI = 8;  // epilogue warps
constexpr int NHS = 3;   // shared-memory stages (32 KB: Q, K then Pt, V, then states)
// TMEM: P = Q K^T at columns 0..127 during the intra part, then the same
// columns hold the weighted-Q A operands, two 64-column slots; the output
// accumulator at 128..255 (Pt V, then every state product added).
constexpr uint32_t kColO = 128;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kTile = L * 128;  // one K-major 128B-swizzled tile: 128 rows x 64 bf16
constexpr int kRows = L + 1;         // events 0 .. L of an interval
// Slot tables of the interval, in one region: first the intra part's tab[e][i]
// for the entry opened at event i <= e (row e at e (e + 1) / 2), later the
// snapshot entries' slots tab[e][x] (row stride kMaxC).
constexpr int kSnapTab = kRows * kMaxC;
constexpr int kIntraTab = kRows * (kRows + 1) / 2;
constexpr int kTabBytes = kSnapTab > kIntraTab ? kSnapTab : kIntraTab;

struct Side {      // the interval's trace
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
  uint8_t hs[NHS][2][kTile];   // [stage][k-half]: Q, K (then Pt), V; the states; finally the output   96 KB
  unsigned char tab[kBig ? 16 : kTabBytes];
  Side side;
  int ids[CAPB];               // pool ids of the list
  float uscale[CAPB];          // scale s_x of each entry (S_x / s_x is stored)
  float qmax[2][L];            // [k-half][row]: max |q| of the half row (Q's fp16 scales)
  int logi[kRows];             // table-build scratch
  float sref;                  // the largest s_x of the list (1 if empty)
  uint64_t full[NHS], empty[NHS];
  uint64_t bar_p, bar_pt, bar_done;
  uint64_t qfree;              // the epilogue holds Q in registers: stage 0 may take state 0
  uint64_t ready[2];           // state x: its A operand in slot x % 2 and its tile landed
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

// Two CTAs per SM: 20 warps share the four sub-partitions, so a thread gets at
// most 96 registers.
// kStream: inputs streamed in by the host while the kernel runs (lambda read
// through L2) and the output copied back piece by piece (per-piece CTA counts).
// kRagged: per-row lengths (padding after them).  Separate instances, so the
// common one keeps its code unchanged.
template <bool kStream, bool kRagged, int CAPB = kMaxC>
__global__ void __launch_bounds__(NT, 2)
    readout_tc_kernel(ReadoutArgs a, const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmS,
                      const __grid_constant__ CUtensorMap tmO, int32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  using Smem = TcSmem<CAPB>;
  constexpr bool kBig = Smem::kBig;
  Smem& sm = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int bh = blockIdx.x, si = blockIdx.y;  // streams fastest: CTAs dispatched interval by interval
  const int b = bh / a.H, h = bh % a.H;
  const int C = a.C;
  // Streamed output: each CTA counts in the piece of its interval pair
  auto count_done = [&](bool fence) {
    if constexpr (kStream) {
      if (a.out_done && tid == 0) {
        if (fence) __threadfence();
        atomicAdd(a.out_done + (si / 2) / a.out_piece_pairs, 1);
      }
    }
  };
  // token row of the row's token 0, and the TMA coordinates of it: (token, batch)
  // = (t, b) in the padded layout, (row_start[b] + t, 0) in the packed one (the
  // per-row-length instance only)
  const long long tok0 = kRagged ? row_tok0(a.row_start, b, a.T) : (long long)b * a.T;
  const bool packed = kRagged && a.row_start != nullptr;
  const int tma_t = packed ? (int)tok0 : 0, tma_b = packed ? 0 : b;
  // this row's end (padding after it)
  const int t_end = kRagged ? row_t_end(a.seq_lens, b, a.t_begin, a.t_end) : a.t_end;
  const int c0 = a.t_begin + si * L;
  if constexpr (kRagged) {
    if (c0 >= t_end) {  // the interval lies past the row's length: o not written
      count_done(false);
      return;
    }
  }
  // with a scan running concurrently: the interval must be complete
  wait_progress(a.progress, a.progress_ctas, bh, a.snap_base + si + 1, a.status);
  if (tid == 0) {
    // thread 0 issues the TMA loads: they read what the scan wrote (pool entries)
    // and the inputs streamed in before its progress
    if (a.progress) asm volatile("fence.proxy.async.global;" ::: "memory");
    // A failed call (a bounded wait that gave up, here or in another kernel, or a
    // device check): the scan may not have written this interval's list, so the
    // CTA does none of the work and leaves o unwritten.
    sm.skip = (*(volatile int32_t*)a.status != 0);
  }
  __syncthreads();
  if (sm.skip) {
    count_done(false);
    return;
  }
  const int Lc = min(L, t_end - c0);
  const long long lrow = (long long)bh * a.snap_stride + a.snap_base + si;
  // list and trace come from the scan: read past L1 (__ldcg).  Live entries of
  // the list, checked against the capacity (a violation is a device-check
  // failure and is clamped, so that nothing indexes out of bounds)
  int m0 = __ldcg(a.snap_m0 + lrow);
  if (m0 < 0 || m0 > C) {
    if (tid == 0) atomicCAS(a.status, 0, 6);
    m0 = min(max(m0, 0), C);
  }
  volatile int* abort = &sm.abort_flag;

  if (tid == 0) {
    mbar_init(&sm.bar_p, 1);
    mbar_init(&sm.bar_pt, NEPI);
    mbar_init(&sm.bar_done, 1);
    for (int i = 0; i < NHS; ++i) {
      mbar_init(&sm.full[i], 1);
      mbar_init(&sm.empty[i], 1);
    }
    for (int j = 0; j < 2; ++j) mbar_init(&sm.ready[j], NEPI);
    mbar_init(&sm.qfree, NEPI);
    sm.abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
    prefetch_tmap(&tmS);
    // units 0, 1, 2: the Q, K and V tiles, each in the stage of its number
    auto load_unit = [&](int g, const CUtensorMap* map) {
      mbar_expect_tx(&sm.full[g], 2 * kTile);
      tma_load_4d(sm.hs[g][0], map, &sm.full[g], 0, h, tma_t + c0, tma_b);
      tma_load_4d(sm.hs[g][1], map, &sm.full[g], 64, h, tma_t + c0, tma_b);
    };
    load_unit(0, &tmQ);
    load_unit(1, &tmK);
    load_unit(2, &tmV);
  }
  if (warp == 0) {  // pool ids and scales of the list, and s_ref
    float smax = 0.f;
    for (int x = lane; x < CAPB; x += 32) {
      int id = -1;
      float sc = 1.f;
      if (x < m0) {
        id = __ldcg(a.snap_ids + lrow * C + x);
        if (id < 0 || id >= a.pool_cap) {  // a pool id outside the pool
          atomicCAS(a.status, 0, 6);
          id = 0;
        }
        sc = __ldcg(a.pool_scale + (long long)bh * a.pool_cap + id);
        smax = fmaxf(smax, sc);
      }
      sm.ids[x] = id;
      sm.uscale[x] = sc;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) smax = fmaxf(smax, __shfl_xor_sync(0xffffffffu, smax, off));
    // the scales are powers of two, so s_x / s_ref is exact
    if (lane == 0) sm.sref = smax > 0.f ? smax : 1.f;
  } else if (warp == 1) {
    tmem_alloc(&sm.tmem_base, kTmemCols);
  } else if (tid - 64 < L) {  // the interval's boundary flags and merge indices
    const int tt = tid - 64;
    const bool in = tt < Lc;
    const long long tr = (long long)bh * a.T + c0 + tt;
    sm.side.bnd[tt] = in ? __ldcg(a.boundary + tr) : (uint8_t)0;
    sm.side.mlog[tt] = in ? __ldcg(a.merge_log + tr) : -1;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int issued[NHS];  // uses of each stage so far
      for (int i = 0; i < NHS; ++i) issued[i] = 1;
      for (int x = 0; x < m0; ++x) {
        const int g = 3 + x, hsi = g % NHS, k = g / NHS;
        // state 0 takes Q's stage as soon as P is complete and the epilogue holds
        // Q in registers; later states wait for the MMAs of the stage's last use
        if (!mbar_wait(x == 0 ? &sm.qfree : &sm.empty[hsi], x == 0 ? 0u : (uint32_t)((k & 1) ^ 1), abort, status))
          break;
        mbar_expect_tx(&sm.full[hsi], 2 * kTile);
        const int row = (int)(((long long)bh * a.pool_cap + sm.ids[x]) * D);
        tma_load_2d(sm.hs[hsi][0], &tmS, &sm.full[hsi], 0, row);
        tma_load_2d(sm.hs[hsi][1], &tmS, &sm.full[hsi], 64, row);
        issued[hsi] = k + 1;
      }
      if (*abort) {  // let copies in flight land before the CTA exits
        for (int i = 0; i < NHS; ++i) mbar_wait_drain(&sm.full[i], (uint32_t)((issued[i] - 1) & 1));
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(L, D);
      auto unit_wait = [&](int g) -> bool {
        if (!mbar_wait(&sm.full[g % NHS], (uint32_t)((g / NHS) & 1), abort, status)) return false;
        tc_fence_after();
        return true;
      };
      // Descriptors: a tile's descriptor plus (byte offset >> 4) addresses a
      // later part of it (shared-memory addresses stay below 2^18).  K step kk
      // of a K-major 128-row tile pair: k-half kk / 4, 32 bytes per step.
      const uint64_t hd0 = desc_kmajor_sw128(smem_u32(sm.hs[0][0]));
      constexpr uint64_t kStage = (2 * kTile) >> 4;
      auto kstep = [](int kk) -> uint64_t { return (uint64_t)((kk >> 2) * (kTile >> 4) + (kk & 3) * 2); };
      // A commit stands only behind MMAs of this thread: after a failed wait
      // with none issued, the thread arrives on the barrier instead.
      bool issued = false;
      auto release = [&](uint64_t* bar) {
        if (issued) mma_commit(bar);
        else mbar_arrive(bar);
      };
      bool ok = unit_wait(0) && unit_wait(1);
      if (ok) {  // P = Q K^T (columns 0..127): Q in stage 0, K in stage 1
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) mma_bf16(tmem, hd0 + kstep(kk), hd0 + kStage + kstep(kk), idesc, kk > 0);
        issued = true;
        mma_commit(&sm.bar_p);
      }
      // O = Pt V (columns 128..255): Pt over the K tile (stage 1, written by the
      // epilogue), V in stage 2 as loaded: [s][j], the MN-major B operand (K
      // step: 16 rows of 128 bytes)
      if (ok && (ok = mbar_wait(&sm.bar_pt, 0, abort, status)) && (ok = unit_wait(2))) {
        constexpr uint32_t idesc_v = idesc_bf16_f32_bmn(L, D);
        const uint64_t vd = desc_mnmajor_sw128(smem_u32(sm.hs[2][0]), kTile);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          mma_bf16(tmem + kColO, hd0 + kStage + kstep(kk), vd + (uint64_t)(kk * (2048 >> 4)), idesc_v, kk > 0);
      }
      for (int i = 0; i < NHS; ++i) release(&sm.empty[i]);  // every stage is free once O is done
      // The state products, added to O: A = the weighted fp16 Q (TMEM slot
      // x % 2, written by the epilogue: one row per lane, two fp16 per column,
      // K step 8 columns), B = the fp16 state (shared memory).
      constexpr uint32_t idesc_h = idesc_f16_f32(L, D);
      for (int x = 0; ok && x < m0; ++x) {
        const int j = x & 1, hsi = (3 + x) % NHS;
        if (!(ok = mbar_wait(&sm.ready[j], (uint32_t)((x >> 1) & 1), abort, status))) break;
        tc_fence_after();
        const uint64_t bd = hd0 + (uint64_t)hsi * kStage;
        const uint32_t ad = tmem + 64u * j;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) mma_ts(tmem + kColO, ad + 8u * kk, bd + kstep(kk), idesc_h, 1u);
        mma_commit(&sm.empty[hsi]);  // the tile's stage, and TMEM slot j for state x + 2
      }
      release(&sm.bar_done);  // every MMA issued above has completed once this fires
      mbar_wait_drain(&sm.bar_done, 0);
    }
  } else {
    // ------------------------------------------------------------ epilogue warps
    // 8 warps: warp w reads TMEM lane quadrant w % 4; epilogue warp ew = w - 2
    // owns the 64-column half ew / 4 of its token rows.
    const int ew = warp - 2;              // 0..7
    const int quad = warp & 3;            // TMEM lane quadrant of this warp
    const int ch = ew >> 2;               // column half
    const int t = quad * 32 + lane;       // token row of this thread
    const uint32_t lane_addr = tmem + ((uint32_t)(quad * 32) << 16);
    const int etid = ew * 32 + lane;      // 0..255
    const long long rowbase = (tok0 + c0) * a.H + h;
    if constexpr (!kBig) {
      if (ew == 0) build_intra_table(sm.side, sm.tab, sm.logi, m0, lane);
    }
    if (etid < L) sm.side.evt[etid] = events_before(sm.side, etid, lane);
    asm volatile("bar.sync 1, 256;" ::: "memory");
    const float* lam_t = (a.lam && t < Lc) ? a.lam + (rowbase + (long long)t * a.H) * C : nullptr;
    // lambda is read-only while the kernel runs (the read-only path), except when
    // the host streams it in beside the work (then through L2)
    auto lam_at = [&](int i) -> float {
      if constexpr (kStream) return __ldcg(lam_t + i);
      else return __ldg(lam_t + i);
    };
    const int evt_t = sm.side.evt[t];
    // an interval without boundary events (the common case) weights every
    // column s <= t of row t by lambda of the open entry: loaded ahead of P
    const bool no_ev = sm.side.evt[L - 1] == 0;  // warp-uniform
    // slot, after this row's events, of the entry opened at event e (0: the open entry)
    auto intra_slot = [&](const unsigned char* trow_, int e) -> int {
      if constexpr (kBig) return min(m0 - 1 + e, C - 1);  // a consistent trace stays below C
      else return trow_[e];
    };
    const float w_open = (no_ev && t < Lc) ? (lam_t ? lam_at(intra_slot(sm.tab, 0)) : 1.f) : 0.f;
    // P = Q K^T is complete, so the Q and K tiles have landed
    bool ok = __all_sync(0xffffffffu, mbar_wait(&sm.bar_p, 0, abort, status));
    // This row's half of Q in fp16 registers: a power-of-two scale per row,
    // agreed on by the two k-halves through qmax, keeps every element below
    // 2^14 and in fp16's normal range (bf16 values fit fp16's significand, so
    // only values below 2^-14 of the row's scale round); the output is
    // multiplied back by its inverse, qinv.  Column c of the half row holds the
    // elements 2c, 2c + 1 (the layout of an A operand in tensor memory).
    uint32_t qh[32];
    float qinv = 1.f, fpt = 1.f;
    const float sref = sm.sref, rsref = 1.f / sref;  // powers of two
    {
      const uint8_t* qtile = sm.hs[0][ch];
      float mx = 0.f;
#pragma unroll
      for (int c8 = 0; c8 < 8; ++c8) {
        uint4 w = make_uint4(0u, 0u, 0u, 0u);
        if (ok) w = *reinterpret_cast<const uint4*>(qtile + t * 128 + ((c8 ^ (t & 7)) << 4));
        qh[4 * c8] = w.x;
        qh[4 * c8 + 1] = w.y;
        qh[4 * c8 + 2] = w.z;
        qh[4 * c8 + 3] = w.w;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&qh[4 * c8 + i]));
          mx = fmaxf(mx, fmaxf(fabsf(f.x), fabsf(f.y)));
        }
      }
      sm.qmax[ch][t] = mx;
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.qfree);  // this warp's reads of the Q tile are done
      asm volatile("bar.sync 1, 256;" ::: "memory");
      const float rm = fmaxf(sm.qmax[0][t], sm.qmax[1][t]);
      int ex = 0;
      if (rm > 0.f) frexpf(rm, &ex);  // rm < 2^ex
      const float sc = ldexpf(1.f, 14 - ex);
      qinv = ldexpf(1.f, ex - 14);
      fpt = sc * rsref;
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&qh[i]));
        const __half2 hh = __floats2half2_rn(f.x * sc, f.y * sc);
        qh[i] = *reinterpret_cast<const uint32_t*>(&hh);
      }
    }
    {  // P -> Pt over the K tile, in the accumulator's units: row t scaled by
       // 2^(14 - ex) / s_ref (a power of two, so no extra rounding)
      // a warp whose rows all lie before its 64 columns (rows 0..63, columns
      // 64..127) writes zeros without reading P
      const bool upper = (ch == 1) && (quad < 2);  // warp-uniform
      if (ok && upper) {
        uint8_t* ptile = sm.hs[1][ch];
#pragma unroll
        for (int c8 = 0; c8 < 8; ++c8) *reinterpret_cast<uint4*>(ptile + t * 128 + (c8 << 4)) = make_uint4(0u, 0u, 0u, 0u);
      } else if (ok) {
        tc_fence_after();
        const uint32_t base = lane_addr + 64 * ch;
        // the weight of column s depends on s only through evt[s], which changes
        // at the interval's boundaries: it is looked up again only then
        const unsigned char* trow = kBig ? sm.tab : sm.tab + evt_t * (evt_t + 1) / 2;
        const int* evs = sm.side.evt;
        int last_e = -1;
        float last_w = 0.f;
        uint8_t* ptile = sm.hs[1][ch];
#pragma unroll
        for (int c = 0; c < 64; c += 16) {
          float p[16];
          tmem_ld16(base + c, p);
#pragma unroll
          for (int h8 = 0; h8 < 2; ++h8) {
            uint32_t pk[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              float w2[2];
#pragma unroll
              for (int u = 0; u < 2; ++u) {
                const int ss = 64 * ch + c + 8 * h8 + 2 * i + u;
                float wt = 0.f;
                if (no_ev) {
                  wt = (ss <= t) ? w_open : 0.f;
                } else if (ss <= t && t < Lc) {
                  const int e = evs[ss];
                  if (e != last_e) {
                    last_e = e;
                    last_w = lam_t ? lam_at(intra_slot(trow, e)) : 1.f;
                  }
                  wt = last_w;
                }
                w2[u] = (p[8 * h8 + 2 * i + u] * wt) * fpt;
              }
              const __nv_bfloat162 pr = __floats2bfloat162_rn(w2[0], w2[1]);
              pk[i] = *reinterpret_cast<const uint32_t*>(&pr);
            }
            const int c8 = (c >> 3) + h8;  // 16-byte chunk of the row
            *reinterpret_cast<uint4*>(ptile + t * 128 + ((c8 ^ (t & 7)) << 4)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
          }
        }
      }
      fence_proxy_async();  // the generic-proxy writes (Pt) feed the tensor core
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.bar_pt);
    }
    asm volatile("bar.sync 1, 256;" ::: "memory");  // every warp is past the intra table and its P reads
    if constexpr (!kBig) {
      if (ew == 0) build_snap_table(sm.side, sm.tab, sm.logi, m0, lane);
    }
    asm volatile("bar.sync 1, 256;" ::: "memory");
    {  // snapshot part: per state x of the list, the A operand
       // A_x[t] = fp16(lambda_{t, L_t(x)} (s_x / s_ref) q~_t) into TMEM slot
       // x % 2; the MMAs add A_x (S_x / s_x)^T to O
      const unsigned char* tab_t = sm.tab + (kBig ? 0 : evt_t * kMaxC);
      // lambda of state x for this row (0 past the interval's end).  With most
      // of the shared memory taken, L1 does not hold the rows of lambda, so
      // the loads are issued two states ahead of their use.
      auto lam_raw = [&](int x) -> float {
        if (x >= m0 || t >= Lc) return 0.f;
        return lam_t ? lam_at(kBig ? x : (int)tab_t[x]) : 1.f;
      };
      float l0 = lam_raw(0), l1 = lam_raw(1);
      for (int x = 0; ok && x < m0; ++x) {
        const int j = x & 1;
        const float wx = l0 * (sm.uscale[x] * rsref);
        l0 = l1;
        l1 = lam_raw(x + 2);
        // slot j is free once the MMAs of state x - 2 are complete (the commit
        // on its tile's stage, unit x + 1), and state x's tile must have landed
        bool w_ok = true;
        if (x >= 2) w_ok = mbar_wait(&sm.empty[(x + 1) % NHS], (uint32_t)(((x + 1) / NHS) & 1), abort, status);
        w_ok = w_ok && mbar_wait(&sm.full[(3 + x) % NHS], (uint32_t)(((3 + x) / NHS) & 1), abort, status);
        if (!(ok = __all_sync(0xffffffffu, w_ok))) break;
        tc_fence_after();
        const uint32_t abase = lane_addr + 64u * j + 32u * ch;
        const __half2 w2 = __float2half2_rn(wx);
#pragma unroll
        for (int cc = 0; cc < 2; ++cc) {
          float hv[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const __half2 hh = __hmul2(*reinterpret_cast<const __half2*>(&qh[16 * cc + i]), w2);
            hv[i] = __uint_as_float(*reinterpret_cast<const uint32_t*>(&hh));
          }
          tmem_st16(abase + 16u * cc, hv);
        }
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.ready[j]);
      }
    }
    // o = the accumulator times qinv s_ref, once every MMA is complete
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&sm.bar_done, 0, abort, status));
    if (ok) tc_fence_after();
    const uint32_t obase = lane_addr + kColO + 64 * ch;
    const float f = qinv * sref;
    // fp32 output of the common instance: staged in stages 0 and 1 (free once
    // every MMA is complete, which this warp has seen) in the 128-byte swizzle
    // and stored by TMA, four 128-row x 32-column tiles (rows past T are
    // clipped); otherwise per-row stores
    bool tma_out = false;
    if constexpr (!kStream && !kRagged) tma_out = (a.out_bf16 == 0);
    if (tma_out) {
      if (ok) {
#pragma unroll 1
        for (int cbl = 0; cbl < 2; ++cbl) {
          float v[32];
          tmem_ld32(obase + 32 * cbl, v);
          const int box = 2 * ch + cbl;
          uint8_t* tile = sm.hs[box >> 1][box & 1];
#pragma unroll
          for (int c = 0; c < 8; ++c)
            *reinterpret_cast<float4*>(tile + t * 128 + ((c ^ (t & 7)) << 4)) =
                make_float4(v[4 * c] * f, v[4 * c + 1] * f, v[4 * c + 2] * f, v[4 * c + 3] * f);
        }
      }
      fence_proxy_async();  // the staged output feeds the TMA engine
      asm volatile("bar.sync 1, 256;" ::: "memory");
      if (ew == 0 && lane == 0 && !*abort) {
        for (int box = 0; box < 4; ++box) tma_store_4d(&tmO, sm.hs[box >> 1][box & 1], 32 * box, h, tma_t + c0, tma_b);
        bulk_commit();
        bulk_wait_read0();  // the CTA's shared memory stays valid until the stores have read it
      }
    } else if (ok && !*abort) {  // warp-uniform: the TMEM loads are warp-wide
      float o[64];
      tmem_ld32x2(obase, obase + 32, o);
#pragma unroll
      for (int i = 0; i < 64; ++i) o[i] *= f;
      const long long orow = (rowbase + (long long)t * a.H) * D + 64 * ch;
      if (t >= Lc) {
      } else if (a.out_bf16) {
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
  count_done(true);
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
  // two CTAs per SM: the whole shared-memory carve-out
  e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
  if (e != cudaSuccess) return e;
  if (a.nsnap > 65535) return cudaErrorInvalidConfiguration;
  dim3 grid(a.B * a.H, a.nsnap);  // streams x intervals
  // the common instance stores an fp32 output by TMA (the map is unused otherwise)
  if (!stream && !ragged && !a.out_bf16) {
    if (!tmap_out_f32(&mo, a.o, a.B, a.T, a.H)) return cudaErrorInvalidValue;
  } else {
    mo = mq;
  }
  kern<<<grid, NT, smem, st>>>(a, mq, mk, mv, ms, mo, status);
  return cudaGetLastError();
}

size_t readout_tc_smem_bytes() { return sizeof(TcSmem<kMaxC>) + 1024; }

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

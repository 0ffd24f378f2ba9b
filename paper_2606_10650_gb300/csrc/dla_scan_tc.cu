// dla_scan_tc.cu -- K1 on the 5th-generation tensor cores: the sequential scan
// of Algorithm 1 / Algorithm 2 with the open state S_open (d_v x d_k, fp32) in
// tensor memory and every d x d contraction on tcgen05 (bf16 in, fp32 out),
// bf16 inputs, d = 128, one CTA per (batch, head) stream.
//
// The decisions of a 64-token chunk c need, per token t, only
//   a_t    = |k_t|^2 |v_t|^2,
//   beta_t = v_t^T S k_t over the open segment before t,
//   gamma  = |S|^2 of that segment,
// and the Gram tables of the chunk (K0: gs, Q, a).  The part of beta_t that
// comes from before the chunk is x_t = v_t^T S_open(c) k_t with S_open(c) the
// open state at the chunk's start.  If chunk c-1 had no boundary,
//   S_open(c) = S_open(c-1) + sum_{s in c-1} v_s k_s^T,
//   x_t = y_t + sum_{s in c-1} G'_ts,  y_t = v_t^T S_open(c-1) k_t,
// with G'_ts = (k_t.k_s)(v_t.v_s) the cross-chunk Gram entries; if its last
// boundary was at j, S_open(c) holds tokens j.. of chunk c-1 only and
// x_t = sum_{j <= s < 64} G'_ts.  Both sums are K0's cross table cs[j][t].  So
// y of chunk c is formed from the state one chunk older than the chunk before
// it, and the state work of chunk c-1 (its builds, closes and merges) runs
// while the decisions of chunk c are taken:
//   warp 0     decisions: boundary passes and the replay of Algorithm 2 on
//              register-resident cache metadata (as in dla_scan_mma.cu), with
//              x_t and |S_open|^2 from the y values and the cross table;
//   warp 1     TMA loads of the chunks' k and v tiles (four stages);
//   warp 2     tcgen05.mma issue (one thread, commands from the state warps), TMEM allocation;
//   warp 3     bulk copies of the Gram tables (two buffers);
//   warps 4-7  the state: per chunk the masked V_seg^T K_seg builds of the
//              chunk's segments into TMEM (the closed states stored to their
//              cache slots, merges as slot adds), then S_open split into bf16
//              hi + lo in TMEM and Z = S_open K^T (A from TMEM) for the chunk
//              two ahead, y_t = sum_j v_t[j] Z[j][t]; snapshots for the
//              read-out at interval ends.
// A segment's tokens are selected per 16-token K step: whole steps inside the
// segment use the V tile, partial steps a copy of its 16 rows with the rows
// outside the segment zeroed.
// |S_open(c)|^2 = |S_open(c-1)|^2 (exact, from the state) + the chunk's
// recurrence terms (from x, gs, Q, a), so no drift accumulates.  All waits
// are bounded; after a failed wait every role leaves its loop and the CTA
// ends with the status word set.
#include <mutex>

#include "dla_common.cuh"
#include "dla_mma.cuh"
#include "dla_sm100.cuh"
#include "dla_tmap.h"

namespace dla {

namespace {

using namespace sm100;

constexpr int L = kScanL;   // 64 tokens per chunk
constexpr int D = 128;
constexpr int NT = 256;
constexpr int W_DEC = 0, W_KV = 1, W_MMA = 2, W_TAB = 3;  // warps 4..7: state
constexpr int NKV = 3;                                   // k, v stages
constexpr uint32_t kHalf = L * 128;                      // 64 rows x 64 bf16, 128B-swizzled: 8 KB
constexpr uint32_t kTile = 2 * kHalf;                    // one chunk of k or v
constexpr uint32_t kSlabHalf = 16 * 128;                 // 16 rows of one half
constexpr uint32_t kColsZ = 256, kColsHi = 320, kColsLo = 384, kTmemCols = 512;  // region 0 at 0 (128 fp32)

enum : int { OP_CLOSE = 0, OP_MERGE = 1 };
enum : int { CMD_BUILD = 1, CMD_Z = 2, CMD_END = 3 };

struct DecBuf {         // decisions of one chunk (warp 0 -> state warps)
  int ops[3 * L + 4][4];
  int nops, js, Lc, m_chunk, open_slot, m_after;
  int bnd[L];
  int mlog[L];
};
struct SnapBuf {        // snapshot jobs of one interval end
  int src[kMaxC][2];    // pool id, source physical slot (-1: the open entry)
  float scale[kMaxC];   // scale s of each job's fp16 entry (S / s is stored)
  int ids[kMaxC];
  int njobs, m;
};

struct TcScanSmem {
  uint8_t kv[NKV][2][kTile];       // [stage][k, v]: two 64-column halves each, TMA 128B swizzle    96 KB
  uint8_t out[2][16384];           // staging of TMA stores: two 128-row tiles of 128 bytes          32 KB
  uint8_t slab[2][2][kSlabHalf];   // masked 16-row copies of v                                      8 KB
  float tab[2][kGramBlockTc];      // Gram tables of two chunks                                     66 KB
  DecBuf dec[2];
  SnapBuf snap[2];
  float ybuf[2][L + 4];            // y_t and |S_open|^2 of a chunk
  float red[4][L];
  float gred[4];
  int slot0[kMaxC];
  float scale0[kMaxC];             // scales of the round's first snapshot (every live entry)
  int gcnt[kMaxGramBlk];
  int cmd[2][8];                   // MMA commands: kind, stage, region, acc, source of each K step
  uint64_t kv_full[NKV], kv_empty[NKV], tab_full[2], tab_empty[2], dec_full[2], y_full[2], cmd_full[2],
      cmd_done[2];
  uint32_t tmem_base;
  int abort_flag;
  int m0;
};

// (x, y) as packed bf16 hi = bf16(x, y) and lo = bf16(x - hi, y - hi).
__device__ __forceinline__ void split_pair(float x, float y, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(x, y);
  const float2 f = __bfloat1622float2(h);
  const __nv_bfloat162 l = __floats2bfloat162_rn(x - f.x, y - f.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

// Gram feed of a pre-pass running beside the scan (see dla_scan_mma.cu).
__device__ __forceinline__ bool tab_feed_wait(const int32_t* ready, int nblk, int* cnt, int gc, volatile int* abort,
                                              int32_t* status) {
  if (!ready) return true;
  const int blk = gc % nblk, need = gc / nblk + 1;
  if (cnt[blk] < need) {
    const long long t0 = clock64();
    long long lim = -1;
    while (true) {
      const int c = ld_acquire_gpu(ready + blk);
      if (c >= need) {
        cnt[blk] = c;
        break;
      }
      if (*abort) return false;
      if (*(volatile int32_t*)status != 0 || wait_expired(t0, lim, status)) {
        *abort = 1;
        atomicCAS(status, 0, kStatusTimeout);
        return false;
      }
    }
  }
  asm volatile("fence.proxy.async.global;" ::: "memory");
  return true;
}

// AND of `ok` over the 128 threads of the state warps (named barrier 1).
__device__ __forceinline__ bool state_all(bool ok) {
  int r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.b32 p, %1, 0;\n bar.red.and.pred q, 1, 128, p;\n selp.b32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"((int)ok)
      : "memory");
  return r != 0;
}
__device__ __forceinline__ void state_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

}  // namespace

__global__ void __launch_bounds__(NT, 1)
    scan_tc_kernel(ScanArgs a, const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                   const __grid_constant__ CUtensorMap tmS, const __grid_constant__ CUtensorMap tmP) {
  extern __shared__ uint8_t smem_raw[];
  TcScanSmem& sm = *reinterpret_cast<TcScanSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int bh = blockIdx.x;
  const int b = bh / a.H, h = bh % a.H;
  const int C = a.C;
  const int ntok = a.t_end - a.t_begin;
  const int nchunks = (ntok + L - 1) / L;
  float* states = a.states + (long long)bh * C * D * D;
  constexpr long long kEntry = (long long)D * D;  // a pool entry: S / s in fp16, D rows
  __half* pool = a.pool ? reinterpret_cast<__half*>(a.pool) + (long long)bh * a.pool_cap * kEntry : nullptr;
  uint8_t* bnd_out = a.boundary + (long long)bh * a.T;
  int32_t* mlog_out = a.merge_log + (long long)bh * a.T;
  volatile int* abort = &sm.abort_flag;

  // ---------------------------------------------------------------- set-up
  if (tid == 0) {
    if (a.started) atomicAdd(a.started, 1);  // the read-out stream's gate counts the resident scan CTAs
    int m0 = a.m[bh];
    if (m0 < 0 || m0 > C) {
      atomicCAS(a.status, 0, 6);
      m0 = 0;
    }
    sm.m0 = m0;
    sm.abort_flag = 0;
    for (int i = 0; i < NKV; ++i) {
      mbar_init(&sm.kv_full[i], 1);
      mbar_init(&sm.kv_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.tab_full[i], 1);
      mbar_init(&sm.tab_empty[i], 1);
      mbar_init(&sm.dec_full[i], 1);
      mbar_init(&sm.y_full[i], 1);
    }
    mbar_init(&sm.cmd_full[0], 1);
    mbar_init(&sm.cmd_full[1], 1);
    mbar_init(&sm.cmd_done[0], 1);
    mbar_init(&sm.cmd_done[1], 1);
    for (int i = 0; i < kMaxGramBlk; ++i) sm.gcnt[i] = 0;
    fence_mbar_init();
  }
  for (int i = tid; i < C; i += NT) {
    int sl = a.slot[(long long)bh * C + i];
    if (sl < 0 || sl >= C) {
      atomicCAS(a.status, 0, 6);
      sl = i;
    }
    sm.slot0[i] = sl;
    // a round that restarts its pool copies every live entry first
    if (a.pool && !a.carry_in) sm.scale0[i] = f16_scale(a.nbound[(long long)bh * C + i]);
  }
  if (warp == W_MMA) tmem_alloc(&sm.tmem_base, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  const int m_start = sm.m0;

  if (warp == W_DEC) {
    // ============================================================ decisions
    const float Df = (float)(D * D), invDf = 1.f / Df;
    int e_n[2] = {0, 0}, e_slot[2] = {0, 0}, e_pid[2] = {-1, -1}, e_dirty[2] = {0, 0};
    double e_ib[2] = {0.0, 0.0};
    float e_nb[2] = {0.f, 0.f};  // upper bounds of |S|_F (the scales of the fp16 snapshots)
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int i = lane + 32 * r;
      if (i < C) {
        e_n[r] = a.n[(long long)bh * C + i];
        e_ib[r] = a.ibar[(long long)bh * C + i];
        e_slot[r] = sm.slot0[i];
        if (pool && i < m_start) e_nb[r] = a.nbound[(long long)bh * C + i];
      }
    }
    int pool_next = 0;
    if (pool) {
      if (a.carry_in) {
        pool_next = a.pstate[bh];
#pragma unroll
        for (int r = 0; r < 2; ++r)
          if (lane + 32 * r < m_start) e_pid[r] = a.pstate[a.B * a.H + (long long)bh * C + lane + 32 * r];
      } else {
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int i = lane + 32 * r;
          if (i < m_start) {
            e_pid[r] = i;
            a.pool_scale[(long long)bh * a.pool_cap + i] = sm.scale0[i];
          }
        }
        pool_next = m_start;
      }
    }
    int m = m_start;
    bool bnd_prev = false;  // the previous chunk had a boundary, the last at jl
    int jl = 0;
    float rec = 0.f;        // recurrence part of |S_open|^2 over the previous chunk
    const int ta = 2 * lane, tb = ta + 1;
    for (int c = 0; c < nchunks; ++c) {
      const int bb = c & 1;
      const int t0 = a.t_begin + c * L;
      const int Lc = min(L, a.t_end - t0);
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.tab_full[bb], (uint32_t)((c >> 1) & 1), abort, a.status))) break;
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.y_full[bb], (uint32_t)((c >> 1) & 1), abort, a.status))) break;
      const float* gsp = sm.tab[bb];
      const float* qp = gsp + kPackTri;
      const float* av = gsp + 2 * kPackTri;
      const float* csp = av + L;
      const float* yb = sm.ybuf[bb];
      DecBuf& dc = sm.dec[bb];
      const int m_chunk = m;
      // x_t (the open state before the chunk against token t) and |S_open|^2
      float xa = 0.f, xb = 0.f, gam_open = 0.f;
      if (m_chunk > 0) {
        if (c == 0) {
          xa = yb[ta];
          xb = yb[tb];
          gam_open = yb[L];
        } else if (bnd_prev) {
          xa = csp[jl * L + ta];
          xb = csp[jl * L + tb];
          gam_open = rec;
        } else {
          xa = yb[ta] + csp[ta];
          xb = yb[tb] + csp[tb];
          gam_open = yb[L] + rec;
        }
      }
      if (ta >= Lc) xa = 0.f;
      if (tb >= Lc) xb = 0.f;
      const float aa = (ta < Lc) ? av[ta] : 0.f, ab = (tb < Lc) ? av[tb] : 0.f;
      if (m_chunk > 0) entry_set(e_nb, m_chunk - 1, sqrtf(fmaxf(gam_open, 0.f)));
      // exclusive prefix sums X, A of x and a over the chunk
      float xpa, xpb, apa, apb, xtot, atot;
      {
        float ix = xa + xb, ia = aa + ab;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const float ux = __shfl_up_sync(0xffffffffu, ix, o);
          const float ua = __shfl_up_sync(0xffffffffu, ia, o);
          if (lane >= o) {
            ix += ux;
            ia += ua;
          }
        }
        xtot = __shfl_sync(0xffffffffu, ix, 31);
        atot = __shfl_sync(0xffffffffu, ia, 31);
        xpa = __shfl_up_sync(0xffffffffu, ix, 1);
        apa = __shfl_up_sync(0xffffffffu, ia, 1);
        if (lane == 0) xpa = apa = 0.f;
        xpb = xpa + xa;
        apb = apa + aa;
      }
      // ---- boundary passes: score every undecided token as if the open segment
      // ran to it, take the first that fires, restart the segment there
      float Ia = 0.f, Ib = 0.f;
      int cur = 0, js = 0, pre = (m_chunk > 0) ? 1 : 0;
      unsigned long long bmask = 0;
      if (m_chunk == 0) {  // the very first token of an empty cache opens state 0 (score 0)
        bmask = 1;
        cur = 1;
      }
      while (cur < Lc) {
        const float xpj = __shfl_sync(0xffffffffu, (js & 1) ? xpb : xpa, js >> 1);
        const float apj = __shfl_sync(0xffffffffu, (js & 1) ? apb : apa, js >> 1);
        const float g0 = pre ? gam_open : 0.f;
        const int rowj = pack_row(js) - js;
        bool fa = false, fb = false;
        if (ta >= cur && ta < Lc) {
          const float ba = (pre ? xa : 0.f) + gsp[rowj + ta];
          const float ea = (pre ? 2.f * (xpa - xpj) : 0.f) + 2.f * qp[rowj + ta] + (apa - apj);
          Ia = info_score_fast(aa, ba, g0 + ea, invDf, a.sp);
          fa = (Ia >= a.sp.tau_f);
        }
        if (tb >= cur && tb < Lc) {
          const float bb2 = (pre ? xb : 0.f) + gsp[rowj + tb];
          const float eb = (pre ? 2.f * (xpb - xpj) : 0.f) + 2.f * qp[rowj + tb] + (apb - apj);
          Ib = info_score_fast(ab, bb2, g0 + eb, invDf, a.sp);
          fb = (Ib >= a.sp.tau_f);
        }
        const unsigned bal = __ballot_sync(0xffffffffu, fa || fb);
        if (!bal) break;
        const int src = __ffs(bal) - 1;
        const int ts = 2 * src + (__shfl_sync(0xffffffffu, (int)fa, src) ? 0 : 1);
        bmask |= 1ull << ts;
        js = ts;
        pre = 0;
        cur = ts + 1;
      }
      dc.bnd[ta] = (int)((bmask >> ta) & 1);
      dc.bnd[tb] = (int)((bmask >> tb) & 1);
      dc.mlog[ta] = -1;
      dc.mlog[tb] = -1;
      // ---- replay of the decisions (Algorithm 2) on the register-resident metadata
      auto run_sum = [&](int u0, int u1) -> float {
        const float v = ((ta >= u0 && ta < u1) ? Ia : 0.f) + ((tb >= u0 && tb < u1) ? Ib : 0.f);
        return warp_sum(v);
      };
      int seg_u0 = 0, nops = 0, run0 = 0;
      unsigned long long pend = bmask;
      __syncwarp();
      while (true) {
        const int t = pend ? (__ffsll((long long)pend) - 1) : Lc;
        pend &= pend - 1;
        if (t > run0) {  // tokens [run0, t) joined the open state (entry m - 1)
          const double part = (double)run_sum(run0, t);
          // |S + sum v k^T|_F <= |S|_F + sum |v| |k|, and |v_t| |k_t| = sqrt(a_t)
          const float grow =
              warp_sum(((ta >= run0 && ta < t) ? sqrtf(aa) : 0.f) + ((tb >= run0 && tb < t) ? sqrtf(ab) : 0.f));
          const int e = m - 1;
          if ((e & 31) == lane) {
            if (e < 32) {
              e_n[0] += t - run0; e_ib[0] += part; e_dirty[0] = 1; e_nb[0] += grow;
            } else {
              e_n[1] += t - run0; e_ib[1] += part; e_dirty[1] = 1; e_nb[1] += grow;
            }
          }
        }
        run0 = t + 1;
        if (t >= Lc) break;
        if (m > 0) {
          const int sl = entry_get(e_slot, m - 1);
          if (lane == 0) {
            dc.ops[nops][0] = OP_CLOSE;
            dc.ops[nops][1] = sl;
            dc.ops[nops][2] = seg_u0;
            dc.ops[nops][3] = t;
          }
          ++nops;
        }
        int j = -1, phys_new = m;
        if (m == C) {
          // pair densities (Ibar_i + Ibar_{i+1}) / (n_i + n_{i+1}): fp64 sums, compared in fp32
          int nn[2], ns[2], np_[2], nd[2];
          double nb[2];
          float nnb[2];
          entry_next(e_n, nn);
          entry_next(e_ib, nb);
          entry_next(e_nb, nnb);
          entry_next(e_slot, ns);
          entry_next(e_pid, np_);
          entry_next(e_dirty, nd);
          float best = __int_as_float(0x7f800000);
          int bi = 0x7fffffff;
          if (lane + 1 < m) {
            best = (float)(e_ib[0] + nb[0]) / (float)(e_n[0] + nn[0]);
            bi = lane;
          }
          if (lane + 33 < m) {
            const float d1 = (float)(e_ib[1] + nb[1]) / (float)(e_n[1] + nn[1]);
            if (d1 < best) {
              best = d1;
              bi = lane + 32;
            }
          }
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, best, o);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
            if (ov < best || (ov == best && oi < bi)) {
              best = ov;
              bi = oi;
            }
          }
          j = bi;
          const int dst = entry_get(e_slot, j), srcs = entry_get(e_slot, j + 1);
          if (lane == 0) {
            dc.ops[nops][0] = OP_MERGE;
            dc.ops[nops][1] = dst;
            dc.ops[nops][2] = srcs;
            dc.ops[nops][3] = 0;
          }
          ++nops;
#pragma unroll
          for (int r = 0; r < 2; ++r) {
            const int i = lane + 32 * r;
            if (i == j) {
              e_n[r] += nn[r]; e_ib[r] += nb[r]; e_dirty[r] = 1; e_pid[r] = -1; e_nb[r] += nnb[r];
            } else if (i > j && i < m - 1) {
              e_n[r] = nn[r]; e_ib[r] = nb[r]; e_slot[r] = ns[r]; e_pid[r] = np_[r]; e_dirty[r] = nd[r];
              e_nb[r] = nnb[r];
            }
          }
          phys_new = srcs;
          m -= 1;
        }
        const float it = __shfl_sync(0xffffffffu, (t & 1) ? Ib : Ia, t >> 1);
        entry_set(e_nb, m, sqrtf(__shfl_sync(0xffffffffu, (t & 1) ? ab : aa, t >> 1)));
        entry_set(e_slot, m, phys_new);
        entry_set(e_n, m, 1);
        entry_set(e_ib, m, (double)it);
        entry_set(e_pid, m, -1);
        entry_set(e_dirty, m, 1);
        if (lane == 0) dc.mlog[t] = j;
        m += 1;
        seg_u0 = t;
      }
      // ---- recurrence part of |S_open|^2 over this chunk, for the next chunk:
      // the open segment at the chunk end starts at seg_u0 (with the state from
      // before the chunk when the chunk had no boundary)
      {
        const bool any = bmask != 0;
        const int jf = seg_u0;
        const float xpj = __shfl_sync(0xffffffffu, (jf & 1) ? xpb : xpa, jf >> 1);
        const float apj = __shfl_sync(0xffffffffu, (jf & 1) ? apb : apa, jf >> 1);
        const bool pre_f = !any && m_chunk > 0;
        rec = (pre_f ? 2.f * (xtot - xpj) : 0.f) + 2.f * qp[pack_row(jf) - jf + Lc] + (atot - apj);
        bnd_prev = any;
        jl = jf;
      }
      const int oslot = (m > 0) ? entry_get(e_slot, m - 1) : 0;
      // ---- snapshot jobs at an interval end: entries whose state changed get a fresh pool entry
      const bool ivl_end = ((c + 1) % a.snap_chunks) == 0;
      const int snap_idx = (c + 1) / a.snap_chunks;
      if (pool && ivl_end && (snap_idx < a.nsnap || a.snap_at_end)) {
        SnapBuf& sb = sm.snap[snap_idx & 1];
        int nj = 0;
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int i = lane + 32 * r;
          const bool need = (i < m) && (e_dirty[r] || e_pid[r] < 0);
          const unsigned bal = __ballot_sync(0xffffffffu, need);
          if (need) {
            const int rank_ = nj + __popc(bal & ((1u << lane) - 1u));
            int p = pool_next + rank_;
            if (p >= a.pool_cap) {  // cannot happen with a correctly sized workspace
              atomicCAS(a.status, 0, 6);
              p = a.pool_cap - 1;
            }
            e_pid[r] = p;
            e_dirty[r] = 0;
            sb.src[rank_][0] = p;
            sb.src[rank_][1] = (i == m - 1) ? -1 : e_slot[r];
            const float sc = f16_scale(e_nb[r]);
            sb.scale[rank_] = sc;
            a.pool_scale[(long long)bh * a.pool_cap + p] = sc;
          }
          nj += __popc(bal);
          if (i < m) sb.ids[i] = e_pid[r];
        }
        pool_next += nj;
        if (lane == 0) {
          sb.njobs = nj;
          sb.m = m;
        }
      }
      if (lane == 0) {
        dc.nops = nops;
        dc.js = seg_u0;
        dc.Lc = Lc;
        dc.m_chunk = m_chunk;
        dc.open_slot = oslot;
        dc.m_after = m;
      }
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&sm.tab_empty[bb]);
        mbar_arrive(&sm.dec_full[bb]);
      }
    }
    // ---------------------------------------------------------------- round end: metadata
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int i = lane + 32 * r;
      if (i < C) {
        a.slot[(long long)bh * C + i] = e_slot[r];
        a.n[(long long)bh * C + i] = (i < m) ? e_n[r] : 0;
        a.ibar[(long long)bh * C + i] = (i < m) ? e_ib[r] : 0.0;
      }
      if (pool && a.pstate && i < m) a.pstate[a.B * a.H + (long long)bh * C + i] = e_pid[r];
      if (pool && i < m) a.nbound[(long long)bh * C + i] = e_nb[r];
    }
    if (lane == 0) {
      a.m[bh] = m;
      if (pool && a.pstate) a.pstate[bh] = pool_next;
    }
  } else if (warp == W_KV) {
    // ============================================================ k, v tiles (TMA)
    if (lane == 0) {
      prefetch_tmap(&tmK);
      prefetch_tmap(&tmV);
      int issued[NKV] = {};
      for (int c = 0; c < nchunks; ++c) {
        const int s = c % NKV, n = c / NKV;
        if (n > 0 && !mbar_wait(&sm.kv_empty[s], (uint32_t)((n - 1) & 1), abort, a.status)) break;
        const int t0 = a.t_begin + c * L;
        mbar_expect_tx(&sm.kv_full[s], 2 * kTile);
        tma_load_4d(sm.kv[s][0], &tmK, &sm.kv_full[s], 0, h, t0, b);
        tma_load_4d(sm.kv[s][0] + kHalf, &tmK, &sm.kv_full[s], 64, h, t0, b);
        tma_load_4d(sm.kv[s][1], &tmV, &sm.kv_full[s], 0, h, t0, b);
        tma_load_4d(sm.kv[s][1] + kHalf, &tmV, &sm.kv_full[s], 64, h, t0, b);
        issued[s] = n + 1;
      }
      if (*abort)  // let copies in flight land before the CTA exits
        for (int s = 0; s < NKV; ++s)
          if (issued[s] > 0) mbar_wait_drain(&sm.kv_full[s], (uint32_t)((issued[s] - 1) & 1));
    }
  } else if (warp == W_TAB) {
    // ============================================================ Gram tables (bulk copies)
    if (lane == 0) {
      int issued[2] = {0, 0};
      for (int c = 0; c < nchunks; ++c) {
        const int bb = c & 1, n = c >> 1;
        if (n > 0 && !mbar_wait(&sm.tab_empty[bb], (uint32_t)((n - 1) & 1), abort, a.status)) break;
        const int gc = a.t_begin / L + c;
        if (!tab_feed_wait(a.gram_ready ? a.gram_ready + (long long)bh * a.gram_nblk : nullptr, a.gram_nblk, sm.gcnt,
                           gc, abort, a.status))
          break;
        mbar_expect_tx(&sm.tab_full[bb], (uint32_t)kGramBlockTc * 4u);
        bulk_g2s(sm.tab[bb], a.gram + ((long long)bh * a.gram_chunks + gc) * kGramBlockTc, (uint32_t)kGramBlockTc * 4u,
                 &sm.tab_full[bb]);
        issued[bb] = n + 1;
      }
      if (*abort)
        for (int bb = 0; bb < 2; ++bb)
          if (issued[bb] > 0) mbar_wait_drain(&sm.tab_full[bb], (uint32_t)((issued[bb] - 1) & 1));
    }
  } else if (warp == W_MMA) {
    // ============================================================ tcgen05.mma issue
    if (lane == 0) {
      // build: D[j][k] += sum_t V[t][j] K[t][k]: A = V^T and B = K, both MN-major
      // (64-wide blocks 8 KB apart in a tile, 2 KB in a slab; 1 KB per 8 rows)
      constexpr uint32_t idb = idesc_bf16_f32(128, 128) | (1u << 15) | (1u << 16);
      // Z[j][t] = sum_k S[j][k] K[t][k]: A = S as bf16 hi + lo in TMEM, B = K K-major, N = 64 tokens
      constexpr uint32_t idz = idesc_bf16_f32(128, 64);
      int n = 0;
      for (;; ++n) {
        const int sl = n & 1;
        if (!mbar_wait(&sm.cmd_full[sl], (uint32_t)((n >> 1) & 1), abort, a.status)) break;
        tc_fence_after();
        const int kind = sm.cmd[sl][0];
        if (kind == CMD_END) break;
        const int stg = sm.cmd[sl][1];
        const uint32_t kbase = smem_u32(sm.kv[stg][0]), vbase = smem_u32(sm.kv[stg][1]);
        if (kind == CMD_BUILD) {
          const uint32_t dcol = tmem + 128u * (uint32_t)sm.cmd[sl][2];
          uint32_t acc = (uint32_t)sm.cmd[sl][3];
          for (int kk = 0; kk < 4; ++kk) {
            const int src = sm.cmd[sl][4 + kk];
            if (src < 0) continue;
            const uint64_t ad = (src == 0) ? desc_mnmajor_sw128(vbase + kk * 2048, kHalf)
                                           : desc_mnmajor_sw128(smem_u32(sm.slab[src - 1][0]), kSlabHalf);
            mma_bf16(dcol, ad, desc_mnmajor_sw128(kbase + kk * 2048, kHalf), idb, acc);
            acc = 1;
          }
        } else {
#pragma unroll
          for (int kk = 0; kk < 8; ++kk)
            mma_ts(tmem + kColsZ, tmem + kColsHi + kk * 8,
                   desc_kmajor_sw128(kbase + (kk >> 2) * kHalf + (kk & 3) * 32), idz, kk > 0);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk)
            mma_ts(tmem + kColsZ, tmem + kColsLo + kk * 8,
                   desc_kmajor_sw128(kbase + (kk >> 2) * kHalf + (kk & 3) * 32), idz, 1u);
        }
        mma_commit(&sm.cmd_done[sl]);
      }
      if (n > 0)  // every MMA issued has completed before TMEM is freed
        mbar_wait_drain(&sm.cmd_done[(n - 1) & 1], (uint32_t)(((n - 1) >> 1) & 1));
    }
  } else {
    // ============================================================ state warps
    const int st = tid - 128;  // TMEM lane = state row j
    const int qd = warp & 3;
    const uint32_t lrow = (uint32_t)(qd * 32) << 16;  // TMEM lane field of this warp's rows
    const int j = st;
    int ncmd = 0;  // MMA commands sent so far
    constexpr int cur = 0;  // TMEM region of the open state (region 1 is unused)
    // One MMA command to warp 2, after the fences that make this warp group's
    // shared / tensor memory writes visible to the tensor core; every thread
    // waits for its completion.
    auto issue = [&](int kind, int stg, int region, int acc, const int* src) -> bool {
      fence_proxy_async();
      tc_fence_before();
      state_sync();
      const int sl = ncmd & 1;
      if (st == 0) {
        sm.cmd[sl][0] = kind;
        sm.cmd[sl][1] = stg;
        sm.cmd[sl][2] = region;
        sm.cmd[sl][3] = acc;
        for (int kk = 0; kk < 4; ++kk) sm.cmd[sl][4 + kk] = src ? src[kk] : -1;
        mbar_arrive(&sm.cmd_full[sl]);
      }
      const bool ok = state_all(mbar_wait(&sm.cmd_done[sl], (uint32_t)((ncmd >> 1) & 1), abort, a.status));
      ++ncmd;
      __syncwarp();
      tc_fence_after();
      return ok;
    };
    auto issue_z = [&](int stg) -> bool { return issue(CMD_Z, stg, 0, 0, nullptr); };
    // tokens [u0, u1) of stage stg into region (accumulating onto it, or not)
    auto build = [&](int stg, int region, int u0, int u1, int acc) -> bool {
      int src[4];
      int nsl = 0;
      for (int kk = 0; kk < 4; ++kk) {
        const int lo = 16 * kk, hi = lo + 16;
        if (u1 <= lo || u0 >= hi) {
          src[kk] = -1;
        } else if (u0 <= lo && u1 >= hi) {
          src[kk] = 0;
        } else {  // rows lo .. lo + 15 of v with those outside [u0, u1) zeroed
          src[kk] = 1 + nsl;
          for (int e = st; e < 256; e += 128) {
            const int r = e >> 4, hf = (e >> 3) & 1, ch = e & 7;
            const int t = lo + r;
            uint4 v = *reinterpret_cast<const uint4*>(sm.kv[stg][1] + hf * kHalf + t * 128 + ch * 16);
            if (!(t >= u0 && t < u1)) v = make_uint4(0u, 0u, 0u, 0u);
            *reinterpret_cast<uint4*>(sm.slab[nsl][hf] + r * 128 + ch * 16) = v;
          }
          ++nsl;
        }
      }
      return issue(CMD_BUILD, stg, region, acc, src);
    };
    // Rows of this warp group (row j by this thread) into the staging tile
    // `tile` in the 128-byte swizzle of the TMA maps: 32 words of row j.
    auto stage_row = [&](uint8_t* tile, const float* v) {
#pragma unroll
      for (int i = 0; i < 8; ++i)
        *reinterpret_cast<uint4*>(tile + j * 128 + ((i ^ (j & 7)) << 4)) =
            make_uint4(__float_as_uint(v[4 * i]), __float_as_uint(v[4 * i + 1]), __float_as_uint(v[4 * i + 2]),
                       __float_as_uint(v[4 * i + 3]));
    };
    // both staging tiles out by TMA (thread 0), once every thread has written them;
    // returns when the tiles may be written again
    auto flush_tiles = [&](const CUtensorMap* map, int x0, int y0, int x1, int y1) {
      fence_proxy_async();
      state_sync();
      if (st == 0) {
        tma_store_2d(map, sm.out[0], x0, y0);
        tma_store_2d(map, sm.out[1], x1, y1);
        bulk_commit();
        bulk_wait_read0();
      }
      state_sync();
    };
    // the stores so far are complete and visible to the generic proxy
    auto stores_done = [&]() {
      if (st == 0) {
        bulk_wait0();
        asm volatile("fence.proxy.async.global;" ::: "memory");
      }
      state_sync();
    };
    // region -> the fp32 rows of cache slot `phys` (four 32-column tiles)
    auto store_region = [&](int region, int phys) {
      const int row0 = (bh * C + phys) * D;
#pragma unroll 1
      for (int r = 0; r < 2; ++r) {
        float v[64];
        tmem_ld32x2(tmem + lrow + 128u * region + 64 * r, tmem + lrow + 128u * region + 64 * r + 32, v);
        stage_row(sm.out[0], v);
        stage_row(sm.out[1], v + 32);
        flush_tiles(&tmS, 64 * r, row0, 64 * r + 32, row0);
      }
    };
    // region -> bf16 hi + lo (TMEM, the y GEMM's A operand); returns this row's |S|^2.
    // (One bf16 rounding of S would leave the scores about 4e-6 relative off on
    // coherent streams, too close to the tie margin of the merge decisions.)
    auto split = [&](int region) -> float {
      float g = 0.f;
#pragma unroll 1
      for (int half = 0; half < 2; ++half) {
        float v[64];
        tmem_ld32x2(tmem + lrow + 128u * region + 64 * half, tmem + lrow + 128u * region + 64 * half + 32, v);
#pragma unroll
        for (int cc = 0; cc < 2; ++cc) {
          float hi[16], lo[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float x0 = v[32 * cc + 2 * i], x1 = v[32 * cc + 2 * i + 1];
            g += x0 * x0 + x1 * x1;
            uint32_t hw, lw;
            split_pair(x0, x1, hw, lw);
            hi[i] = __uint_as_float(hw);
            lo[i] = __uint_as_float(lw);
          }
          tmem_st16(tmem + lrow + kColsHi + 32 * half + 16 * cc, hi);
          tmem_st16(tmem + lrow + kColsLo + 32 * half + 16 * cc, lo);
        }
      }
      tmem_st_wait();
      return g;
    };
    // y_t = sum_j v_t[j] Z[j][t] of the chunk in stage stg into ybuf[ybi], with
    // |S|^2 = the sum of the rows' g; then warp 0 may read them
    auto y_epilogue = [&](int stg, int ybi, float g) {
      float p[64];
      tmem_ld32x2(tmem + lrow + kColsZ, tmem + lrow + kColsZ + 32, p);
      const uint8_t* vt = sm.kv[stg][1] + (j >> 6) * kHalf;
      const int jj = j & 63;
#pragma unroll
      for (int t = 0; t < 64; ++t)
        p[t] *= __bfloat162float(*reinterpret_cast<const __nv_bfloat16*>(vt + sw128_offset(t, jj)));
      // reduce-scatter over the warp's 32 rows: lane l ends with tokens 2l, 2l + 1
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const bool up = (lane & 16) != 0;
        const float send = up ? p[i] : p[32 + i], keep = up ? p[32 + i] : p[i];
        p[i] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
      }
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const bool up = (lane & 8) != 0;
        const float send = up ? p[i] : p[16 + i], keep = up ? p[16 + i] : p[i];
        p[i] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const bool up = (lane & 4) != 0;
        const float send = up ? p[i] : p[8 + i], keep = up ? p[8 + i] : p[i];
        p[i] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const bool up = (lane & 2) != 0;
        const float send = up ? p[i] : p[4 + i], keep = up ? p[4 + i] : p[i];
        p[i] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
      }
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const bool up = (lane & 1) != 0;
        const float send = up ? p[i] : p[2 + i], keep = up ? p[2 + i] : p[i];
        p[i] = keep + __shfl_xor_sync(0xffffffffu, send, 1);
      }
      sm.red[qd][2 * lane] = p[0];
      sm.red[qd][2 * lane + 1] = p[1];
      g = warp_sum(g);
      if (lane == 0) sm.gred[qd] = g;
      state_sync();
      if (st < L) sm.ybuf[ybi][st] = sm.red[0][st] + sm.red[1][st] + sm.red[2][st] + sm.red[3][st];
      if (st == L) sm.ybuf[ybi][L] = sm.gred[0] + sm.gred[1] + sm.gred[2] + sm.gred[3];
      state_sync();
      if (st == 0) mbar_arrive(&sm.y_full[ybi]);
    };
    // dst += src over one d x d state (coalesced, all 128 threads)
    auto add_state = [&](float* dst, const float* src) {
      constexpr int N4 = D * D / 4;
#pragma unroll 1
      for (int base = st; base < N4; base += 4 * 128) {
        float4 x[4], y[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          x[i] = load4(dst + (base + i * 128) * 4);
          y[i] = load4(src + (base + i * 128) * 4);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
          store4(dst + (base + i * 128) * 4, make_float4(x[i].x + y[i].x, x[i].y + y[i].y, x[i].z + y[i].z, x[i].w + y[i].w));
      }
    };
    // fp32 state -> fp16 pool entry S / s (inv = 1 / s), coalesced
    auto copy_f16 = [&](__half* entry, const float* src, float inv) {
      constexpr int N4 = D * D / 4;
#pragma unroll 1
      for (int base = st; base < N4; base += 4 * 128) {
        float4 v[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) v[i] = load4(src + (base + i * 128) * 4);
#pragma unroll
        for (int i = 0; i < 4; ++i) *reinterpret_cast<uint2*>(entry + (base + i * 128) * 4) = f16x4(v[i], inv);
      }
    };

    // ---------------------------------------------------------------- round start
    if (st == 0) {
      prefetch_tmap(&tmS);
      prefetch_tmap(&tmP);
    }
    if (m_start > 0) {  // the open state into region 0
      const float* row = states + (long long)sm.slot0[m_start - 1] * D * D + (long long)j * D;
#pragma unroll 1
      for (int cc = 0; cc < 8; ++cc) {
        float v[16];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float4 x = load4(row + 16 * cc + 4 * i);
          v[4 * i] = x.x; v[4 * i + 1] = x.y; v[4 * i + 2] = x.z; v[4 * i + 3] = x.w;
        }
        tmem_st16(tmem + lrow + 16 * cc, v);
      }
      tmem_st_wait();
    }
    if (pool && !a.carry_in) {  // snapshot 0: every live entry at the start of the round
      const long long lst = (long long)bh * a.snap_stride + a.snap_base;
      for (int i = 0; i < m_start && i < a.pool_cap; ++i)
        copy_f16(pool + (long long)i * kEntry, states + (long long)sm.slot0[i] * D * D, 1.f / sm.scale0[i]);
      if (st == 0) a.snap_m0[lst] = m_start;
      if (st < m_start) a.snap_ids[lst * C + st] = st;
    }
    bool ok = true;
    // y of the first two chunks against the starting state (zero for an empty cache)
    if (m_start > 0) {
      tc_fence_before();
      state_sync();
      tc_fence_after();
      const float g = split(0);
      for (int cc = 0; ok && cc < 2 && cc < nchunks; ++cc) {
        ok = state_all(mbar_wait(&sm.kv_full[cc], 0u, abort, a.status)) && issue_z(cc);
        if (ok) y_epilogue(cc, cc, g);
      }
    } else {
      for (int cc = 0; cc < 2 && cc < nchunks; ++cc) {
        if (st <= L) sm.ybuf[cc][st] = 0.f;
        state_sync();
        if (st == 0) mbar_arrive(&sm.y_full[cc]);
      }
    }
    // ---------------------------------------------------------------- chunks
    for (int c = 0; ok && c < nchunks; ++c) {
      const int bb = c & 1;
      if (!(ok = state_all(mbar_wait(&sm.dec_full[bb], (uint32_t)((c >> 1) & 1), abort, a.status)))) break;
      const DecBuf& dc = sm.dec[bb];
      const int Lc = dc.Lc, t0 = a.t_begin + c * L, stg = c % NKV;
      if (st < Lc) {
        bnd_out[t0 + st] = (uint8_t)dc.bnd[st];
        mlog_out[t0 + st] = dc.mlog[st];
      }
      if (!(ok = state_all(mbar_wait(&sm.kv_full[stg], (uint32_t)((c / NKV) & 1), abort, a.status)))) break;
      bool built = false;
      const int nops = dc.nops;
      for (int op = 0; ok && op < nops; ++op) {
        if (dc.ops[op][0] == OP_CLOSE) {
          const int acc = (!built && dc.m_chunk > 0) ? 1 : 0;
          ok = build(stg, cur, dc.ops[op][2], dc.ops[op][3], acc);
          built = true;
          if (ok) store_region(cur, dc.ops[op][1]);
        } else {
          stores_done();  // the closed states' TMA stores, before the generic reads of the add
          add_state(states + (long long)dc.ops[op][1] * D * D, states + (long long)dc.ops[op][2] * D * D);
          state_sync();
        }
      }
      if (!ok) break;
      // the chunk's tail joins the open state (or starts it)
      if (!(ok = build(stg, cur, dc.js, Lc, (!built && dc.m_chunk > 0) ? 1 : 0))) break;
      if (st == 0) mbar_arrive(&sm.kv_empty[stg]);  // the stage's tiles are no longer read
      const bool need_y = (c + 2 < nchunks);
      const bool ivl_end = ((c + 1) % a.snap_chunks) == 0;
      const int snap_idx = (c + 1) / a.snap_chunks;
      const bool do_snap = pool && ivl_end && (snap_idx < a.nsnap || a.snap_at_end);
      float g = 0.f;
      if (need_y) g = split(cur);  // the y operand (snapshots take the fp32 state itself)
      if (need_y) {  // y of chunk c + 2 against S_open at the start of chunk c + 1
        const int s2 = (c + 2) % NKV;
        if (!(ok = state_all(mbar_wait(&sm.kv_full[s2], (uint32_t)(((c + 2) / NKV) & 1), abort, a.status)))) break;
        if (!(ok = issue_z(s2))) break;
        y_epilogue(s2, (c + 2) & 1, g);
      }
      if (ivl_end) {
        // interval snap_base + snap_idx - 1 is complete: its trace is written and the
        // snapshot of its start (taken at the previous interval end) has landed (a
        // concurrent read-out waits for this)
        stores_done();
        if (a.progress && st == 0) st_release_gpu(a.progress + 2 * bh, a.snap_base + snap_idx);
      }
      if (do_snap) {  // the cache at the interval end into the pool (entries that changed)
        const SnapBuf& sb = sm.snap[snap_idx & 1];
        const long long list_row = (long long)bh * a.snap_stride + a.snap_base + snap_idx;
        for (int jj = 0; jj < sb.njobs; ++jj) {
          __half* entry = pool + (long long)sb.src[jj][0] * kEntry;
          const int srcslot = sb.src[jj][1];
          const float inv = 1.f / sb.scale[jj];
          if (srcslot < 0) {  // the open entry: its fp32 rows from TMEM, scaled into fp16, by TMA
            const int row0 = (bh * a.pool_cap + sb.src[jj][0]) * D;
#pragma unroll 1
            for (int half = 0; half < 2; ++half) {
              float v[64], w[32];
              tmem_ld32x2(tmem + lrow + 128u * cur + 64 * half, tmem + lrow + 128u * cur + 64 * half + 32, v);
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                const uint2 h = f16x4(make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]), inv);
                w[2 * i] = __uint_as_float(h.x);
                w[2 * i + 1] = __uint_as_float(h.y);
              }
              stage_row(sm.out[half], w);  // columns 64 * half .. + 63 of row j
            }
            flush_tiles(&tmP, 0, row0, 64, row0);
          } else {
            copy_f16(entry, states + (long long)srcslot * D * D, inv);
          }
        }
        if (st < sb.m) a.snap_ids[list_row * C + st] = sb.ids[st];
        if (st == 0) a.snap_m0[list_row] = sb.m;
      }
    }
    // ---------------------------------------------------------------- round end
    if (ok && nchunks > 0) {
      const DecBuf& dl = sm.dec[(nchunks - 1) & 1];
      if (dl.m_after > 0) store_region(cur, dl.open_slot);
    }
    stores_done();
    if (st == 0) {  // warp 2 leaves its command loop
      sm.cmd[ncmd & 1][0] = CMD_END;
      mbar_arrive(&sm.cmd_full[ncmd & 1]);
    }
    if (a.progress) {  // every interval of this launch is complete
      __threadfence();
      state_sync();
      if (st == 0) st_release_gpu(a.progress + 2 * bh, a.snap_base + a.nsnap);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == W_MMA) tmem_dealloc(tmem, kTmemCols);
}

// ---------------------------------------------------------------- host side
size_t scan_tc_smem_bytes() { return sizeof(TcScanSmem) + 1024; }

cudaError_t launch_scan_tc(const ScanArgs& a, cudaStream_t s) {
  CUtensorMap mk, mv, ms, mp;
  if (!a.pool || !tmap_tokens(&mk, a.k, a.B, a.T, a.H, L) || !tmap_tokens(&mv, a.v, a.B, a.T, a.H, L) ||
      !tmap_states(&ms, a.states, (long long)a.B * a.H * a.C * D) ||
      !tmap_pool(&mp, a.pool, (long long)a.B * a.H * a.pool_cap * D, true))
    return cudaErrorInvalidValue;
  if (!a.gram || a.seq_lens || a.piece_ready || a.snap_chunks != 2) return cudaErrorInvalidValue;
  const size_t smem = scan_tc_smem_bytes();
  cudaError_t e = cudaFuncSetAttribute(scan_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  scan_tc_kernel<<<a.B * a.H, NT, smem, s>>>(a, mk, mv, ms, mp);
  return cudaGetLastError();
}

int scan_tc_resident_streams() {
  static int cache[64];
  static bool init = false;
  static std::mutex mu;
  int dev = 0, sms = 0, per_sm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  std::lock_guard<std::mutex> g(mu);
  if (!init) {
    for (int& c : cache) c = -1;
    init = true;
  }
  if (cache[dev] < 0) {
    const size_t smem = scan_tc_smem_bytes();
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaFuncSetAttribute(scan_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, scan_tc_kernel, NT, smem) != cudaSuccess)
      return 0;
    cache[dev] = per_sm * sms;
  }
  return cache[dev];
}

cudaError_t preload_scan_tc_kernel() {
  cudaFuncAttributes fa;
  return cudaFuncGetAttributes(&fa, scan_tc_kernel);
}

}  // namespace dla

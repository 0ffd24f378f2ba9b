// dla_scan_mma.cu -- K1 for bf16 inputs with its three contractions on the
// tensor cores (warp-level mma.sync m16n8k16, bf16 in, fp32 accumulate):
//   x_t  = v_t^T S_open k_t      via X = K S_open^T (S_open as bf16 hi + lo)
//   G    = (K K^T) o (V V^T)     the chunk's Gram entries (exact bf16 products)
//   S   += V_seg^T K_seg         the state build, masked to a token range
// The open state S_open (d_v x d_k, fp32) never leaves the CTA while it stays
// open: it lives in the mma accumulator registers, warp w owning a 16-row band.
// The decision logic (score-all / first-fire passes, the ordered replay of
// Algorithm 2 in one warp, the state operations, snapshots) is the same as in
// the CUDA-core scan (dla_scan.cu), which remains the fp32-input kernel.
//
// Shapes per 64-token chunk: X is 64 x d x d, the Grams 2 x 64 x 64 x d and the
// build d x d x 64, i.e. about 6 d^2 * 64 flop, a few thousand mma per CTA.
#include <atomic>
#include <mutex>

#include "dla_common.cuh"
#include "dla_mma.cuh"
#include "dla_sm100.cuh"

namespace dla {

namespace {

constexpr int NT = 256;
constexpr int NW = NT / 32;
constexpr int L = kScanL;
constexpr int GS = L;              // row of a Gram table in shared memory (the pre-pass block, verbatim)

enum : int { OP_CLOSE = 0, OP_MERGE = 1 };

template <int D, int CL, int CAPB = kMaxC>
struct MmaSmem {
  // CAPB > kMaxC: the DLA(I) instance, whose cache metadata lives here (b*)
  static constexpr bool kBig = CAPB > kMaxC;
  static constexpr int NB = kBig ? CAPB : 1;
  static constexpr int RP = D + 8;  // padded bf16 row: 8 rows of a ldmatrix hit 8 bank groups
  __nv_bfloat16 kv[2][2][L * RP];   // [stage][k / v][t][RP]
  __nv_bfloat16 S2[2][D / CL * RP]; // this CTA's rows of the open state as bf16 hi / lo, [j][RP]
  // [stage] the chunk's Gram block, as the pre-pass writes it: suffix table
  // gs[j][t] = sum_{j <= s < t} (k_t.k_s)(v_t.v_s), prefix table
  // Q[j][t] = sum_{j <= u < t} gs[j][u], then a_t = |k_t|^2 |v_t|^2
  float gq[2][kGramBlock];
  uint64_t kvbar[2];                // [stage] the stage's Gram block has landed
  float red[NW][L];
  float xs[2][CL][L + 4];           // [chunk parity][CTA] parts of x_t (t < L) and of |S_open|^2 (at L)
  uint64_t xbar[2];                 // [chunk parity] the partner's parts have arrived (CTA pairs)
  int abort_flag;                   // a wait for the partner gave up
  float gred[NW];
  int slot[CAPB];                   // physical slots at the round start (DLA(I): the live map)
  int open_slot;                    // physical slot of the open entry (m - 1) after the last replay
  int bnd[L];
  int mlog[L];
  int ops[3 * L + 4][4];
  int snap_src[CAPB][2];
  float snap_scale[CAPB];           // scale s of each snapshot job (fp16 pool: S / s is stored)
  // DLA(I) instance: n, Ibar, pool id, changed flag and norm bound of every entry
  double bib[NB];
  int bn[NB], bpid[NB], bdirty[NB];
  float bnb[NB];
  int nops, nsnapjobs;
  int pend;                         // snapshot copies waiting for the next chunk's idle warps (bf16 pool)
  int gcnt[kMaxGramBlk];            // Gram pre-pass counters last read (thread 0)
  int m, cur, js, seg_pre, pool_next;
};

// SA[t] = sum_{u < t} sqrt(a_u), t = 0 .. 64, of a chunk's a values (one warp;
// lane l takes tokens 2l and 2l + 1), and three zeros of padding.
__device__ __forceinline__ void norm_prefix_warp(const float* a, float* sa, int lane) {
  const float s0 = sqrtf(a[2 * lane]), s1 = sqrtf(a[2 * lane + 1]);
  float inc = s0 + s1;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float u = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += u;
  }
  const float ex = inc - s0 - s1;
  sa[2 * lane] = ex;
  sa[2 * lane + 1] = ex + s0;
  if (lane == 31) sa[kScanL] = inc;
  if (lane < 3) sa[kScanL + 1 + lane] = 0.f;
}

// Keep the bf16 halves of a packed pair whose token index lies in [u0, u1).
__device__ __forceinline__ uint32_t mask_pair(uint32_t v, int t, int u0, int u1) {
  const uint32_t lo = (t >= u0 && t < u1) ? 0x0000FFFFu : 0u;
  const uint32_t hi = (t + 1 >= u0 && t + 1 < u1) ? 0xFFFF0000u : 0u;
  return v & (lo | hi);
}

// Gram pre-pass running beside the scan: thread 0 of the scan CTA waits until
// the pre-pass CTA of chunk gc's block (block gc % nblk, which takes chunks
// blk, blk + nblk, ... in order) has published the chunk (its counter counts
// the block's chunks written), remembering the last count of every block.
struct GramFeed {
  const int32_t* ready;  // this stream's [nblk] counters, or nullptr (the pre-pass has finished)
  int nblk;              // blocks of the pre-pass per stream
  int* cnt;              // [nblk] last counter value read (shared memory, thread 0)
};
__device__ __forceinline__ bool gram_feed_wait(GramFeed& f, int gc, volatile int* abort, int32_t* status) {
  if (!f.ready) return true;
  const int blk = gc % f.nblk, need = gc / f.nblk + 1;
  if (f.cnt[blk] < need) {
    const long long t0 = clock64();
    long long lim = -1;
    while (true) {
      const int c = ld_acquire_gpu(f.ready + blk);
      if (c >= need) {
        f.cnt[blk] = c;
        break;
      }
      if (*abort) return false;
      if (*(volatile int32_t*)status != 0 || sm100::wait_expired(t0, lim, status)) {
        *abort = 1;
        atomicCAS(status, 0, sm100::kStatusTimeout);
        return false;
      }
    }
  }
  asm volatile("fence.proxy.async.global;" ::: "memory");  // the block is read by a bulk copy
  return true;
}

// Next chunk's k and v rows (cp.async by threads i0, i0 + ni, ..., zero-filled
// past the sequence end) and its Gram block gc (one bulk copy by thread i0,
// completing on `bar`, skipped after a failed wait for the pre-pass, which sets
// the abort flag).  The k, v copies are waited for with cp.async.wait_group by
// the threads that issued them, the Gram block with the mbarrier.
// With inputs streamed in by the host (piece_ready non-null), every issuing
// thread first waits (acquire, bounded) until the piece holding the chunk has
// arrived: piece_need pieces, the count last read kept in piece_known.
template <int D>
__device__ __forceinline__ void prefetch_chunk(__nv_bfloat16* dk, __nv_bfloat16* dv, const __nv_bfloat16* ks,
                                               const __nv_bfloat16* vs, int row_stride, int valid, float* dgq,
                                               const float* gsrc, uint64_t* bar, GramFeed& feed, int gc,
                                               volatile int* abort, int32_t* status, int i0, int ni,
                                               const int32_t* piece_ready, int piece_need, int& piece_known) {
  constexpr int RP = D + 8;
  constexpr int V16 = D / 8;
  if (piece_ready && piece_known < piece_need) {
    const long long t0 = clock64();
    long long lim = -1;
    while ((piece_known = ld_acquire_gpu(piece_ready)) < piece_need) {
      if (*abort) break;
      if (*(volatile int32_t*)status != 0 || sm100::wait_expired(t0, lim, status)) {
        *abort = 1;
        atomicCAS(status, 0, sm100::kStatusTimeout);
        break;
      }
    }
  }
  if (i0 == 0 && gsrc && gram_feed_wait(feed, gc, abort, status)) {
    sm100::mbar_expect_tx(bar, (uint32_t)kGramBlock * 4u);
    sm100::bulk_g2s(dgq, gsrc, (uint32_t)kGramBlock * 4u, bar);
  }
  for (int e = i0; e < L * V16; e += ni) {
    const int r = e / V16, c = (e % V16) * 8;
    const int nbytes = (r < valid) ? 16 : 0;
    const __nv_bfloat16* sk = (r < valid) ? ks + (long long)r * row_stride + c : ks;
    const __nv_bfloat16* sv = (r < valid) ? vs + (long long)r * row_stride + c : vs;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(su32(dk + r * RP + c)), "l"(sk), "r"(nbytes)
                 : "memory");
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(su32(dv + r * RP + c)), "l"(sv), "r"(nbytes)
                 : "memory");
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
}

// Gram entries of one chunk with mma.sync: Gout[t][s] = (k_t.k_s)(v_t.v_s) for
// s < t (0 elsewhere, row stride L + 1), aout[t] = |k_t|^2 |v_t|^2.  All 8
// warps; warp w takes the 16-token band w % 4 and the 32 columns w / 4.
template <int D>
__device__ __forceinline__ void gram_tile(const __nv_bfloat16* Ks, const __nv_bfloat16* Vs, float* Gout, float* aout) {
  constexpr int RP = D + 8;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> 2, tg = lane & 3, q = lane >> 3, r8 = lane & 7;
  const int mt = warp & 3, sb = 32 * (warp >> 2);
  float kk4[4][4], vv4[4][4];
#pragma unroll
  for (int n = 0; n < 4; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) kk4[n][e] = vv4[n][e] = 0.f;
#pragma unroll 2
  for (int kk = 0; kk < D; kk += 16) {
    uint32_t ak[4], av[4];
    ldsm4(ak, Ks + (16 * mt + (q & 1) * 8 + r8) * RP + kk + (q >> 1) * 8);
    ldsm4(av, Vs + (16 * mt + (q & 1) * 8 + r8) * RP + kk + (q >> 1) * 8);
#pragma unroll
    for (int np = 0; np < 2; ++np) {
      uint32_t bk[4], bv[4];
      ldsm4(bk, Ks + (sb + 16 * np + (q >> 1) * 8 + r8) * RP + kk + (q & 1) * 8);
      ldsm4(bv, Vs + (sb + 16 * np + (q >> 1) * 8 + r8) * RP + kk + (q & 1) * 8);
      mma16816(kk4[2 * np], ak, bk[0], bk[1]);
      mma16816(kk4[2 * np + 1], ak, bk[2], bk[3]);
      mma16816(vv4[2 * np], av, bv[0], bv[1]);
      mma16816(vv4[2 * np + 1], av, bv[2], bv[3]);
    }
  }
#pragma unroll
  for (int n = 0; n < 4; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int t = 16 * mt + g + 8 * (e >> 1);
      const int s2 = sb + 8 * n + 2 * tg + (e & 1);
      const float gv = kk4[n][e] * vv4[n][e];
      Gout[t * (L + 1) + s2] = (s2 < t) ? gv : 0.f;
      if (s2 == t) aout[t] = gv;
    }
}

// gram_tile computing only the 16 x 16 tiles on or below the diagonal (the
// Gram pre-pass; the scan keeps its own copy).
template <int D>
__device__ __forceinline__ void gram_tile_lower(const __nv_bfloat16* Ks, const __nv_bfloat16* Vs, float* Gout, float* aout) {
  constexpr int RP = D + 8;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> 2, tg = lane & 3, q = lane >> 3, r8 = lane & 7;
  const int mt = warp & 3, sb = 32 * (warp >> 2);
  // only 16 x 16 tiles with columns s <= the band's last row are needed (s < t,
  // and the diagonal for a_t): column block sb / 16 + np against row band mt
  const bool need0 = (sb >> 4) <= mt, need1 = (sb >> 4) + 1 <= mt;  // warp-uniform
  float kk4[4][4], vv4[4][4];
#pragma unroll
  for (int n = 0; n < 4; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) kk4[n][e] = vv4[n][e] = 0.f;
#pragma unroll 2
  for (int kk = 0; kk < D; kk += 16) {
    if (!need0) break;
    uint32_t ak[4], av[4];
    ldsm4(ak, Ks + (16 * mt + (q & 1) * 8 + r8) * RP + kk + (q >> 1) * 8);
    ldsm4(av, Vs + (16 * mt + (q & 1) * 8 + r8) * RP + kk + (q >> 1) * 8);
#pragma unroll
    for (int np = 0; np < 2; ++np) {
      if (np == 1 && !need1) continue;
      uint32_t bk[4], bv[4];
      ldsm4(bk, Ks + (sb + 16 * np + (q >> 1) * 8 + r8) * RP + kk + (q & 1) * 8);
      ldsm4(bv, Vs + (sb + 16 * np + (q >> 1) * 8 + r8) * RP + kk + (q & 1) * 8);
      mma16816(kk4[2 * np], ak, bk[0], bk[1]);
      mma16816(kk4[2 * np + 1], ak, bk[2], bk[3]);
      mma16816(vv4[2 * np], av, bv[0], bv[1]);
      mma16816(vv4[2 * np + 1], av, bv[2], bv[3]);
    }
  }
#pragma unroll
  for (int n = 0; n < 4; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int t = 16 * mt + g + 8 * (e >> 1);
      const int s2 = sb + 8 * n + 2 * tg + (e & 1);
      const float gv = kk4[n][e] * vv4[n][e];
      Gout[t * (L + 1) + s2] = (s2 < t) ? gv : 0.f;
      if (s2 == t) aout[t] = gv;
    }
}

// Row suffix sums in place: G[t][j] <- sum_{j <= s < t} G[t][s] (a warp per row).
__device__ __forceinline__ void suffix_rows(float* G) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int t = warp; t < L; t += NW) {
    float* row = G + t * (L + 1);
    const float g0 = row[2 * lane], g1 = row[2 * lane + 1];
    float r = g0 + g1;  // reverse inclusive scan over lanes
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float dn = __shfl_down_sync(0xffffffffu, r, o);
      if (lane + o < 32) r += dn;
    }
    const float after = __shfl_down_sync(0xffffffffu, r, 1);
    const float tail = (lane < 31) ? after : 0.f;
    row[2 * lane + 1] = g1 + tail;
    row[2 * lane] = g0 + g1 + tail;
  }
}

// Exclusive prefix sums along rows: dst[j * ds + t] = sum_{u < t} src[j * rs + u * cs]
// (a warp per row j, two elements per lane).
__device__ __forceinline__ void prefix_rows(const float* src, int rs, int cs, float* dst, int ds) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int j = warp; j < L; j += NW) {
    const float g0 = src[j * rs + (2 * lane) * cs], g1 = src[j * rs + (2 * lane + 1) * cs];
    float inc = g0 + g1;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float up = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += up;
    }
    float ex = __shfl_up_sync(0xffffffffu, inc, 1);
    if (lane == 0) ex = 0.f;
    dst[j * ds + 2 * lane] = ex;
    dst[j * ds + 2 * lane + 1] = ex + g0;
  }
}

// suffix_rows / prefix_rows with the warp's L / NW rows scanned together (as
// many independent shuffle chains; the same sums in the same order per row), for
// the Gram pre-pass, which has the registers to spare.
__device__ __forceinline__ void suffix_rows_ilp(float* G) {
  constexpr int R = L / NW;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float g0[R], g1[R], r[R];
#pragma unroll
  for (int i = 0; i < R; ++i) {
    const float* row = G + (warp + i * NW) * (L + 1);
    g0[i] = row[2 * lane];
    g1[i] = row[2 * lane + 1];
    r[i] = g0[i] + g1[i];
  }
#pragma unroll
  for (int o = 1; o < 32; o <<= 1)
#pragma unroll
    for (int i = 0; i < R; ++i) {
      const float dn = __shfl_down_sync(0xffffffffu, r[i], o);
      if (lane + o < 32) r[i] += dn;
    }
#pragma unroll
  for (int i = 0; i < R; ++i) {
    const float after = __shfl_down_sync(0xffffffffu, r[i], 1);
    const float tail = (lane < 31) ? after : 0.f;
    float* row = G + (warp + i * NW) * (L + 1);
    row[2 * lane + 1] = g1[i] + tail;
    row[2 * lane] = g0[i] + g1[i] + tail;
  }
}
__device__ __forceinline__ void prefix_rows_ilp(const float* src, int rs, int cs, float* dst, int ds) {
  constexpr int R = L / NW;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float g0[R], inc[R];
#pragma unroll
  for (int i = 0; i < R; ++i) {
    const int j = warp + i * NW;
    g0[i] = src[j * rs + (2 * lane) * cs];
    inc[i] = g0[i] + src[j * rs + (2 * lane + 1) * cs];
  }
#pragma unroll
  for (int o = 1; o < 32; o <<= 1)
#pragma unroll
    for (int i = 0; i < R; ++i) {
      const float up = __shfl_up_sync(0xffffffffu, inc[i], o);
      if (lane >= o) inc[i] += up;
    }
#pragma unroll
  for (int i = 0; i < R; ++i) {
    float ex = __shfl_up_sync(0xffffffffu, inc[i], 1);
    if (lane == 0) ex = 0.f;
    const int j = warp + i * NW;
    dst[j * ds + 2 * lane] = ex;
    dst[j * ds + 2 * lane + 1] = ex + g0[i];
  }
}

// State copies (NR rows of a D x D state) move NR*D/4/NT float4 per thread;
// loads are issued in batches (four for copies, up to eight for adds and fp16
// conversions: measured 2.5 % off the scan) before their stores so that a copy
// costs a few memory latencies, not one per element (the compiler cannot
// reorder a load past a possibly aliasing store).  A bf16 pool entry is hi rows [D][D]
// followed by lo rows [D][D]: dst points at this CTA's first hi row.
template <int D, int NR = D>
__device__ __forceinline__ void copy_state_g(float* dst, const float* src) {
  constexpr int PER = NR * D / 4 / NT;
  for (int base = 0; base < PER; base += 4) {
    float4 v[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) v[i] = load4(src + ((base + i) * NT + threadIdx.x) * 4);
#pragma unroll
    for (int i = 0; i < 4; ++i) store4(dst + ((base + i) * NT + threadIdx.x) * 4, v[i]);
  }
}
// NR rows of an fp32 state into an fp16 pool entry (scaled by inv = 1 / s), by
// threads i0, i0 + ni, ...
template <int D, int NR>
__device__ __forceinline__ void copy_state_f16(__half* dst, const float* src, float inv, int i0, int ni) {
  constexpr int N4 = NR * D / 4;
  for (int base = i0; base < N4; base += 8 * ni) {
    float4 v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int e4 = base + i * ni;
      v[i] = (e4 < N4) ? load4(src + e4 * 4) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int e4 = base + i * ni;
      if (e4 < N4) *reinterpret_cast<uint2*>(dst + e4 * 4) = f16x4(v[i], inv);
    }
  }
}
// (x, y) as packed bf16 hi = bf16(x, y) and lo = bf16(x - hi, y - hi): the
// open state's operand split, as the publish stores it.
__device__ __forceinline__ void split_hi_lo(float x, float y, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(x, y);
  const float2 f = __bfloat1622float2(h);
  const __nv_bfloat162 l = __floats2bfloat162_rn(x - f.x, y - f.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

// dst += src over one D x D state, batched like copy_state_g.
template <int D, int NR = D>
__device__ __forceinline__ void add_state_g(float* dst, const float* src) {
  constexpr int PER = NR * D / 4 / NT;
  constexpr int BAT = PER < 8 ? PER : 8;
  for (int base = 0; base < PER; base += BAT) {
    float4 x[BAT], y[BAT];
#pragma unroll
    for (int i = 0; i < BAT; ++i) {
      const int e = ((base + i) * NT + threadIdx.x) * 4;
      x[i] = load4(dst + e);
      y[i] = load4(src + e);
    }
#pragma unroll
    for (int i = 0; i < BAT; ++i)
      store4(dst + ((base + i) * NT + threadIdx.x) * 4,
             make_float4(x[i].x + y[i].x, x[i].y + y[i].y, x[i].z + y[i].z, x[i].w + y[i].w));
  }
}

// One pair of adjacent state elements (k, k+1 of row j) into an fp32 pool entry.
__device__ __forceinline__ void put_pair(float* entry, int D, int j, int k, float v0, float v1) {
  *reinterpret_cast<float2*>(entry + j * D + k) = make_float2(v0, v1);
}

}  // namespace

// One stream per CTA (CL = 1) or per CTA pair (CL = 2, a thread-block
// cluster): with a pair, each CTA owns d/2 rows of the open state (and of every
// state it copies or adds), forms its part of x_t and |S_open|^2, and the two
// parts meet through distributed shared memory once per chunk; both CTAs then
// take the same decisions from the same sums (x = part of rank 0 + part of
// rank 1 in both), and rank 0 writes the trace, the lists and the metadata.
// kRagged: per-row lengths (padding after them); a separate instance, so the
// common one keeps its code.
template <int D, typename Tpool, int CL, bool kRagged = false, int CAPB = kMaxC>
__global__ void __launch_bounds__(NT, 1) scan_mma_kernel(ScanArgs a) {
  constexpr bool kBig = CAPB > kMaxC;  // DLA(I): up to CAPB states, no capacity merge
  constexpr int RP = D + 8;
  constexpr int R = D / CL;           // state rows of this CTA
  constexpr int MT = R / 16;          // 16-row bands of those rows
  constexpr int WPM = NW / MT;        // warps per band
  constexpr int KC = D / WPM;         // state columns per warp
  constexpr int NT8 = KC / 8;         // n8 tiles per warp in the state build
  static_assert(L == 64 && KC % 16 == 0, "x GEMM tiling");
  extern __shared__ __align__(16) unsigned char smem_raw[];
  MmaSmem<D, CL, CAPB>& sm = *reinterpret_cast<MmaSmem<D, CL, CAPB>*>(smem_raw);

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = lane >> 2, tg = lane & 3;
  const int rank = (CL > 1) ? (int)cluster_rank() : 0;
  const bool lead = (rank == 0);      // writes what both CTAs of a pair hold
  const int bh = blockIdx.x / CL;
  const int b = bh / a.H, h = bh % a.H;
  const int C = a.C;
  const float Df = (float)(D * D);
  // token row of the row's first token (the packed layout only in the per-row-length instance)
  const long long tok0 = kRagged ? row_tok0(a.row_start, b, a.T) : (long long)b * a.T;
  const __nv_bfloat16* kbase = reinterpret_cast<const __nv_bfloat16*>(a.k) + (tok0 * a.H + h) * D;
  const __nv_bfloat16* vbase = reinterpret_cast<const __nv_bfloat16*>(a.v) + (tok0 * a.H + h) * D;
  const int row_stride = a.H * D;
  const int rbase = rank * R;         // first state row of this CTA
  float* states = a.states + (long long)bh * C * D * D;
  constexpr long long kEntry = (long long)D * D;
  constexpr bool kF16 = sizeof(Tpool) == 2;  // fp16 pool entries (tensor-core read-out)
  Tpool* pool = a.pool ? reinterpret_cast<Tpool*>(a.pool) + (long long)bh * a.pool_cap * kEntry : nullptr;
  uint8_t* bnd_out = a.boundary + (long long)bh * a.T;
  int32_t* mlog_out = a.merge_log + (long long)bh * a.T;
  // this CTA's rows of state slot p
  auto srows = [&](int p) { return states + (long long)p * D * D + (long long)rbase * D; };

  // this warp's band of the open state: local rows j0 .. j0+15 (global rbase + j0 ..),
  // columns k0 .. k0+KC-1
  const int j0 = 16 * (warp % MT), k0 = KC * (warp / MT);
  const int jg0 = rbase + j0;
  float acc[NT8][4];

  // ---------------------------------------------------------------- round start
  if (tid == 0) {
    if (a.started) atomicAdd(a.started, 1);  // the read-out stream's gate counts the resident scan CTAs
    int m0 = a.m[bh];
    if (m0 < 0 || m0 > C) {
      atomicExch(a.status, 6);
      m0 = 0;
    }
    sm.m = m0;
    sm.pool_next = 0;
    sm.pend = 0;
    sm.abort_flag = 0;
    sm100::mbar_init(&sm.kvbar[0], 1);
    sm100::mbar_init(&sm.kvbar[1], 1);
    if constexpr (CL > 1) {
      sm100::mbar_init(&sm.xbar[0], 1);
      sm100::mbar_init(&sm.xbar[1], 1);
    }
    sm100::fence_mbar_init();
  }
  __syncthreads();
  for (int i = tid; i < C; i += NT) {
    int sl = a.slot[(long long)bh * C + i];
    if (sl < 0 || sl >= C) {
      atomicExch(a.status, 6);
      sl = i;
    }
    sm.slot[i] = sl;
  }
  __syncthreads();
  const int m_start = sm.m;
  if (tid == 0) sm.open_slot = (m_start > 0) ? sm.slot[m_start - 1] : 0;  // rewritten by every replay
  // Warp 0 keeps n, Ibar, physical slot, pool id, "changed since the last
  // snapshot" and (fp16 pool) an upper bound of |S|_F of every entry in
  // registers (entry i: lane i % 32, element i / 32).
  int e_n[2] = {0, 0}, e_slot[2] = {0, 0}, e_pid[2] = {-1, -1}, e_dirty[2] = {0, 0};
  double e_ib[2] = {0.0, 0.0};
  float e_nb[2] = {0.f, 0.f};
  if constexpr (kBig) {  // in shared memory: n, Ibar, pool id, changed, norm bound
    for (int i = tid; i < C; i += NT) {
      sm.bn[i] = a.n[(long long)bh * C + i];
      sm.bib[i] = a.ibar[(long long)bh * C + i];
      sm.bpid[i] = -1;
      sm.bdirty[i] = 0;
      sm.bnb[i] = (kF16 && pool && i < m_start) ? a.nbound[(long long)bh * C + i] : 0.f;
      // no merge ever freed a physical slot: the live entries use slots 0 .. m - 1
      if (i < m_start && sm.slot[i] >= m_start) atomicCAS(a.status, 0, 6);
    }
  } else if (warp == 0) {
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int i = lane + 32 * r;
      if (i < C) {
        e_n[r] = a.n[(long long)bh * C + i];
        e_ib[r] = a.ibar[(long long)bh * C + i];
        e_slot[r] = sm.slot[i];
        if (kF16 && pool && i < m_start) e_nb[r] = a.nbound[(long long)bh * C + i];
      }
    }
  }
  {
    const float* src = m_start > 0 ? states + (long long)sm.slot[m_start - 1] * D * D : nullptr;
#pragma unroll
    for (int n = 0; n < NT8; ++n) {
      const int k = k0 + 8 * n + 2 * tg;
      float2 lo = make_float2(0.f, 0.f), hi = make_float2(0.f, 0.f);
      if (src) {
        lo = *reinterpret_cast<const float2*>(src + (jg0 + g) * D + k);
        hi = *reinterpret_cast<const float2*>(src + (jg0 + g + 8) * D + k);
      }
      acc[n][0] = lo.x; acc[n][1] = lo.y; acc[n][2] = hi.x; acc[n][3] = hi.y;
    }
  }
  if (pool) {
    const long long lst = (long long)bh * a.snap_stride + a.snap_base;  // list row of this round's first interval
    if (a.carry_in) {  // the pool continues: the previous round wrote this interval's list
      if (tid == 0) sm.pool_next = a.pstate[bh];
      if constexpr (kBig) {
        for (int i = tid; i < m_start; i += NT) sm.bpid[i] = a.pstate[a.B * a.H + (long long)bh * C + i];
      } else if (warp == 0) {
#pragma unroll
        for (int r = 0; r < 2; ++r)
          if (lane + 32 * r < m_start) e_pid[r] = a.pstate[a.B * a.H + (long long)bh * C + lane + 32 * r];
      }
    } else {  // snapshot 0: every live entry at the start of the round
      if constexpr (kF16) {
        if constexpr (kBig) {
          __syncthreads();  // the norm bounds above
          for (int i = tid; i < m_start && i < a.pool_cap; i += NT) {
            const float sc = f16_scale(sm.bnb[i]);
            sm.snap_scale[i] = sc;
            sm.bpid[i] = i;
            if (lead) a.pool_scale[(long long)bh * a.pool_cap + i] = sc;
          }
        } else if (warp == 0) {
#pragma unroll
          for (int r = 0; r < 2; ++r) {
            const int i = lane + 32 * r;
            if (i < m_start && i < a.pool_cap) {
              const float sc = f16_scale(e_nb[r]);
              sm.snap_scale[i] = sc;
              if (lead) a.pool_scale[(long long)bh * a.pool_cap + i] = sc;
            }
          }
        }
        __syncthreads();
        for (int i = 0; i < m_start && i < a.pool_cap; ++i)
          copy_state_f16<D, R>(pool + (long long)i * kEntry + (long long)rbase * D, srows(sm.slot[i]),
                               1.f / sm.snap_scale[i], tid, NT);
      } else {
        for (int i = 0; i < m_start && i < a.pool_cap; ++i)
          copy_state_g<D, R>(pool + (long long)i * kEntry + (long long)rbase * D, srows(sm.slot[i]));
      }
      if (warp == 0)
#pragma unroll
        for (int r = 0; r < 2; ++r)
          if (lane + 32 * r < m_start) e_pid[r] = lane + 32 * r;
      if (tid == 0) sm.pool_next = m_start;
      if (lead) {
        if (tid == 0) a.snap_m0[lst] = m_start;
        for (int i = tid; i < m_start; i += NT) a.snap_ids[lst * C + i] = i;
      }
    }
  }

  // this CTA's rows of the open state -> bf16 hi / lo operand, and its part of
  // |S_open|^2 into xs[buf][rank][L]
  auto publish_state = [&](int buf) {
    float gp = 0.f;
#pragma unroll
    for (int n = 0; n < NT8; ++n) {
      const int k = k0 + 8 * n + 2 * tg;
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        const float v0 = acc[n][2 * hf], v1 = acc[n][2 * hf + 1];
        const int j = j0 + g + 8 * hf;
        const __nv_bfloat162 hi = __floats2bfloat162_rn(v0, v1);
        const float2 f = __bfloat1622float2(hi);
        *reinterpret_cast<__nv_bfloat162*>(&sm.S2[0][j * RP + k]) = hi;
        *reinterpret_cast<__nv_bfloat162*>(&sm.S2[1][j * RP + k]) = __floats2bfloat162_rn(v0 - f.x, v1 - f.y);
        gp += v0 * v0 + v1 * v1;
      }
    }
    gp = warp_sum(gp);
    if (lane == 0) sm.gred[warp] = gp;
    __syncthreads();
    if (tid == 0) {
      float gs = 0.f;
      for (int w = 0; w < NW; ++w) gs += sm.gred[w];
      sm.xs[buf][rank][L] = gs;
    }
  };
  // acc += V^T K over chunk tokens [u0, u1) of stage st
  auto build = [&](int st, int u0, int u1) {
    const __nv_bfloat16* Ks = sm.kv[st][0];
    const __nv_bfloat16* Vs = sm.kv[st][1];
    const int q = lane >> 3, r8 = lane & 7;
    for (int ks = 0; ks < L / 16; ++ks) {
      const int t0 = 16 * ks;
      if (t0 >= u1 || t0 + 16 <= u0) continue;
      uint32_t af[4];
      ldsm4t(af, Vs + (t0 + (q >> 1) * 8 + r8) * RP + jg0 + (q & 1) * 8);
      af[0] = mask_pair(af[0], t0 + 2 * tg, u0, u1);
      af[1] = mask_pair(af[1], t0 + 2 * tg, u0, u1);
      af[2] = mask_pair(af[2], t0 + 8 + 2 * tg, u0, u1);
      af[3] = mask_pair(af[3], t0 + 8 + 2 * tg, u0, u1);
#pragma unroll
      for (int np = 0; np < NT8 / 2; ++np) {
        uint32_t bf[4];
        ldsm4t(bf, Ks + (t0 + (q & 1) * 8 + r8) * RP + k0 + 16 * np + (q >> 1) * 8);
        mma16816(acc[2 * np], af, bf[0], bf[1]);
        mma16816(acc[2 * np + 1], af, bf[2], bf[3]);
      }
    }
  };
  // The snapshot copies listed in sm.snap_src[0 .. n) into fp16 pool entries
  // (scaled by 1 / sm.snap_scale): the open state from its bf16 hi / lo operand
  // in shared memory (hi + lo is the fp32 value to 2^-17), closed states from
  // their fp32 slots.  Threads i0, i0 + ni, ...
  auto snapshot_copies = [&](int n, int i0, int ni) {
    for (int jj = 0; jj < n; ++jj) {
      const int p = sm.snap_src[jj][0], srcslot = sm.snap_src[jj][1];
      const float inv = 1.f / sm.snap_scale[jj];
      Tpool* entry = pool + (long long)p * kEntry;
      if constexpr (kF16) {
        if (srcslot < 0) {  // 8 elements per 16-byte store, rows in order
          for (int e = i0; e < R * (D / 8); e += ni) {
            const int j = e / (D / 8), k8 = (e % (D / 8)) * 8;
            const uint4 hv = *reinterpret_cast<const uint4*>(&sm.S2[0][j * RP + k8]);
            const uint4 lv = *reinterpret_cast<const uint4*>(&sm.S2[1][j * RP + k8]);
            const uint32_t hw[4] = {hv.x, hv.y, hv.z, hv.w}, lw[4] = {lv.x, lv.y, lv.z, lv.w};
            float f[8];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const float2 h2 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&hw[i]));
              const float2 l2 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&lw[i]));
              f[2 * i] = h2.x + l2.x;
              f[2 * i + 1] = h2.y + l2.y;
            }
            const uint2 a0 = f16x4(make_float4(f[0], f[1], f[2], f[3]), inv);
            const uint2 a1 = f16x4(make_float4(f[4], f[5], f[6], f[7]), inv);
            *reinterpret_cast<uint4*>(entry + (rbase + j) * D + k8) = make_uint4(a0.x, a0.y, a1.x, a1.y);
          }
        } else {
          copy_state_f16<D, R>(entry + (long long)rbase * D, srows(srcslot), inv, i0, ni);
        }
      }
    }
  };
  // x_t or |S_open|^2 of the whole state (index i of xs[buf][.]): the CTAs'
  // parts added in rank order
  auto whole = [&](int buf, int i) -> float {
    if constexpr (CL == 1) {
      return sm.xs[buf][0][i];
    } else {
      return sm.xs[buf][0][i] + sm.xs[buf][1][i];
    }
  };

  if constexpr (CL > 1) cluster_sync();  // both CTAs run (barriers initialised) before the first exchange
  publish_state(0);
  __syncthreads();

  // this row's end of the round (the call's t_end unless per-row lengths are given)
  const int t_end_r = kRagged ? row_t_end(a.seq_lens, b, a.t_begin, a.t_end) : 0;
#define DLA_T_END (kRagged ? t_end_r : a.t_end)
  const int ntok = DLA_T_END - a.t_begin;
  const int nchunks = (ntok + L - 1) / L;
  const long long gchunk0 = (long long)bh * a.gram_chunks + a.t_begin / L;  // Gram block of the round's first chunk
  GramFeed feed;
  feed.ready = a.gram_ready ? a.gram_ready + (long long)bh * a.gram_nblk : nullptr;
  feed.nblk = a.gram_nblk;
  feed.cnt = sm.gcnt;
  int piece_known = 0;  // streamed inputs: pieces known to have arrived (this thread)
  if (tid == 0)
    for (int i = 0; i < kMaxGramBlk; ++i) sm.gcnt[i] = 0;
  if (!kRagged || ntok > 0)  // a row that ended before this round has no chunk to load
  prefetch_chunk<D>(sm.kv[0][0], sm.kv[0][1], kbase + (long long)a.t_begin * row_stride,
                      vbase + (long long)a.t_begin * row_stride, row_stride, min(L, ntok), sm.gq[0],
                      a.gram ? a.gram + gchunk0 * kGramStride : nullptr, &sm.kvbar[0], feed, a.t_begin / L,
                      &sm.abort_flag, a.status, tid, NT, a.piece_ready,
                      a.piece_chunks ? a.t_begin / L / a.piece_chunks + 1 : 0, piece_known);
  int rel_pending = 0;  // thread NT - 32: progress value not yet released
  for (int c = 0; c < nchunks; ++c) {
    const int t0 = a.t_begin + c * L;
    const int Lc = min(L, DLA_T_END - t0);
    const int st = c & 1;
    // ------------------------------------------------ 1. k, v of this chunk (issued during the
    // previous chunk's passes, or before the loop)
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    if (a.gram) sm100::mbar_wait(&sm.kvbar[st], (uint32_t)((c >> 1) & 1), &sm.abort_flag, a.status);
    if (tid < L) sm.mlog[tid] = -1;
    __syncthreads();
    const int m_chunk = sm.m;
    const __nv_bfloat16* Ks = sm.kv[st][0];
    const __nv_bfloat16* Vs = sm.kv[st][1];
    const int q = lane >> 3, r8 = lane & 7;
    // ------------------------------------------------ 2. x_t = v_t^T S_open k_t (this CTA's rows)
    // Each warp adds sum_{j, k} v_t[j] S[j][k] k_t[k] over its band of the open
    // state (rows j0 .. j0 + 15, columns k0 .. k0 + KC - 1): S straight from its
    // accumulators (two m16n8 accumulator tiles are the m16n8k16 A fragment of
    // those 16 columns) as bf16 hi + lo, k_t from the chunk's K tile, so that
    // Y[j][t] = sum_k S[j][k] k_t[k] on mma.sync; then the v_t[j] weights.
    if (m_chunk > 0) {
      float Y[L / 8][4];
#pragma unroll
      for (int n = 0; n < L / 8; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e) Y[n][e] = 0.f;
#pragma unroll
      for (int s8 = 0; s8 < KC / 16; ++s8) {
        uint32_t ah[4], al[4];
        split_hi_lo(acc[2 * s8][0], acc[2 * s8][1], ah[0], al[0]);          // row g, k 2tg, 2tg + 1
        split_hi_lo(acc[2 * s8][2], acc[2 * s8][3], ah[1], al[1]);          // row g + 8
        split_hi_lo(acc[2 * s8 + 1][0], acc[2 * s8 + 1][1], ah[2], al[2]);  // row g, k 2tg + 8, 2tg + 9
        split_hi_lo(acc[2 * s8 + 1][2], acc[2 * s8 + 1][3], ah[3], al[3]);  // row g + 8
#pragma unroll
        for (int np = 0; np < L / 16; ++np) {  // tokens 16 np .. 16 np + 15: two n8 tiles
          uint32_t bf[4];
          ldsm4(bf, Ks + (16 * np + (q >> 1) * 8 + r8) * RP + k0 + 16 * s8 + (q & 1) * 8);
          mma16816(Y[2 * np], ah, bf[0], bf[1]);
          mma16816(Y[2 * np], al, bf[0], bf[1]);
          mma16816(Y[2 * np + 1], ah, bf[2], bf[3]);
          mma16816(Y[2 * np + 1], al, bf[2], bf[3]);
        }
      }
      // this thread's terms: tokens 8n + 2tg (+1) of rows jg0 + g and jg0 + g + 8
      float pv[L / 4];  // [2n + e]: token 8n + 2tg + e
      const int ja = jg0 + g, jb = ja + 8;
#pragma unroll
      for (int n = 0; n < L / 8; ++n) {
        const int t = 8 * n + 2 * tg;
        pv[2 * n] = Y[n][0] * __bfloat162float(Vs[t * RP + ja]) + Y[n][2] * __bfloat162float(Vs[t * RP + jb]);
        pv[2 * n + 1] =
            Y[n][1] * __bfloat162float(Vs[(t + 1) * RP + ja]) + Y[n][3] * __bfloat162float(Vs[(t + 1) * RP + jb]);
      }
      // sum over the eight lanes of equal tg (g = 0 .. 7) by halving exchanges
      // (lane bits 4, 3, 2 = bits 2, 1, 0 of g): afterwards lane (g, tg) holds
      // tokens 8g + 2tg and 8g + 2tg + 1 in pv[0], pv[1]
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const bool up = (g & 4) != 0;
        const float send = up ? pv[k] : pv[8 + k], keep = up ? pv[8 + k] : pv[k];
        pv[k] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const bool up = (g & 2) != 0;
        const float send = up ? pv[k] : pv[4 + k], keep = up ? pv[4 + k] : pv[k];
        pv[k] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
      }
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const bool up = (g & 1) != 0;
        const float send = up ? pv[k] : pv[2 + k], keep = up ? pv[2 + k] : pv[k];
        pv[k] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
      }
      sm.red[warp][8 * g + 2 * tg] = pv[0];
      sm.red[warp][8 * g + 2 * tg + 1] = pv[1];
    }
    // ------------------------------------------------ 3. Gram suffix table and a_t
    // Normally prefetched from the Gram pre-pass; formed here when the call has
    // no room for the pre-pass output (scan-only calls).
    if (!a.gram) {
      float* G = sm.gq[st ^ 1];  // scratch: no Gram block is prefetched into the other stage here
      gram_tile<D>(Ks, Vs, G, sm.gq[st] + 2 * L * L);
      __syncthreads();
      suffix_rows(G);
      __syncthreads();
      for (int e = tid; e < L * L; e += NT) {  // transpose to the [j][t] layout the passes read
        const int t = e % L, j = e / L;
        sm.gq[st][j * GS + t] = G[t * (L + 1) + j];
      }
      __syncthreads();
      prefix_rows(sm.gq[st], GS, 1, sm.gq[st] + L * L, GS);
      if (warp == 0) norm_prefix_warp(sm.gq[st] + 2 * L * L, sm.gq[st] + kGramSA, lane);
    }
    __syncthreads();
    if (tid < L) {  // this CTA's part of x_t
      float x = 0.f;
      if (m_chunk > 0)
#pragma unroll
        for (int w8 = 0; w8 < NW; ++w8) x += sm.red[w8][tid];
      sm.xs[st][rank][tid] = x;
      if constexpr (CL > 1) {  // this CTA's parts of x_t and |S_open|^2 into the partner's copy
        const uint32_t peer = (uint32_t)(rank ^ 1);
        const uint32_t rbar = mapa_u32(&sm.xbar[st], peer);
        st_async_f32(mapa_u32(&sm.xs[st][rank][tid], peer), x, rbar);
        if (tid == 0) st_async_f32(mapa_u32(&sm.xs[st][rank][L], peer), sm.xs[st][rank][L], rbar);
      }
    }
    __syncthreads();
    // ------------------------------------------------ 3b. work beside warp 0's passes (warps 1..)
    // First the progress word of the interval that ended with the last chunk:
    // here the wait of its release for earlier memory operations costs warp 0
    // nothing, and issued before the loads below it does not wait for them.
    if (rel_pending > 0) {
      st_release_gpu(a.progress + 2 * bh + rank, rel_pending);
      rel_pending = 0;
    }
    // The next chunk's k, v and Gram block are issued here as well (warps 1..;
    // buffers st ^ 1, which the previous chunk used, are free).
    if (warp != 0 && c + 1 < nchunks) {
      const int t1 = t0 + L;
      prefetch_chunk<D>(sm.kv[st ^ 1][0], sm.kv[st ^ 1][1], kbase + (long long)t1 * row_stride,
                        vbase + (long long)t1 * row_stride, row_stride, min(L, DLA_T_END - t1), sm.gq[st ^ 1],
                        a.gram ? a.gram + (gchunk0 + c + 1) * kGramStride : nullptr, &sm.kvbar[st ^ 1], feed,
                        a.t_begin / L + c + 1, &sm.abort_flag, a.status, tid - 32, NT - 32, a.piece_ready,
                        a.piece_chunks ? (a.t_begin / L + c + 1) / a.piece_chunks + 1 : 0, piece_known);
    }
    // Then the previous interval's snapshot copies: they read the staged open
    // state and closed slots, which only the state updates and the publish below
    // change.
    if constexpr (sizeof(Tpool) == 2)
      if (warp != 0 && sm.pend > 0) snapshot_copies(sm.pend, tid - 32, NT - 32);
    // ------------------------------------------------ 4. boundary passes (warp 0, tokens 2 lane, 2 lane + 1)
    // Each pass scores every undecided token as if the open segment ran to it,
    // takes the first that fires, and restarts the segment there.
    // ------------------------------------------------ 5. replay of the decisions (Algorithm 2, warp 0)
    if (warp == 0) {
      if constexpr (CL > 1) {  // the partner's parts (L + 1 floats) for this chunk
        if (lane == 0) sm100::mbar_expect_tx(&sm.xbar[st], (L + 1) * 4);
        __syncwarp();
        sm100::mbar_wait_cluster(&sm.xbar[st], (uint32_t)((c >> 1) & 1), &sm.abort_flag, a.status);
      }
      const int ta = 2 * lane, tb = ta + 1;
      const float xa = (m_chunk > 0) ? whole(st, ta) : 0.f;
      const float xb = (m_chunk > 0) ? whole(st, tb) : 0.f;
      const float gam_open = (m_chunk > 0) ? whole(st, L) : 0.f;
      const float* gst = sm.gq[st];
      const float* qst = gst + L * L;
      const float aa = gst[2 * L * L + ta], ab = gst[2 * L * L + tb];
      // fp16 pool: the open entry's norm bound restarts from its exact norm
      if constexpr (kBig) {
        if (m_chunk > 0 && lane == 0) sm.bnb[m_chunk - 1] = sqrtf(fmaxf(gam_open, 0.f));
      } else {
        if (kF16 && m_chunk > 0) entry_set(e_nb, m_chunk - 1, sqrtf(fmaxf(gam_open, 0.f)));
      }
      // exclusive prefix sums of x_t and a_t over the chunk: with the table Q,
      // sum_{js <= u < t} (2 beta_u + a_u) = 2 (X(t) - X(js)) [open state] + 2 Q[js][t] + A(t) - A(js)
      float xpa, xpb, apa, apb;
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
        xpa = __shfl_up_sync(0xffffffffu, ix, 1);
        apa = __shfl_up_sync(0xffffffffu, ia, 1);
        if (lane == 0) xpa = apa = 0.f;
        xpb = xpa + xa;
        apb = apa + aa;
      }
      const float invDf = 1.f / Df;
      float Ia = 0.f, Ib = 0.f;  // final scores of tokens ta, tb
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
        bool fa = false, fb = false;
        if (ta >= cur && ta < Lc) {
          const float ba = (pre ? xa : 0.f) + gst[js * GS + ta];
          const float ea = (pre ? 2.f * (xpa - xpj) : 0.f) + 2.f * qst[js * GS + ta] + (apa - apj);
          Ia = info_score_fast(aa, ba, g0 + ea, invDf, a.sp);
          fa = (Ia >= a.sp.tau_f);
        }
        if (tb >= cur && tb < Lc) {
          const float bb = (pre ? xb : 0.f) + gst[js * GS + tb];
          const float eb = (pre ? 2.f * (xpb - xpj) : 0.f) + 2.f * qst[js * GS + tb] + (apb - apj);
          Ib = info_score_fast(ab, bb, g0 + eb, invDf, a.sp);
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
      sm.bnd[ta] = (int)((bmask >> ta) & 1);
      sm.bnd[tb] = (int)((bmask >> tb) & 1);
      // score sum of the tokens [u0, u1) of the chunk (fp32 warp sum; Ibar itself is fp64)
      auto run_sum = [&](int u0, int u1) -> float {
        const float v = ((ta >= u0 && ta < u1) ? Ia : 0.f) + ((tb >= u0 && tb < u1) ? Ib : 0.f);
        return warp_sum(v);
      };
      // fp16 pool: a run [u0, u1) grows its entry's norm bound by SA(u1) - SA(u0)
      // (the chunk's prefix sums of |v_t| |k_t| = sqrt(a_t), in its Gram block)
      const float* sa_blk = gst + kGramSA;
      if constexpr (kBig) {
        // DLA(I): entries only open and grow; a boundary into a full cache would
        // need the capacity merge this instance does not hold
        int m = m_chunk;
        int seg_u0 = 0, nops = 0, run0 = 0;
        unsigned long long pend = bmask;
        while (true) {
          const int t = pend ? (__ffsll((long long)pend) - 1) : Lc;
          pend &= pend - 1;
          if (t > run0) {  // tokens [run0, t) joined the open state (entry m - 1)
            const double part = (double)run_sum(run0, t);
            if (lane == 0) {
              const int e = m - 1;
              sm.bn[e] += t - run0;
              sm.bib[e] += part;
              sm.bdirty[e] = 1;
              sm.bnb[e] += sa_blk[t] - sa_blk[run0];
            }
          }
          run0 = t + 1;
          if (t >= Lc) break;
          if (m >= C) {  // no room: the call fails its device check (results undefined)
            if (lane == 0) {
              atomicCAS(a.status, 0, 6);
              sm.mlog[t] = -1;
              sm.bnd[t] = 0;  // the trace stays a valid replay: no entry was opened
            }
            run0 = t;  // the token stays in the open state
            continue;
          }
          if (m > 0) {
            if (lane == 0) {
              sm.ops[nops][0] = OP_CLOSE;
              sm.ops[nops][1] = sm.slot[m - 1];
              sm.ops[nops][2] = seg_u0;
              sm.ops[nops][3] = t;
            }
            ++nops;
          }
          const float it = __shfl_sync(0xffffffffu, (t & 1) ? Ib : Ia, t >> 1);
          if (lane == 0) {
            sm.slot[m] = m;  // slots 0 .. m - 1 are the live ones: slot m is free
            sm.bn[m] = 1;
            sm.bib[m] = (double)it;
            sm.bpid[m] = -1;
            sm.bdirty[m] = 1;
            sm.bnb[m] = sa_blk[t + 1] - sa_blk[t];
            sm.mlog[t] = -1;
          }
          m += 1;
          seg_u0 = t;
        }
        __syncwarp();
        if (lane == 0) {
          sm.m = m;
          sm.nops = nops;
          sm.js = seg_u0;
          sm.open_slot = (m > 0) ? sm.slot[m - 1] : 0;
        }
      } else {
        int m = m_chunk;
        int seg_u0 = 0, nops = 0, run0 = 0;
        unsigned long long pend = bmask;
        while (true) {
          const int t = pend ? (__ffsll((long long)pend) - 1) : Lc;
          pend &= pend - 1;
          if (t > run0) {  // tokens [run0, t) joined the open state (entry m - 1)
            const double part = (double)run_sum(run0, t);
            // |S + sum v k^T|_F <= |S|_F + sum |v| |k|, and |v_t| |k_t| = sqrt(a_t)
            float grow = 0.f;
            if constexpr (kF16) grow = sa_blk[t] - sa_blk[run0];
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
              sm.ops[nops][0] = OP_CLOSE;
              sm.ops[nops][1] = sl;
              sm.ops[nops][2] = seg_u0;
              sm.ops[nops][3] = t;
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
              sm.ops[nops][0] = OP_MERGE;
              sm.ops[nops][1] = dst;
              sm.ops[nops][2] = srcs;
              sm.ops[nops][3] = 0;
            }
            ++nops;
            // entry j absorbs j + 1; entries j + 2 .. m - 1 move down by one
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
          if constexpr (kF16) entry_set(e_nb, m, sa_blk[t + 1] - sa_blk[t]);
          entry_set(e_slot, m, phys_new);
          entry_set(e_n, m, 1);
          entry_set(e_ib, m, (double)it);
          entry_set(e_pid, m, -1);
          entry_set(e_dirty, m, 1);
          if (lane == 0) sm.mlog[t] = j;
          m += 1;
          seg_u0 = t;
        }
        const int oslot = (m > 0) ? entry_get(e_slot, m - 1) : 0;
        if (lane == 0) {
          sm.m = m;
          sm.nops = nops;
          sm.js = seg_u0;
          sm.open_slot = oslot;
        }
      }
    }
    __syncthreads();
    if (tid == 0) sm.pend = 0;  // every warp is past the deferred copies (read before this barrier)
    // ------------------------------------------------ 6. state updates (this CTA's rows)
    {
      const int nops = sm.nops;
      for (int op = 0; op < nops; ++op) {
        if (sm.ops[op][0] == OP_CLOSE) {
          const int phys = sm.ops[op][1];
          build(st, sm.ops[op][2], sm.ops[op][3]);
          float* dst = states + (long long)phys * D * D;
#pragma unroll
          for (int n = 0; n < NT8; ++n) {
            const int k = k0 + 8 * n + 2 * tg;
            *reinterpret_cast<float2*>(dst + (jg0 + g) * D + k) = make_float2(acc[n][0], acc[n][1]);
            *reinterpret_cast<float2*>(dst + (jg0 + g + 8) * D + k) = make_float2(acc[n][2], acc[n][3]);
            acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;
          }
        } else {
          add_state_g<D, R>(srows(sm.ops[op][1]), srows(sm.ops[op][2]));
        }
        __syncthreads();
      }
      build(st, sm.js, Lc);  // the chunk's tail joins the open state
    }
    if (lead && tid < Lc) {
      bnd_out[t0 + tid] = (uint8_t)sm.bnd[tid];
      mlog_out[t0 + tid] = sm.mlog[tid];
    }
    publish_state(st ^ 1);  // operand of the next chunk's x GEMM and |S_open|^2
    __syncthreads();
    // ------------------------------------------------ 7. read-out snapshot
    const bool interval_end = ((c + 1) % a.snap_chunks) == 0;
    const int snap_idx = (c + 1) / a.snap_chunks;
    const long long lrow = (long long)bh * a.snap_stride + a.snap_base + snap_idx;
    if (pool && interval_end && (snap_idx < a.nsnap || a.snap_at_end)) {
      if (kBig && warp == 0) {  // the same over the shared-memory metadata
        const int m = sm.m;
        int nj = 0;
        for (int base = 0; base < m; base += 32) {
          const int i = base + lane;
          const bool need = (i < m) && (sm.bdirty[i] || sm.bpid[i] < 0);
          const unsigned bal = __ballot_sync(0xffffffffu, need);
          if (need) {
            const int rank_ = nj + __popc(bal & ((1u << lane) - 1u));
            int p = sm.pool_next + rank_;
            if (p >= a.pool_cap) {  // cannot happen with a correctly sized workspace
              atomicExch(a.status, 6);
              p = a.pool_cap - 1;
            }
            sm.bpid[i] = p;
            sm.bdirty[i] = 0;
            sm.snap_src[rank_][0] = p;
            sm.snap_src[rank_][1] = (i == m - 1) ? -1 : sm.slot[i];
            const float sc = f16_scale(sm.bnb[i]);
            sm.snap_scale[rank_] = sc;
            if (lead) a.pool_scale[(long long)bh * a.pool_cap + p] = sc;
          }
          nj += __popc(bal);
          if (lead && i < m) a.snap_ids[lrow * C + i] = sm.bpid[i];
        }
        __syncwarp();
        if (lane == 0) {
          sm.pool_next += nj;
          sm.nsnapjobs = nj;
          if (lead) a.snap_m0[lrow] = m;
        }
      } else if (warp == 0) {  // entries whose state changed get a fresh pool entry
        const int m = sm.m;
        int nj = 0;
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int i = lane + 32 * r;
          const bool need = (i < m) && (e_dirty[r] || e_pid[r] < 0);
          const unsigned bal = __ballot_sync(0xffffffffu, need);
          if (need) {
            const int rank_ = nj + __popc(bal & ((1u << lane) - 1u));
            int p = sm.pool_next + rank_;
            if (p >= a.pool_cap) {  // cannot happen with a correctly sized workspace
              atomicExch(a.status, 6);
              p = a.pool_cap - 1;
            }
            e_pid[r] = p;
            e_dirty[r] = 0;
            sm.snap_src[rank_][0] = p;
            sm.snap_src[rank_][1] = (i == m - 1) ? -1 : e_slot[r];
            if constexpr (kF16) {
              const float sc = f16_scale(e_nb[r]);
              sm.snap_scale[rank_] = sc;
              if (lead) a.pool_scale[(long long)bh * a.pool_cap + p] = sc;
            }
          }
          nj += __popc(bal);
          if (lead && i < m) a.snap_ids[lrow * C + i] = e_pid[r];
        }
        __syncwarp();
        if (lane == 0) {
          sm.pool_next += nj;
          sm.nsnapjobs = nj;
          if (lead) a.snap_m0[lrow] = m;
        }
      }
      if constexpr (sizeof(Tpool) == 2) {
        if (tid == 0) sm.pend = sm.nsnapjobs;  // copied during the next chunk's passes (or at round end)
        __syncthreads();
        // interval snap_base + snap_idx - 1 is complete: its trace is written and its
        // starting snapshot was copied during its first chunk (a concurrent read-out
        // waits for this); released at the start of the next chunk's copies, or by
        // the final release below
        if (a.progress && tid == NT - 32) rel_pending = a.snap_base + snap_idx;
      } else {  // fp32 pool (d = 64): copied now, the open state straight from the accumulators
        __syncthreads();
        for (int jj = 0; jj < sm.nsnapjobs; ++jj) {
          const int p = sm.snap_src[jj][0], srcslot = sm.snap_src[jj][1];
          Tpool* entry = pool + (long long)p * kEntry;
          if (srcslot < 0) {
#pragma unroll
            for (int n = 0; n < NT8; ++n) {
              const int k = k0 + 8 * n + 2 * tg;
              put_pair(entry, D, jg0 + g, k, acc[n][0], acc[n][1]);
              put_pair(entry, D, jg0 + g + 8, k, acc[n][2], acc[n][3]);
            }
          } else {
            copy_state_g<D, R>(entry + (long long)rbase * D, srows(srcslot));
          }
        }
        __syncthreads();
      }
    }
  }
  if constexpr (sizeof(Tpool) == 2) {  // the last interval's copies, if no chunk followed
    if (sm.pend > 0) {
      snapshot_copies(sm.pend, tid, NT);
      __syncthreads();
    }
  }
  if (a.progress) {  // every interval of this launch is complete
    __syncthreads();
    if (tid == 0) st_release_gpu(a.progress + 2 * bh + rank, a.snap_base + a.nsnap);
  }
  // ---------------------------------------------------------------- round end
  if constexpr (kRagged)
    if (lead) fill_padding_trace(bnd_out, mlog_out, t_end_r, a.t_end, tid, NT);
#undef DLA_T_END
  {
    const int m = sm.m;
    if (m > 0) {
      float* dst = states + (long long)sm.open_slot * D * D;
#pragma unroll
      for (int n = 0; n < NT8; ++n) {
        const int k = k0 + 8 * n + 2 * tg;
        *reinterpret_cast<float2*>(dst + (jg0 + g) * D + k) = make_float2(acc[n][0], acc[n][1]);
        *reinterpret_cast<float2*>(dst + (jg0 + g + 8) * D + k) = make_float2(acc[n][2], acc[n][3]);
      }
    }
    if (kBig && lead && warp == 0) {
      for (int i = lane; i < C; i += 32) {
        a.slot[(long long)bh * C + i] = (i < m) ? sm.slot[i] : i;
        a.n[(long long)bh * C + i] = (i < m) ? sm.bn[i] : 0;
        a.ibar[(long long)bh * C + i] = (i < m) ? sm.bib[i] : 0.0;
        if (pool && a.pstate && i < m) a.pstate[a.B * a.H + (long long)bh * C + i] = sm.bpid[i];
        if (pool && i < m) a.nbound[(long long)bh * C + i] = sm.bnb[i];
      }
      if (lane == 0) {
        a.m[bh] = m;
        if (pool && a.pstate) a.pstate[bh] = sm.pool_next;
      }
    } else if (lead && warp == 0) {
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const int i = lane + 32 * r;
        if (i < C) {
          a.slot[(long long)bh * C + i] = e_slot[r];
          a.n[(long long)bh * C + i] = (i < m) ? e_n[r] : 0;
          a.ibar[(long long)bh * C + i] = (i < m) ? e_ib[r] : 0.0;
        }
        if (pool && a.pstate && i < m) a.pstate[a.B * a.H + (long long)bh * C + i] = e_pid[r];
        if (kF16 && pool && i < m) a.nbound[(long long)bh * C + i] = e_nb[r];
      }
      if (lane == 0) {
        a.m[bh] = m;
        if (pool && a.pstate) a.pstate[bh] = sm.pool_next;  // counters for a following round that continues this pool
      }
    }
  }
  if constexpr (CL > 1) cluster_sync();  // the partner may still read this CTA's shared memory
}

// K0: Gram pre-pass.  One CTA per (64-token chunk, stream): the suffix table
// gs[j][t] = sum_{j <= s < t} (k_t.k_s)(v_t.v_s), its running sums
// Q[j][t] = sum_{j <= u < t} gs[j][u] and a_t of every chunk, so that the
// sequential scan reads beta_t and the segment's sum of 2 beta_u + a_u for any
// segment start with two loads.  Depends on k and v only, so it runs on the
// other SMs ahead of the scan.
template <int D>
struct GramSmem {
  static constexpr int RP = D + 8;
  __nv_bfloat16 k[L * RP];     // the chunk's k rows (then the next chunk's, once G is formed)
  __nv_bfloat16 v[L * RP];
  float G[L * (L + 1)];        // G[t][s], then in place gs[s][t]
  float Q[L * (L + 1)];        // Q[j][t]
  float a[L];
};

// K0: each CTA walks the chunks of one block of one stream in order, one k, v
// buffer (three CTAs per SM): the next chunk's rows are in flight (cp.async)
// while this chunk's tables are scanned and written.  With `ready` set, the
// count of the block's chunks written is published (release) after each of its
// first four chunks, every fourth and its last, for a scan that runs
// concurrently and reads the blocks through the async proxy.
template <int D>
__global__ void __launch_bounds__(NT) gram_kernel(GramArgs a) {
  constexpr int RP = D + 8;
  constexpr int V16 = D / 8;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  GramSmem<D>& sm = *reinterpret_cast<GramSmem<D>*>(smem_raw);
  const int bh = blockIdx.x, blk = blockIdx.y;
  const int b = bh / a.H, h = bh % a.H;
  // this block's chunks: chunk0 + blk + i * nblk, i < n_mine (interleaved, so
  // that the early chunks of every stream, which a concurrent scan needs first,
  // come out together)
  if (blk >= a.count) return;
  const int n_mine = (a.count - blk + a.nblk - 1) / a.nblk;
  auto chunk_of = [&](int i) { return a.chunk0 + blk + i * a.nblk; };
  const int row_stride = a.H * D;
  const long long tok0 = row_tok0(a.row_start, b, a.T);
  const __nv_bfloat16* k0 = reinterpret_cast<const __nv_bfloat16*>(a.k) + (tok0 * a.H + h) * D;
  const __nv_bfloat16* v0 = reinterpret_cast<const __nv_bfloat16*>(a.v) + (tok0 * a.H + h) * D;
  const int row_len = a.seq_lens ? max(0, min(a.T, __ldg(a.seq_lens + b))) : a.T;
  auto load = [&](int c) {  // rows past the row's end are zero-filled, not read
    const int t0 = c * L, valid = min(L, row_len - t0);
    const __nv_bfloat16* kz = reinterpret_cast<const __nv_bfloat16*>(a.k);  // address of a zero-filled row
    const __nv_bfloat16* vz = reinterpret_cast<const __nv_bfloat16*>(a.v);
    for (int e = threadIdx.x; e < L * V16; e += NT) {
      const int r = e / V16, cc = (e % V16) * 8;
      const bool in = r < valid;
      const long long off = (long long)(t0 + r) * row_stride + cc;
      const int nbytes = in ? 16 : 0;
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(su32(sm.k + r * RP + cc)),
                   "l"(in ? k0 + off : kz), "r"(nbytes) : "memory");
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(su32(sm.v + r * RP + cc)),
                   "l"(in ? v0 + off : vz), "r"(nbytes) : "memory");
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  load(chunk_of(0));
  for (int i = 0; i < n_mine; ++i) {
    const int c = chunk_of(i);
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    gram_tile_lower<D>(sm.k, sm.v, sm.G, sm.a);
    __syncthreads();
    if (i + 1 < n_mine) load(chunk_of(i + 1));  // k, v are free: in flight during the scans below
    suffix_rows_ilp(sm.G);  // G[t][j] = gs[j][t]
    __syncthreads();
    prefix_rows_ilp(sm.G, 1, L + 1, sm.Q, L + 1);  // Q[j][t] = sum_{u < t} gs[j][u]
    __syncthreads();
    // out: gs[j][t], Q[j][t] (four consecutive t per thread), a[t]
    float* out = a.out + ((long long)bh * a.nchunks + c) * kGramStride;
    for (int e = threadIdx.x; e < L * L / 4; e += NT) {
      const int j = e / (L / 4), t = (e % (L / 4)) * 4;
      const float4 g4 = make_float4(sm.G[t * (L + 1) + j], sm.G[(t + 1) * (L + 1) + j], sm.G[(t + 2) * (L + 1) + j],
                                    sm.G[(t + 3) * (L + 1) + j]);
      const float* qr = sm.Q + j * (L + 1) + t;
      *reinterpret_cast<float4*>(out + j * L + t) = g4;
      *reinterpret_cast<float4*>(out + L * L + j * L + t) = make_float4(qr[0], qr[1], qr[2], qr[3]);
    }
    if (threadIdx.x < L / 4)
      *reinterpret_cast<float4*>(out + 2 * L * L + 4 * threadIdx.x) = *reinterpret_cast<const float4*>(sm.a + 4 * threadIdx.x);
    if (threadIdx.x >= NT - 32) norm_prefix_warp(sm.a, out + kGramSA, threadIdx.x & 31);
    // published after the first chunk, then every fourth and after the last
    // (the scan reads the blocks by bulk copy: async proxy)
    const bool publish = a.ready && (i < 4 || (i & 3) == 3 || i + 1 == n_mine);
    if (publish) asm volatile("fence.proxy.async.global;" ::: "memory");
    __syncthreads();  // the block is written; G, Q, a are reused by the next chunk
    if (publish && threadIdx.x == 0) {
      __threadfence();
      st_release_gpu(a.ready + (long long)bh * a.nblk + blk, i + 1);
    }
  }
}

// Cross Gram block of two chunks with mma.sync: Gout[t][s] = (k_t.k'_s)(v_t.v'_s)
// for every t of this chunk (K, V) and s of the previous one (Kp, Vp), row
// stride L + 1.  All 8 warps; warp w takes the 16-token band w % 4 and the 32
// columns w / 4.
template <int D>
__device__ __forceinline__ void gram_cross(const __nv_bfloat16* Ks, const __nv_bfloat16* Vs, const __nv_bfloat16* Kp,
                                           const __nv_bfloat16* Vp, float* Gout) {
  constexpr int RP = D + 8;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> 2, tg = lane & 3, q = lane >> 3, r8 = lane & 7;
  const int mt = warp & 3, sb = 32 * (warp >> 2);
  float kk4[4][4], vv4[4][4];
#pragma unroll
  for (int n = 0; n < 4; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) kk4[n][e] = vv4[n][e] = 0.f;
#pragma unroll 2
  for (int kk = 0; kk < D; kk += 16) {
    uint32_t ak[4], av[4];
    ldsm4(ak, Ks + (16 * mt + (q & 1) * 8 + r8) * RP + kk + (q >> 1) * 8);
    ldsm4(av, Vs + (16 * mt + (q & 1) * 8 + r8) * RP + kk + (q >> 1) * 8);
#pragma unroll
    for (int np = 0; np < 2; ++np) {
      uint32_t bk[4], bv[4];
      ldsm4(bk, Kp + (sb + 16 * np + (q >> 1) * 8 + r8) * RP + kk + (q & 1) * 8);
      ldsm4(bv, Vp + (sb + 16 * np + (q >> 1) * 8 + r8) * RP + kk + (q & 1) * 8);
      mma16816(kk4[2 * np], ak, bk[0], bk[1]);
      mma16816(kk4[2 * np + 1], ak, bk[2], bk[3]);
      mma16816(vv4[2 * np], av, bv[0], bv[1]);
      mma16816(vv4[2 * np + 1], av, bv[2], bv[3]);
    }
  }
#pragma unroll
  for (int n = 0; n < 4; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int t = 16 * mt + g + 8 * (e >> 1);
      const int s2 = sb + 8 * n + 2 * tg + (e & 1);
      Gout[t * (L + 1) + s2] = kk4[n][e] * vv4[n][e];
    }
}

// K0 for the tensor-core scan: the same tables as gram_kernel in the packed
// layout (kGramBlockTc floats per chunk) plus the cross table cs of the chunk
// against the previous one.  Each CTA walks its block's chunks like
// gram_kernel, loading the chunk and the one before it.
template <int D>
struct GramTcSmem {
  static constexpr int RP = D + 8;
  __nv_bfloat16 k[L * RP], v[L * RP];    // this chunk
  __nv_bfloat16 kp[L * RP], vp[L * RP];  // the previous chunk (zero rows before the sequence)
  float G[L * (L + 1)];                  // G[t][s], then in place gs[s][t]
  float X[L * (L + 1)];                  // cross G'[t][s], then in place cs[s][t]
  float a[L];
  // Q[j][t] lives in the previous chunk's k and v rows (adjacent), free once the
  // Gram blocks are formed
  __device__ float* Q() { return reinterpret_cast<float*>(kp); }
  static_assert(2 * sizeof(__nv_bfloat16) * L * RP >= sizeof(float) * L * (L + 1), "Q fits the k, v rows");
};

template <int D>
__global__ void __launch_bounds__(NT) gram_tc_kernel(GramArgs a) {
  constexpr int RP = D + 8;
  constexpr int V16 = D / 8;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  GramTcSmem<D>& sm = *reinterpret_cast<GramTcSmem<D>*>(smem_raw);
  const int bh = blockIdx.x, blk = blockIdx.y;
  const int b = bh / a.H, h = bh % a.H;
  if (blk >= a.count) return;
  const int n_mine = (a.count - blk + a.nblk - 1) / a.nblk;
  auto chunk_of = [&](int i) { return a.chunk0 + blk + i * a.nblk; };
  const int row_stride = a.H * D;
  const __nv_bfloat16* k0 = reinterpret_cast<const __nv_bfloat16*>(a.k) + ((long long)b * a.T * a.H + h) * D;
  const __nv_bfloat16* v0 = reinterpret_cast<const __nv_bfloat16*>(a.v) + ((long long)b * a.T * a.H + h) * D;
  // rows of chunk c (c >= 0) into (dk, dv); rows outside [0, T) zero-filled
  auto load = [&](int c, __nv_bfloat16* dk, __nv_bfloat16* dv) {
    const int t0 = c * L;
    for (int e = threadIdx.x; e < L * V16; e += NT) {
      const int r = e / V16, cc = (e % V16) * 8;
      const int t = t0 + r;
      const bool ok = (c >= 0) && (t < a.T);
      const long long off = (long long)(ok ? t : 0) * row_stride + cc;
      const int nbytes = ok ? 16 : 0;
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(su32(dk + r * RP + cc)), "l"(k0 + off),
                   "r"(nbytes) : "memory");
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(su32(dv + r * RP + cc)), "l"(v0 + off),
                   "r"(nbytes) : "memory");
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  for (int i = 0; i < n_mine; ++i) {
    const int c = chunk_of(i);
    __syncthreads();  // the buffers of the previous chunk are no longer read
    load(c, sm.k, sm.v);
    load(c - 1, sm.kp, sm.vp);
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    gram_tile_lower<D>(sm.k, sm.v, sm.G, sm.a);
    gram_cross<D>(sm.k, sm.v, sm.kp, sm.vp, sm.X);
    __syncthreads();
    suffix_rows_ilp(sm.G);  // G[t][j] = gs[j][t]
    suffix_rows_ilp(sm.X);  // X[t][j] = cs[j][t]
    __syncthreads();
    float* const Qs = sm.Q();
    prefix_rows_ilp(sm.G, 1, L + 1, Qs, L + 1);  // Q[j][t] = sum_{u < t} gs[j][u], t < L
    __syncthreads();
    float* out = a.out + ((long long)bh * a.nchunks + c) * kGramStride;
    float* ogs = out;
    float* oq = out + kPackTri;
    float* oa = out + 2 * kPackTri;
    float* ocs = oa + L;
    // packed rows j (a warp each), t in [j, 64]; Q[j][64] = Q[j][63] + gs[j][63]
    {
      const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
      for (int j = warp; j < L; j += NW) {
        const int base = pack_row(j);
        for (int t = j + lane; t <= L; t += 32) {
          ogs[base + t - j] = (t < L) ? sm.G[t * (L + 1) + j] : 0.f;
          oq[base + t - j] = (t < L) ? Qs[j * (L + 1) + t] : Qs[j * (L + 1) + L - 1] + sm.G[(L - 1) * (L + 1) + j];
        }
      }
    }
    if (threadIdx.x < L) oa[threadIdx.x] = sm.a[threadIdx.x];
    for (int e = threadIdx.x; e < L * L / 4; e += NT) {
      const int j = e / (L / 4), t = (e % (L / 4)) * 4;
      *reinterpret_cast<float4*>(ocs + j * L + t) = make_float4(sm.X[t * (L + 1) + j], sm.X[(t + 1) * (L + 1) + j],
                                                                sm.X[(t + 2) * (L + 1) + j], sm.X[(t + 3) * (L + 1) + j]);
    }
    const bool publish = a.ready && (i < 4 || (i & 3) == 3 || i + 1 == n_mine);
    if (publish) asm volatile("fence.proxy.async.global;" ::: "memory");
    __syncthreads();
    if (publish && threadIdx.x == 0) {
      __threadfence();
      st_release_gpu(a.ready + (long long)bh * a.nblk + blk, i + 1);
    }
  }
}

template <int D>
static cudaError_t launch_gram_t(const GramArgs& a, cudaStream_t s) {
  const size_t smem = a.packed ? sizeof(GramTcSmem<D>) : sizeof(GramSmem<D>);
  auto kern = a.packed ? gram_tc_kernel<D> : gram_kernel<D>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  if (a.nblk < 1 || a.nblk > kMaxGramBlk || (long long)a.nblk * a.per_blk < a.count) return cudaErrorInvalidValue;
  dim3 grid(a.B * a.H, a.nblk);  // streams fastest: every stream's first block is scheduled first
  kern<<<grid, NT, smem, s>>>(a);
  return cudaGetLastError();
}

void gram_blocks(int BH, int count, int slots, int* nblk, int* per_blk) {
  int n = slots / BH;  // one wave
  if (n > kMaxGramBlk) n = kMaxGramBlk;
  if (n > count) n = count;
  if (n < 1) n = 1;
  *per_blk = (count + n - 1) / n;
  *nblk = (count + *per_blk - 1) / *per_blk;
}

cudaError_t launch_gram(const GramArgs& a, int d, cudaStream_t s) {
  return d == 128 ? launch_gram_t<128>(a, s) : launch_gram_t<64>(a, s);
}

template <int D, typename Tpool, int CL, bool kRagged, int CAPB = kMaxC>
static cudaError_t launch_scan_mma_r(const ScanArgs& a, cudaStream_t s) {
  const size_t smem = sizeof(MmaSmem<D, CL, CAPB>);
  auto kern = scan_mma_kernel<D, Tpool, CL, kRagged, CAPB>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.B * a.H * CL);
  cfg.blockDim = dim3(NT);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = CL;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = CL > 1 ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, a);
}
template <int D, typename Tpool, int CL>
static cudaError_t launch_scan_mma_t(const ScanArgs& a, cudaStream_t s) {
  return a.seq_lens ? launch_scan_mma_r<D, Tpool, CL, true>(a, s) : launch_scan_mma_r<D, Tpool, CL, false>(a, s);
}

int scan_mma_ctas_per_stream(int BH, int d) {
  int dev = 0, sms = 0;
  if (d != 128 || cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 1;
  return (2LL * BH <= sms) ? 2 : 1;
}
// CTA pairs when two CTAs per stream still fit on the device in one wave.
static bool use_pairs(const ScanArgs& a) { return scan_mma_ctas_per_stream(a.B * a.H, 128) == 2; }

static int resident_streams_query(int BH, int d) {
  int dev = 0, sms = 0, per_sm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 0;
  if (scan_mma_ctas_per_stream(BH, d) == 2) {
    auto kern = scan_mma_kernel<128, __half, 2>;
    const size_t smem = sizeof(MmaSmem<128, 2>);
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess) return 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * BH);
    cfg.blockDim = dim3(NT);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&clusters, kern, &cfg) != cudaSuccess) return 0;
    return clusters;
  }
  if (d == 128) {
    auto kern = scan_mma_kernel<128, __half, 1>;
    const size_t smem = sizeof(MmaSmem<128, 1>);
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, NT, smem) != cudaSuccess)
      return 0;
  } else {
    auto kern = scan_mma_kernel<64, __half, 1>;
    const size_t smem = sizeof(MmaSmem<64, 1>);
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, NT, smem) != cudaSuccess)
      return 0;
  }
  return per_sm * sms;
}
int scan_mma_resident_streams(int BH, int d) {  // cached per device and kernel variant
  static std::atomic<int> cache[64][3];
  static std::atomic<bool> init{false};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  const int var = (d != 128) ? 2 : scan_mma_ctas_per_stream(BH, d) - 1;
  if (!init.load()) {
    std::lock_guard<std::mutex> g(mu);
    if (!init.load()) {
      for (auto& row : cache)
        for (auto& c : row) c.store(-1);
      init.store(true);
    }
  }
  int v = cache[dev][var].load();
  if (v < 0) {
    v = resident_streams_query(BH, d);
    cache[dev][var].store(v);
  }
  return v;
}

__global__ void gate_kernel(const int32_t* started, int n, int32_t* status) {
  const long long t0 = clock64();
  long long lim = -1;
  while (ld_acquire_gpu(started) < n)
    if (*(volatile int32_t*)status != 0 || sm100::wait_expired(t0, lim, status)) {
      atomicCAS(status, 0, 5);  // a failure reported elsewhere keeps its code
      return;
    }
}
cudaError_t preload_scan_kernels() {
  cudaFuncAttributes fa;
  cudaError_t e;
  if ((e = cudaFuncGetAttributes(&fa, scan_mma_kernel<128, __half, 2>)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, scan_mma_kernel<128, __half, 1>)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, scan_mma_kernel<128, __half, 2, true>)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, scan_mma_kernel<128, __half, 1, true>)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, scan_mma_kernel<128, __half, 2, false, kMaxCBig>)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, scan_mma_kernel<128, __half, 1, false, kMaxCBig>)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, gram_kernel<128>)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, gram_tc_kernel<128>)) != cudaSuccess) return e;
  return cudaFuncGetAttributes(&fa, gate_kernel);
}
cudaError_t launch_gate(const int32_t* started, int n, int32_t* status, cudaStream_t s) {
  gate_kernel<<<1, 1, 0, s>>>(started, n, status);
  return cudaGetLastError();
}

cudaError_t launch_scan_mma(const ScanArgs& a, int d, bool pool_f16, cudaStream_t s) {
  if (a.C > kMaxC) {  // DLA(I): bf16 inputs, d = 128, whole rows
    if (d != 128 || !pool_f16 || a.C > kMaxCBig || a.seq_lens) return cudaErrorInvalidValue;
    return use_pairs(a) ? launch_scan_mma_r<128, __half, 2, false, kMaxCBig>(a, s)
                        : launch_scan_mma_r<128, __half, 1, false, kMaxCBig>(a, s);
  }
  if (d == 128) {
    if (use_pairs(a))
      return pool_f16 ? launch_scan_mma_t<128, __half, 2>(a, s) : launch_scan_mma_t<128, float, 2>(a, s);
    return pool_f16 ? launch_scan_mma_t<128, __half, 1>(a, s) : launch_scan_mma_t<128, float, 1>(a, s);
  }
  return pool_f16 ? launch_scan_mma_t<64, __half, 1>(a, s) : launch_scan_mma_t<64, float, 1>(a, s);
}

}  // namespace dla

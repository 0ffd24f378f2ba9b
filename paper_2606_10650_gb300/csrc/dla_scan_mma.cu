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
#include "dla_common.cuh"
#include "dla_mma.cuh"

namespace dla {

namespace {

constexpr int NT = 256;
constexpr int NW = NT / 32;
constexpr int L = kScanL;
constexpr int GS = L + 4;          // row of a suffix table in shared memory
constexpr int kGramBlock = L * L + L;  // floats per chunk of the Gram pre-pass output

enum : int { OP_CLOSE = 0, OP_MERGE = 1 };

template <int D, int CL>
struct MmaSmem {
  static constexpr int RP = D + 8;  // padded bf16 row: 8 rows of a ldmatrix hit 8 bank groups
  static constexpr int GS = L + 4;  // suffix-table row (16-byte aligned for cp.async)
  __nv_bfloat16 kv[2][2][L * RP];   // [stage][k / v][t][RP]
  __nv_bfloat16 S2[2][D / CL * RP]; // this CTA's rows of the open state as bf16 hi / lo, [j][RP]
  float gs[2][L * GS];              // [stage] suffix table sg[j][t] = sum_{j <= s < t} (k_t.k_s)(v_t.v_s)
  float as[2][L];                   // [stage] a_t = |k_t|^2 |v_t|^2
  float G[L * (L + 1)];             // Gram rows, when the scan forms them itself
  float red[NW][L];
  float xs[2][L + 4];               // [chunk parity] this CTA's part of x_t (t < L) and of |S_open|^2 (at L)
  float gred[NW];
  float wsum[4];
  float Itok[L];
  double ibar[kMaxC];
  int n[kMaxC];
  int slot[kMaxC];
  int pid[kMaxC];
  int dirty[kMaxC];
  int bnd[L];
  int mlog[L];
  int ops[3 * L + 4][4];
  int snap_src[kMaxC][2];
  int first_fire[2];
  int nops, nsnapjobs;
  int m, cur, js, seg_pre, pool_next;
};

// Keep the bf16 halves of a packed pair whose token index lies in [u0, u1).
__device__ __forceinline__ uint32_t mask_pair(uint32_t v, int t, int u0, int u1) {
  const uint32_t lo = (t >= u0 && t < u1) ? 0x0000FFFFu : 0u;
  const uint32_t hi = (t + 1 >= u0 && t + 1 < u1) ? 0xFFFF0000u : 0u;
  return v & (lo | hi);
}

template <int D>
__device__ __forceinline__ void prefetch_kv(__nv_bfloat16* dk, __nv_bfloat16* dv, const __nv_bfloat16* ks,
                                            const __nv_bfloat16* vs, int row_stride, int valid, float* dgs,
                                            float* das, const float* gsrc) {
  constexpr int RP = D + 8;
  constexpr int V16 = D / 8;
  for (int e = threadIdx.x; e < L * V16; e += NT) {
    const int r = e / V16, c = (e % V16) * 8;
    const int nbytes = (r < valid) ? 16 : 0;
    const __nv_bfloat16* sk = (r < valid) ? ks + (long long)r * row_stride + c : ks;
    const __nv_bfloat16* sv = (r < valid) ? vs + (long long)r * row_stride + c : vs;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(su32(dk + r * RP + c)), "l"(sk), "r"(nbytes)
                 : "memory");
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(su32(dv + r * RP + c)), "l"(sv), "r"(nbytes)
                 : "memory");
  }
  if (gsrc) {  // suffix table [j][t] (64 x 64) and a_t of this chunk from the Gram pre-pass
    for (int e = threadIdx.x; e < L * (L / 4) + L / 4; e += NT) {
      const bool is_a = e >= L * (L / 4);
      const int r = is_a ? 0 : e / (L / 4), c4 = is_a ? (e - L * (L / 4)) * 4 : (e % (L / 4)) * 4;
      float* dst = is_a ? das + c4 : dgs + r * GS + c4;
      const float* src = is_a ? gsrc + L * L + c4 : gsrc + r * L + c4;
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(su32(dst)), "l"(src) : "memory");
    }
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

// State copies (NR rows of a D x D state) move NR*D/4/NT float4 per thread;
// loads are issued in batches of four before their stores so that a copy costs
// a few memory latencies, not one per element (the compiler cannot reorder a
// load past a possibly aliasing store).  A bf16 pool entry is hi rows [D][D]
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
template <int D, int NR = D>
__device__ __forceinline__ void copy_state_g(__nv_bfloat16* dst, const float* src) {
  constexpr int PER = NR * D / 4 / NT;
  for (int base = 0; base < PER; base += 4) {
    float4 v[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) v[i] = load4(src + ((base + i) * NT + threadIdx.x) * 4);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int e = ((base + i) * NT + threadIdx.x) * 4;
      const float4 x = v[i];
      const __nv_bfloat162 h01 = __floats2bfloat162_rn(x.x, x.y), h23 = __floats2bfloat162_rn(x.z, x.w);
      const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
      store4(dst + e, make_float4(f01.x, f01.y, f23.x, f23.y));
      store4(dst + D * D + e, make_float4(x.x - f01.x, x.y - f01.y, x.z - f23.x, x.w - f23.y));
    }
  }
}
// dst += src over one D x D state, batched like copy_state_g.
template <int D, int NR = D>
__device__ __forceinline__ void add_state_g(float* dst, const float* src) {
  constexpr int PER = NR * D / 4 / NT;
  for (int base = 0; base < PER; base += 4) {
    float4 x[4], y[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int e = ((base + i) * NT + threadIdx.x) * 4;
      x[i] = load4(dst + e);
      y[i] = load4(src + e);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
      store4(dst + ((base + i) * NT + threadIdx.x) * 4,
             make_float4(x[i].x + y[i].x, x[i].y + y[i].y, x[i].z + y[i].z, x[i].w + y[i].w));
  }
}

// One pair of adjacent state elements (k, k+1 of row j) into an fp32 pool entry.
__device__ __forceinline__ void put_pair(float* entry, int D, int j, int k, float v0, float v1) {
  *reinterpret_cast<float2*>(entry + j * D + k) = make_float2(v0, v1);
}

template <typename Tpool>
constexpr int parts_of() { return sizeof(Tpool) == 2 ? 2 : 1; }

}  // namespace

// One stream per CTA (CL = 1) or per CTA pair (CL = 2, a thread-block
// cluster): with a pair, each CTA owns d/2 rows of the open state (and of every
// state it copies or adds), forms its part of x_t and |S_open|^2, and the two
// parts meet through distributed shared memory once per chunk; both CTAs then
// take the same decisions from the same sums (x = part of rank 0 + part of
// rank 1 in both), and rank 0 writes the trace, the lists and the metadata.
template <int D, typename Tpool, int CL>
__global__ void __launch_bounds__(NT, 1) scan_mma_kernel(ScanArgs a) {
  constexpr int RP = D + 8;
  constexpr int R = D / CL;           // state rows of this CTA
  constexpr int MT = R / 16;          // 16-row bands of those rows
  constexpr int WPM = NW / MT;        // warps per band
  constexpr int KC = D / WPM;         // state columns per warp
  constexpr int NT8 = KC / 8;         // n8 tiles per warp in the state build
  constexpr int NJ8 = R / 8 / NW;     // n8 tiles per warp in the x GEMM
  static_assert(NJ8 == 1 || NJ8 == 2, "x GEMM tiling");
  extern __shared__ __align__(16) unsigned char smem_raw[];
  MmaSmem<D, CL>& sm = *reinterpret_cast<MmaSmem<D, CL>*>(smem_raw);

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = lane >> 2, tg = lane & 3;
  const int rank = (CL > 1) ? (int)cluster_rank() : 0;
  const bool lead = (rank == 0);      // writes what both CTAs of a pair hold
  const int bh = blockIdx.x / CL;
  const int b = bh / a.H, h = bh % a.H;
  const int C = a.C;
  const float Df = (float)(D * D);
  const __nv_bfloat16* kbase = reinterpret_cast<const __nv_bfloat16*>(a.k) + ((long long)b * a.T * a.H + h) * D;
  const __nv_bfloat16* vbase = reinterpret_cast<const __nv_bfloat16*>(a.v) + ((long long)b * a.T * a.H + h) * D;
  const int row_stride = a.H * D;
  const int rbase = rank * R;         // first state row of this CTA
  float* states = a.states + (long long)bh * C * D * D;
  constexpr long long kEntry = (long long)parts_of<Tpool>() * D * D;
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
    int m0 = a.m[bh];
    if (m0 < 0 || m0 > C) {
      atomicExch(a.status, 6);
      m0 = 0;
    }
    sm.m = m0;
    sm.pool_next = 0;
  }
  __syncthreads();
  for (int i = tid; i < C; i += NT) {
    int sl = a.slot[(long long)bh * C + i];
    if (sl < 0 || sl >= C) {
      atomicExch(a.status, 6);
      sl = i;
    }
    sm.slot[i] = sl;
    sm.n[i] = a.n[(long long)bh * C + i];
    sm.ibar[i] = a.ibar[(long long)bh * C + i];
    sm.pid[i] = -1;
    sm.dirty[i] = 0;
  }
  __syncthreads();
  const int m_start = sm.m;
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
      for (int i = tid; i < m_start; i += NT) sm.pid[i] = a.pstate[a.B * a.H + (long long)bh * C + i];
    } else {  // snapshot 0: every live entry at the start of the round
      for (int i = 0; i < m_start && i < a.pool_cap; ++i)
        copy_state_g<D, R>(pool + (long long)i * kEntry + (long long)rbase * D, srows(sm.slot[i]));
      if (tid < m_start) sm.pid[tid] = tid;
      if (tid == 0) sm.pool_next = m_start;
      if (lead) {
        if (tid == 0) a.snap_m0[lst] = m_start;
        for (int i = tid; i < m_start; i += NT) a.snap_ids[lst * C + i] = i;
      }
    }
  }

  // this CTA's rows of the open state -> bf16 hi / lo operand, and its part of
  // |S_open|^2 into xs[buf][L]
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
      sm.xs[buf][L] = gs;
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
  // x_t or |S_open|^2 of the whole state: the CTAs' parts added in rank order
  auto whole = [&](const float* p) -> float {
    if constexpr (CL == 1) {
      return *p;
    } else {
      return dsmem_ld(p, 0) + dsmem_ld(p, 1);
    }
  };

  publish_state(0);
  __syncthreads();

  const int ntok = a.t_end - a.t_begin;
  const int nchunks = (ntok + L - 1) / L;
  const long long gchunk0 = (long long)bh * a.gram_chunks + a.t_begin / L;  // Gram block of the round's first chunk
  prefetch_kv<D>(sm.kv[0][0], sm.kv[0][1], kbase + (long long)a.t_begin * row_stride,
                 vbase + (long long)a.t_begin * row_stride, row_stride, min(L, ntok), sm.gs[0], sm.as[0],
                 a.gram ? a.gram + gchunk0 * kGramBlock : nullptr);
  for (int c = 0; c < nchunks; ++c) {
    const int t0 = a.t_begin + c * L;
    const int Lc = min(L, a.t_end - t0);
    const int st = c & 1;
    // ------------------------------------------------ 1. k, v of this chunk; prefetch the next
    if (c + 1 < nchunks) {
      const int t1 = t0 + L;
      prefetch_kv<D>(sm.kv[st ^ 1][0], sm.kv[st ^ 1][1], kbase + (long long)t1 * row_stride,
                     vbase + (long long)t1 * row_stride, row_stride, min(L, a.t_end - t1), sm.gs[st ^ 1],
                     sm.as[st ^ 1], a.gram ? a.gram + (gchunk0 + c + 1) * kGramBlock : nullptr);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    if (tid < L) {
      sm.bnd[tid] = 0;
      sm.mlog[tid] = -1;
      sm.Itok[tid] = 0.f;
    }
    __syncthreads();
    const int m_chunk = sm.m;
    const __nv_bfloat16* Ks = sm.kv[st][0];
    const __nv_bfloat16* Vs = sm.kv[st][1];
    const int q = lane >> 3, r8 = lane & 7;
    // ------------------------------------------------ 2. x_t = v_t^T S_open k_t (this CTA's rows)
    if (m_chunk > 0) {
      float X[4][NJ8][4];
#pragma unroll
      for (int mt = 0; mt < 4; ++mt)
#pragma unroll
        for (int nj = 0; nj < NJ8; ++nj)
#pragma unroll
          for (int e = 0; e < 4; ++e) X[mt][nj][e] = 0.f;
      const int jb = warp * 8 * NJ8;  // local rows of this warp
      for (int kk = 0; kk < D; kk += 16) {
        uint32_t bh_[4], bl_[4];
        if constexpr (NJ8 == 2) {
          ldsm4(bh_, &sm.S2[0][(jb + (q >> 1) * 8 + r8) * RP + kk + (q & 1) * 8]);
          ldsm4(bl_, &sm.S2[1][(jb + (q >> 1) * 8 + r8) * RP + kk + (q & 1) * 8]);
        } else {
          ldsm2(bh_, &sm.S2[0][(jb + r8) * RP + kk + (q & 1) * 8]);
          ldsm2(bl_, &sm.S2[1][(jb + r8) * RP + kk + (q & 1) * 8]);
        }
#pragma unroll
        for (int mt = 0; mt < 4; ++mt) {
          uint32_t af[4];
          ldsm4(af, Ks + (16 * mt + (q & 1) * 8 + r8) * RP + kk + (q >> 1) * 8);
#pragma unroll
          for (int nj = 0; nj < NJ8; ++nj) {
            mma16816(X[mt][nj], af, bh_[2 * nj], bh_[2 * nj + 1]);
            mma16816(X[mt][nj], af, bl_[2 * nj], bl_[2 * nj + 1]);
          }
        }
      }
      // x partial over this warp's j rows: sum_j v_t[j] X[t][j]
#pragma unroll
      for (int mt = 0; mt < 4; ++mt) {
        float p0 = 0.f, p1 = 0.f;  // rows g and g + 8 of the tile
#pragma unroll
        for (int nj = 0; nj < NJ8; ++nj) {
          const int j = rbase + jb + 8 * nj + 2 * tg;
          const int ta = 16 * mt + g, tb8 = ta + 8;
          const float2 va = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(Vs + ta * RP + j));
          const float2 vb = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(Vs + tb8 * RP + j));
          p0 += X[mt][nj][0] * va.x + X[mt][nj][1] * va.y;
          p1 += X[mt][nj][2] * vb.x + X[mt][nj][3] * vb.y;
        }
        p0 += __shfl_xor_sync(0xffffffffu, p0, 1);
        p0 += __shfl_xor_sync(0xffffffffu, p0, 2);
        p1 += __shfl_xor_sync(0xffffffffu, p1, 1);
        p1 += __shfl_xor_sync(0xffffffffu, p1, 2);
        if (tg == 0) {
          sm.red[warp][16 * mt + g] = p0;
          sm.red[warp][16 * mt + g + 8] = p1;
        }
      }
    }
    // ------------------------------------------------ 3. Gram suffix table and a_t
    // Normally prefetched from the Gram pre-pass; formed here when the call has
    // no room for the pre-pass output (scan-only calls).
    if (!a.gram) {
      gram_tile<D>(Ks, Vs, sm.G, sm.as[st]);
      __syncthreads();
      suffix_rows(sm.G);
      __syncthreads();
      for (int e = tid; e < L * L; e += NT) {  // transpose to the [j][t] layout the passes read
        const int t = e % L, j = e / L;
        sm.gs[st][j * GS + t] = sm.G[t * (L + 1) + j];
      }
    }
    __syncthreads();
    if (tid < L) {  // this CTA's part of x_t
      float x = 0.f;
      if (m_chunk > 0)
#pragma unroll
        for (int w8 = 0; w8 < NW; ++w8) x += sm.red[w8][tid];
      sm.xs[st][tid] = x;
    }
    if constexpr (CL > 1) {
      cluster_sync();
    } else {
      __syncthreads();
    }
    // ------------------------------------------------ 4. boundary passes (warps 0-1, token t = tid)
    // Each pass scores every undecided token as if the open segment ran to it,
    // takes the first that fires, and restarts the segment there.  Only the
    // two warps that own the tokens take part (64-thread named barrier).
    if (warp < 2) {
      const int t = tid;
      int cur = 0, js = 0, pre = (m_chunk > 0) ? 1 : 0;
      if (m_chunk == 0) {  // the very first token of an empty cache opens state 0
        if (t == 0) {
          sm.bnd[0] = 1;
          sm.Itok[0] = 0.f;
        }
        cur = 1;
      }
      const float xt = (m_chunk > 0) ? whole(&sm.xs[st][t]) : 0.f;
      const float gam_open = (m_chunk > 0) ? whole(&sm.xs[st][L]) : 0.f;
      const float at = sm.as[st][t];
      const float* gst = sm.gs[st];
      while (cur < Lc) {
        float beta = 0.f, w = 0.f;
        if (t >= js && t < Lc) {
          beta = (pre ? xt : 0.f) + gst[js * GS + t];
          w = 2.f * beta + at;
        }
        float inc = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const float up = __shfl_up_sync(0xffffffffu, inc, o);
          if (lane >= o) inc += up;
        }
        if (lane == 31) sm.wsum[warp] = inc;
        asm volatile("bar.sync 1, 64;" ::: "memory");
        const float excl = inc - w + (warp == 1 ? sm.wsum[0] : 0.f);
        bool fire = false;
        if (t >= cur && t < Lc) {
          const float gam = (pre ? gam_open : 0.f) + excl;
          const float I = info_score(at, beta, gam, Df, a.sp);
          sm.Itok[t] = I;
          fire = ((double)I >= a.sp.tau);
        }
        const unsigned bal = __ballot_sync(0xffffffffu, fire);
        if (lane == 0) sm.first_fire[warp] = bal ? (warp * 32 + __ffs(bal) - 1) : L;
        asm volatile("bar.sync 1, 64;" ::: "memory");
        const int ts = min(sm.first_fire[0], sm.first_fire[1]);
        if (ts >= Lc) break;
        if (t == ts) sm.bnd[ts] = 1;
        js = ts;
        pre = 0;
        cur = ts + 1;
      }
    }
    __syncthreads();
    // ------------------------------------------------ 5. replay decisions (warp 0)
    if (warp == 0) {
      int m = sm.m;
      int seg_u0 = 0;
      int nops = 0;
      int run0 = 0;
      // boundary tokens of the chunk as a bit mask (Lc <= 64)
      const unsigned lo = __ballot_sync(0xffffffffu, sm.bnd[lane] != 0);
      const unsigned hi = __ballot_sync(0xffffffffu, sm.bnd[lane + 32] != 0);
      unsigned long long pend = ((unsigned long long)hi << 32) | lo;
      while (true) {
        const int t = pend ? (__ffsll((long long)pend) - 1) : Lc;
        pend &= pend - 1;
        if (t > run0) {  // tokens [run0, t) joined the open state
          float part = 0.f;
          for (int u = run0 + lane; u < t; u += 32) part += sm.Itok[u];
          part = warp_sum(part);
          if (lane == 0) {
            sm.n[m - 1] += t - run0;
            sm.ibar[m - 1] += (double)part;
            sm.dirty[m - 1] = 1;
          }
          __syncwarp();
        }
        run0 = t + 1;
        if (t >= Lc) break;
        if (m > 0 && lane == 0) {
          sm.ops[nops][0] = OP_CLOSE;
          sm.ops[nops][1] = sm.slot[m - 1];
          sm.ops[nops][2] = seg_u0;
          sm.ops[nops][3] = t;
        }
        if (m > 0) ++nops;
        int j = -1, phys_new = m;
        __syncwarp();
        if (m == C) {
          j = pair_argmin_warp(sm.n, sm.ibar, m);
          const int dst = sm.slot[j], src = sm.slot[j + 1];
          __syncwarp();
          if (lane == 0) {
            sm.ops[nops][0] = OP_MERGE;
            sm.ops[nops][1] = dst;
            sm.ops[nops][2] = src;
            sm.ops[nops][3] = 0;
            sm.n[j] += sm.n[j + 1];
            sm.ibar[j] += sm.ibar[j + 1];
            sm.dirty[j] = 1;
            sm.pid[j] = -1;
          }
          ++nops;
          __syncwarp();
          for (int base = j + 1; base < m - 1; base += 32) {
            const int i = base + lane;
            int nv = 0, sv = 0, pv = 0, dv = 0;
            double iv = 0.0;
            if (i < m - 1) {
              nv = sm.n[i + 1]; sv = sm.slot[i + 1]; pv = sm.pid[i + 1]; dv = sm.dirty[i + 1];
              iv = sm.ibar[i + 1];
            }
            __syncwarp();
            if (i < m - 1) {
              sm.n[i] = nv; sm.slot[i] = sv; sm.pid[i] = pv; sm.dirty[i] = dv; sm.ibar[i] = iv;
            }
            __syncwarp();
          }
          phys_new = src;
          m -= 1;
        }
        if (lane == 0) {
          sm.slot[m] = phys_new;
          sm.n[m] = 1;
          sm.ibar[m] = (double)sm.Itok[t];
          sm.pid[m] = -1;
          sm.dirty[m] = 1;
          sm.mlog[t] = j;
        }
        __syncwarp();
        m += 1;
        seg_u0 = t;
      }
      if (lane == 0) {
        sm.m = m;
        sm.nops = nops;
        sm.js = seg_u0;
      }
    }
    __syncthreads();
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
      if (warp == 0) {  // entries whose state changed get a fresh pool entry
        const int m = sm.m;
        int nj = 0;
        for (int base = 0; base < m; base += 32) {
          const int i = base + lane;
          const bool need = (i < m) && (sm.dirty[i] || sm.pid[i] < 0);
          const unsigned bal = __ballot_sync(0xffffffffu, need);
          if (need) {
            const int rank_ = nj + __popc(bal & ((1u << lane) - 1u));
            int p = sm.pool_next + rank_;
            if (p >= a.pool_cap) {  // cannot happen with a correctly sized workspace
              atomicExch(a.status, 6);
              p = a.pool_cap - 1;
            }
            sm.pid[i] = p;
            sm.dirty[i] = 0;
            sm.snap_src[rank_][0] = p;
            sm.snap_src[rank_][1] = (i == m - 1) ? -1 : sm.slot[i];
          }
          nj += __popc(bal);
        }
        __syncwarp();
        if (lane == 0) {
          sm.pool_next += nj;
          sm.nsnapjobs = nj;
          if (lead) a.snap_m0[lrow] = m;
        }
      }
      __syncthreads();
      const int m = sm.m;
      if (lead)
        for (int i = tid; i < m; i += NT) a.snap_ids[lrow * C + i] = sm.pid[i];
      for (int jj = 0; jj < sm.nsnapjobs; ++jj) {
        const int p = sm.snap_src[jj][0], srcslot = sm.snap_src[jj][1];
        Tpool* entry = pool + (long long)p * kEntry;
        if (srcslot < 0) {  // the open state
          if constexpr (sizeof(Tpool) == 2) {
            // bf16 hi / lo are already staged in shared memory: coalesced 16-byte copies
            for (int e = tid; e < 2 * R * (D / 8); e += NT) {
              const int part = e / (R * (D / 8)), rem = e % (R * (D / 8));
              const int j = rem / (D / 8), k8 = (rem % (D / 8)) * 8;
              *reinterpret_cast<uint4*>(entry + part * D * D + (rbase + j) * D + k8) =
                  *reinterpret_cast<const uint4*>(&sm.S2[part][j * RP + k8]);
            }
          } else {  // fp32 pool: straight from the accumulators
#pragma unroll
            for (int n = 0; n < NT8; ++n) {
              const int k = k0 + 8 * n + 2 * tg;
              put_pair(entry, D, jg0 + g, k, acc[n][0], acc[n][1]);
              put_pair(entry, D, jg0 + g + 8, k, acc[n][2], acc[n][3]);
            }
          }
        } else {
          copy_state_g<D, R>(entry + (long long)rbase * D, srows(srcslot));
        }
      }
      __syncthreads();
    }
  }
  // ---------------------------------------------------------------- round end
  {
    const int m = sm.m;
    if (m > 0) {
      float* dst = states + (long long)sm.slot[m - 1] * D * D;
#pragma unroll
      for (int n = 0; n < NT8; ++n) {
        const int k = k0 + 8 * n + 2 * tg;
        *reinterpret_cast<float2*>(dst + (jg0 + g) * D + k) = make_float2(acc[n][0], acc[n][1]);
        *reinterpret_cast<float2*>(dst + (jg0 + g + 8) * D + k) = make_float2(acc[n][2], acc[n][3]);
      }
    }
    if (lead) {
      for (int i = tid; i < C; i += NT) {
        a.slot[(long long)bh * C + i] = sm.slot[i];
        a.n[(long long)bh * C + i] = (i < m) ? sm.n[i] : 0;
        a.ibar[(long long)bh * C + i] = (i < m) ? sm.ibar[i] : 0.0;
      }
      if (tid == 0) a.m[bh] = m;
      if (pool && a.pstate) {  // counters for a following round that continues this pool
        if (tid == 0) a.pstate[bh] = sm.pool_next;
        for (int i = tid; i < m; i += NT) a.pstate[a.B * a.H + (long long)bh * C + i] = sm.pid[i];
      }
    }
  }
  if constexpr (CL > 1) cluster_sync();  // the partner may still read this CTA's shared memory
}

// K0: Gram pre-pass.  One CTA per (64-token chunk, stream): the suffix table
// sg[j][t] = sum_{j <= s < t} (k_t.k_s)(v_t.v_s) and a_t of every chunk, so the
// sequential scan reads beta_t of any segment start with one load.  Depends on
// k and v only, so it runs on every SM ahead of the scan.
template <int D>
struct GramSmem {
  static constexpr int RP = D + 8;
  __nv_bfloat16 k[L * RP];
  __nv_bfloat16 v[L * RP];
  float G[L * (L + 1)];
  float a[L];
};

template <int D>
__global__ void __launch_bounds__(NT) gram_kernel(GramArgs a) {
  constexpr int RP = D + 8;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  GramSmem<D>& sm = *reinterpret_cast<GramSmem<D>*>(smem_raw);
  const int c = a.chunk0 + blockIdx.x, bh = blockIdx.y;
  const int b = bh / a.H, h = bh % a.H;
  const int t0 = c * L;
  const int valid = min(L, a.T - t0);
  const int row_stride = a.H * D;
  const __nv_bfloat16* ks =
      reinterpret_cast<const __nv_bfloat16*>(a.k) + (((long long)b * a.T + t0) * a.H + h) * D;
  const __nv_bfloat16* vs =
      reinterpret_cast<const __nv_bfloat16*>(a.v) + (((long long)b * a.T + t0) * a.H + h) * D;
  constexpr int V16 = D / 8;
  for (int e = threadIdx.x; e < L * V16; e += NT) {
    const int r = e / V16, cc = (e % V16) * 8;
    uint4 kv = make_uint4(0, 0, 0, 0), vv = make_uint4(0, 0, 0, 0);
    if (r < valid) {
      kv = *reinterpret_cast<const uint4*>(ks + (long long)r * row_stride + cc);
      vv = *reinterpret_cast<const uint4*>(vs + (long long)r * row_stride + cc);
    }
    *reinterpret_cast<uint4*>(sm.k + r * RP + cc) = kv;
    *reinterpret_cast<uint4*>(sm.v + r * RP + cc) = vv;
  }
  __syncthreads();
  gram_tile<D>(sm.k, sm.v, sm.G, sm.a);
  __syncthreads();
  suffix_rows(sm.G);
  __syncthreads();
  float* out = a.out + ((long long)bh * a.nchunks + c) * kGramBlock;
  for (int e = threadIdx.x; e < L * L; e += NT) {
    const int t = e % L, j = e / L;
    out[j * L + t] = sm.G[t * (L + 1) + j];
  }
  if (threadIdx.x < L) out[L * L + threadIdx.x] = sm.a[threadIdx.x];
}

template <int D>
static cudaError_t launch_gram_t(const GramArgs& a, cudaStream_t s) {
  const size_t smem = sizeof(GramSmem<D>);
  auto kern = gram_kernel<D>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid(a.count, a.B * a.H);
  kern<<<grid, NT, smem, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_gram(const GramArgs& a, int d, cudaStream_t s) {
  return d == 128 ? launch_gram_t<128>(a, s) : launch_gram_t<64>(a, s);
}

template <int D, typename Tpool, int CL>
static cudaError_t launch_scan_mma_t(const ScanArgs& a, cudaStream_t s) {
  const size_t smem = sizeof(MmaSmem<D, CL>);
  auto kern = scan_mma_kernel<D, Tpool, CL>;
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

// CTA pairs when two CTAs per stream still fit on the device in one wave.
static bool use_pairs(const ScanArgs& a) {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return false;
  return 2LL * a.B * a.H <= sms;
}

cudaError_t launch_scan_mma(const ScanArgs& a, int d, bool pool_bf16, cudaStream_t s) {
  if (d == 128) {
    if (use_pairs(a))
      return pool_bf16 ? launch_scan_mma_t<128, __nv_bfloat16, 2>(a, s) : launch_scan_mma_t<128, float, 2>(a, s);
    return pool_bf16 ? launch_scan_mma_t<128, __nv_bfloat16, 1>(a, s) : launch_scan_mma_t<128, float, 1>(a, s);
  }
  return pool_bf16 ? launch_scan_mma_t<64, __nv_bfloat16, 1>(a, s) : launch_scan_mma_t<64, float, 1>(a, s);
}

}  // namespace dla

// dla_backward.cu -- K4, gradients of the read-out of Eq. (capacity_bounded_output)
// with the boundary and merge decisions of a forward pass held fixed.
//
// The decisions are piecewise constant in k and v, so their derivative is zero
// almost everywhere; with them fixed every state is a sum of token states over
// a contiguous token range (Sec. 2 recurrent form; a merge of Algorithm 2 joins
// two adjacent ranges) and the read-out is a weighted causal linear attention:
//   o_t = sum_{s <= t} W[t, s] (q_t . k_s) v_s,  W[t, s] = lambda_{t, slot_t(s)},
// slot_t(s) being the logical slot (0 = oldest) of the state holding token s
// after token t.  For a loss with dL/do = G:
//   dQ = ((G V^T) o W) K        dK = ((G V^T) o W)^T Q        dV = ((Q K^T) o W)^T G
//   dlambda_{t, i} = sum_{s <= t, slot_t(s) = i} (q_t . k_s)(g_t . v_s).
//
// Three kernels, bf16 q, k, v, fp32 G and gradients, d in {64, 128}:
//   slots_kernel   one warp per stream replays the trace (boundary flags and
//                  merge indices) on token ranges: after each boundary event e
//                  the first tokens of the live states, firsts[e][0 .. C)
//                  (padded with INT_MAX), and per token the event count evt[t],
//                  so that slot_t(s) = #{i : firsts[evt[t]][i] <= s} - 1.
//   dq_kernel      one CTA per (64-token block of t, stream): over the key
//                  blocks s <= t, P = Q K^T and dP = G V^T on mma.sync, W from
//                  the slot lists, dQ += (dP o W) K, and dlambda accumulated per
//                  (t, slot) in shared memory (the block owns its rows).
//   dkv_kernel     one CTA per (64-token block of s, stream): over the query
//                  blocks t >= s, warps 0-3 form P^T and dV += (P o W)^T G,
//                  warps 4-7 form dP^T and dK += (dP o W)^T Q.
// G and the weighted products P o W, dP o W are fp32 values; as tensor-core
// operands each is split into bf16 hi + lo (x = hi + lo to ~2^-17), and the
// products keep the hi*hi, hi*lo and lo*hi terms, so the gradients carry about
// 2^-16 relative rounding instead of bf16's 2^-9.  The work is quadratic in T
// per stream (every pair s <= t), like the dense form it evaluates.
#include <climits>

#include "dla_common.cuh"
#include "dla_mma.cuh"

namespace dla {

namespace {

constexpr int BT = 64;        // tokens per block (rows of t or s)
constexpr int NTB = 128;      // dq_kernel threads (4 warps x 16 rows)
constexpr int NTK = 256;      // dkv_kernel threads (8 warps)

// ---------------------------------------------------------------- slot lists
__global__ void __launch_bounds__(32) slots_kernel(BackwardArgs a) {
  const int bh = blockIdx.x, lane = threadIdx.x;
  const int C = a.C;
  const uint8_t* bnd = a.boundary + (long long)bh * a.T;
  const int32_t* mlog = a.merge_log + (long long)bh * a.T;
  int32_t* evt = a.evt + (long long)bh * a.T;
  int32_t* lists = a.firsts + (long long)bh * (a.T + 1) * kMaxC;
  // firsts of the live states: entry i in lane i % 32, register i / 32
  int f0 = INT_MAX, f1 = INT_MAX;
  int m = 0, e = 0;
  auto write_list = [&](int ev) {
    lists[(long long)ev * kMaxC + lane] = f0;
    lists[(long long)ev * kMaxC + 32 + lane] = f1;
  };
  write_list(0);
  for (int t0 = 0; t0 < a.T; t0 += 32) {
    const int t = t0 + lane;
    const bool bt = (t < a.T) && (bnd[t] != 0 || (t == 0));
    unsigned bal = __ballot_sync(0xffffffffu, bt);
    const int ev_before = e;
    while (bal) {
      const int l = __ffs(bal) - 1;
      bal &= bal - 1;
      const int tt = t0 + l;
      int j = (m > 0) ? mlog[tt] : -1;
      if (j >= 0 && j + 1 >= m) {  // a merge index outside the live pairs: inconsistent trace
        if (lane == 0) atomicCAS(a.status, 0, 6);
        j = -1;
      }
      if (j >= 0) {  // states j and j + 1 become one: entry j + 1 leaves, the later ones move down
        const int n0 = __shfl_down_sync(0xffffffffu, f0, 1), n1 = __shfl_down_sync(0xffffffffu, f1, 1);
        const int w0 = __shfl_sync(0xffffffffu, f1, 0);  // entry 32 moves to entry 31
        const int s0 = (lane == 31) ? w0 : n0, s1 = (lane == 31) ? INT_MAX : n1;
        if (lane >= j + 1) f0 = s0;
        if (32 + lane >= j + 1) f1 = s1;
        m -= 1;
      }
      if (m >= C) {  // a boundary into a full cache without a merge: inconsistent trace
        if (lane == 0) atomicCAS(a.status, 0, 6);
      } else {
        if (m == lane) f0 = tt;
        if (m == 32 + lane) f1 = tt;
        m += 1;
      }
      e += 1;
      write_list(e);
    }
    // events at or before each token of this group
    if (t < a.T) {
      const unsigned mine = __ballot_sync(0xffffffffu, bt) & (0xffffffffu >> (31 - lane));
      evt[t] = ev_before + __popc(mine);
    } else {
      __ballot_sync(0xffffffffu, bt);
    }
  }
}

// Logical slot of token s in a sorted first-token list of kMaxC entries
// (padded with INT_MAX): the last entry <= s.  f[0] = 0 <= s always (the
// oldest state starts at the first token), so the search starts there.
__device__ __forceinline__ int slot_of(const int* f, int s) {
  int i = 0;
#pragma unroll
  for (int step = kMaxC / 2; step >= 1; step >>= 1)
    if (f[i + step] <= s) i += step;
  return i;
}

// Slot of token s0 and whether tokens s0 .. s0 + 63 all share it (no later
// entry starts inside the block): then one lookup serves a whole tile row.
__device__ __forceinline__ int block_slot(const int* f, int s0, bool& uniform) {
  const int sl = slot_of(f, s0);
  uniform = (sl + 1 >= kMaxC) || (f[sl + 1] > s0 + BT - 1);
  return sl;
}

// ---------------------------------------------------------------- shared tiles
template <int D>
struct BwdTiles {
  static constexpr int RP = D + 8;  // padded row (bf16 elements): ldmatrix without bank conflicts
};

// Loads rows [t0, t0 + n) of one stream's [T, H, D] bf16 tensor (row stride
// H * D) into a [BT][RP] tile; rows >= n are zero.  All threads of the CTA.
template <int D>
__device__ __forceinline__ void load_bf16_rows(__nv_bfloat16* dst, const __nv_bfloat16* src, int row_stride, int n,
                                               int tid, int nthreads) {
  constexpr int RP = BwdTiles<D>::RP, V = D / 8;
  for (int e = tid; e < BT * V; e += nthreads) {
    const int r = e / V, c = (e % V) * 8;
    uint4 val = make_uint4(0, 0, 0, 0);
    if (r < n) val = __ldg(reinterpret_cast<const uint4*>(src + (long long)r * row_stride + c));
    *reinterpret_cast<uint4*>(dst + r * RP + c) = val;
  }
}
// fp32 rows split into bf16 hi and lo tiles.
template <int D>
__device__ __forceinline__ void load_split_rows(__nv_bfloat16* hi, __nv_bfloat16* lo, const float* src, int row_stride,
                                                int n, int tid, int nthreads) {
  constexpr int RP = BwdTiles<D>::RP, V = D / 4;
  for (int e = tid; e < BT * V; e += nthreads) {
    const int r = e / V, c = (e % V) * 4;
    float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
    if (r < n) x = __ldg(reinterpret_cast<const float4*>(src + (long long)r * row_stride + c));
    const __nv_bfloat162 h01 = __floats2bfloat162_rn(x.x, x.y), h23 = __floats2bfloat162_rn(x.z, x.w);
    const float2 g01 = __bfloat1622float2(h01), g23 = __bfloat1622float2(h23);
    const __nv_bfloat162 l01 = __floats2bfloat162_rn(x.x - g01.x, x.y - g01.y);
    const __nv_bfloat162 l23 = __floats2bfloat162_rn(x.z - g23.x, x.w - g23.y);
    *reinterpret_cast<__nv_bfloat162*>(hi + r * RP + c) = h01;
    *reinterpret_cast<__nv_bfloat162*>(hi + r * RP + c + 2) = h23;
    *reinterpret_cast<__nv_bfloat162*>(lo + r * RP + c) = l01;
    *reinterpret_cast<__nv_bfloat162*>(lo + r * RP + c + 2) = l23;
  }
}
// lambda rows (C per token, fp32; ones when lam is null) and the first-token
// lists of the tokens' events, for rows [t0, t0 + n) of one stream.
__device__ __forceinline__ void load_weights(float* lam_s, int* firsts_s, const BackwardArgs& a, int b, int h, int bh,
                                             int t0, int n, int tid, int nthreads) {
  const int C = a.C;
  for (int e = tid; e < BT * kMaxC; e += nthreads) {
    const int r = e / kMaxC, x = e % kMaxC;
    const int t = t0 + r;
    float w = 0.f;
    int f = INT_MAX;
    if (r < n) {
      if (x < C) w = a.lam ? __ldg(a.lam + (((long long)b * a.T + t) * a.H + h) * C + x) : 1.f;
      const int ev = __ldg(a.evt + (long long)bh * a.T + t);
      f = __ldg(a.firsts + ((long long)bh * (a.T + 1) + ev) * kMaxC + x);
    }
    lam_s[r * kMaxC + x] = w;
    firsts_s[r * kMaxC + x] = f;
  }
}

// Two fp32 accumulator tiles (m16n8: columns 8p .. 8p + 15 of a warp's 16 rows)
// as the bf16 hi and lo A fragments of one k16 step.
__device__ __forceinline__ void acc_to_a(const float* c0, const float* c1, uint32_t* ahi, uint32_t* alo) {
  const float v[8] = {c0[0], c0[1], c0[2], c0[3], c1[0], c1[1], c1[2], c1[3]};
  uint32_t h[4], l[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const __nv_bfloat162 hh = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
    const float2 f = __bfloat1622float2(hh);
    const __nv_bfloat162 ll = __floats2bfloat162_rn(v[2 * i] - f.x, v[2 * i + 1] - f.y);
    h[i] = *reinterpret_cast<const uint32_t*>(&hh);
    l[i] = *reinterpret_cast<const uint32_t*>(&ll);
  }
  // a0 = (row g, k 2tg..) = c0[0..1]; a1 = (row g + 8) = c0[2..3]; a2 = (row g, k 8 + 2tg..) = c1[0..1]; a3 = c1[2..3]
  ahi[0] = h[0]; ahi[1] = h[1]; ahi[2] = h[2]; ahi[3] = h[3];
  alo[0] = l[0]; alo[1] = l[1]; alo[2] = l[2]; alo[3] = l[3];
}

// Lane address of an A fragment (16 rows x 16 k) at (row0, k0) of a [.][RP] tile.
template <int RP>
__device__ __forceinline__ const __nv_bfloat16* a_addr(const __nv_bfloat16* tile, int row0, int k0, int lane) {
  const int mi = lane >> 3, r = lane & 7;
  return tile + (row0 + r + 8 * (mi & 1)) * RP + k0 + 8 * (mi >> 1);
}
// Lane address of two B fragments (n8 tiles n0 and n0 + 8, k 16) from a tile
// stored [n][k] (ldmatrix without .trans).
template <int RP>
__device__ __forceinline__ const __nv_bfloat16* bnk_addr(const __nv_bfloat16* tile, int n0, int k0, int lane) {
  const int mi = lane >> 3, r = lane & 7;
  return tile + (n0 + r + 8 * (mi >> 1)) * RP + k0 + 8 * (mi & 1);
}
// The same from a tile stored [k][n] (ldmatrix .trans).
template <int RP>
__device__ __forceinline__ const __nv_bfloat16* bkn_addr(const __nv_bfloat16* tile, int n0, int k0, int lane) {
  const int mi = lane >> 3, r = lane & 7;
  return tile + (k0 + r + 8 * (mi & 1)) * RP + n0 + 8 * (mi >> 1);
}

template <int D>
struct DqSmem {
  static constexpr int RP = D + 8;
  __nv_bfloat16 Q[BT * RP], Ghi[BT * RP], Glo[BT * RP], K[BT * RP], V[BT * RP];
  float lam[BT * kMaxC];
  int firsts[BT * kMaxC];
  float dlam[BT * kMaxC];
};

// dQ and dlambda of one 64-token block of t of one stream.
template <int D>
__global__ void __launch_bounds__(NTB) dq_kernel(BackwardArgs a) {
  constexpr int RP = D + 8, NJ = D / 8;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  DqSmem<D>& sm = *reinterpret_cast<DqSmem<D>*>(smem_raw);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = lane >> 2, tg = lane & 3;
  const int nb = (a.T + BT - 1) / BT;
  const int tb = nb - 1 - blockIdx.x;  // the longest blocks (late t) first
  const int bh = blockIdx.y, b = bh / a.H, h = bh % a.H;
  const int t0 = tb * BT, nt = min(BT, a.T - t0);
  const int row_stride = a.H * D;
  const long long base = ((long long)b * a.T) * a.H + h;  // row index of token 0 of the stream
  const __nv_bfloat16* q = reinterpret_cast<const __nv_bfloat16*>(a.q) + base * D;
  const __nv_bfloat16* k = reinterpret_cast<const __nv_bfloat16*>(a.k) + base * D;
  const __nv_bfloat16* v = reinterpret_cast<const __nv_bfloat16*>(a.v) + base * D;
  const float* gsrc = a.g + base * D;

  load_bf16_rows<D>(sm.Q, q + (long long)t0 * row_stride, row_stride, nt, tid, NTB);
  load_split_rows<D>(sm.Ghi, sm.Glo, gsrc + (long long)t0 * row_stride, row_stride, nt, tid, NTB);
  load_weights(sm.lam, sm.firsts, a, b, h, bh, t0, nt, tid, NTB);
  for (int e = tid; e < BT * kMaxC; e += NTB) sm.dlam[e] = 0.f;

  const int r0 = 16 * warp;  // this warp's 16 rows of the block
  float dq[NJ][4];
#pragma unroll
  for (int j = 0; j < NJ; ++j) dq[j][0] = dq[j][1] = dq[j][2] = dq[j][3] = 0.f;

  for (int sb = 0; sb <= tb; ++sb) {
    const int s0 = sb * BT, ns = min(BT, a.T - s0);
    __syncthreads();  // the previous block's K, V are no longer read
    load_bf16_rows<D>(sm.K, k + (long long)s0 * row_stride, row_stride, ns, tid, NTB);
    load_bf16_rows<D>(sm.V, v + (long long)s0 * row_stride, row_stride, ns, tid, NTB);
    __syncthreads();
    float p[8][4], dp[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) p[i][0] = p[i][1] = p[i][2] = p[i][3] = dp[i][0] = dp[i][1] = dp[i][2] = dp[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      uint32_t aq[4], ah[4], al[4];
      ldsm4(aq, a_addr<RP>(sm.Q, r0, 16 * kk, lane));
      ldsm4(ah, a_addr<RP>(sm.Ghi, r0, 16 * kk, lane));
      ldsm4(al, a_addr<RP>(sm.Glo, r0, 16 * kk, lane));
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t bk[4], bv[4];
        ldsm4(bk, bnk_addr<RP>(sm.K, 16 * np, 16 * kk, lane));
        ldsm4(bv, bnk_addr<RP>(sm.V, 16 * np, 16 * kk, lane));
        mma16816(p[2 * np], aq, bk[0], bk[1]);
        mma16816(p[2 * np + 1], aq, bk[2], bk[3]);
        mma16816(dp[2 * np], ah, bv[0], bv[1]);
        mma16816(dp[2 * np + 1], ah, bv[2], bv[3]);
        mma16816(dp[2 * np], al, bv[0], bv[1]);
        mma16816(dp[2 * np + 1], al, bv[2], bv[3]);
      }
    }
    // W[t, s], dlambda and dP o W; per row the thread's columns rise with the
    // tile index, and so do their slots: runs of one slot are summed before
    // they are added to the block's dlambda row
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int rl = r0 + g + 8 * half, t = t0 + rl;
      const int* f = sm.firsts + rl * kMaxC;
      const float* lw = sm.lam + rl * kMaxC;
      bool uni = false;
      const int slu = (rl < nt) ? block_slot(f, s0, uni) : 0;  // the common case: one entry over the tile
      int run_slot = -1;
      float run = 0.f;
#pragma unroll
      for (int nt8 = 0; nt8 < 8; ++nt8) {
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const int s = s0 + 8 * nt8 + 2 * tg + c;
          const int idx = 2 * half + c;
          float w = 0.f;
          if (s <= t && rl < nt && s < a.T) {
            const int sl = uni ? slu : slot_of(f, s);
            w = lw[sl];
            const float pd = p[nt8][idx] * dp[nt8][idx];
            if (sl != run_slot) {
              if (run_slot >= 0) atomicAdd(&sm.dlam[rl * kMaxC + run_slot], run);
              run_slot = sl;
              run = 0.f;
            }
            run += pd;
          }
          dp[nt8][idx] *= w;
        }
      }
      if (run_slot >= 0) atomicAdd(&sm.dlam[rl * kMaxC + run_slot], run);
    }
    // dQ += (dP o W) K: k runs over the block's 64 tokens s, K as stored [s][j] is [k][n]
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) {
      uint32_t ahi[4], alo[4];
      acc_to_a(dp[2 * ks], dp[2 * ks + 1], ahi, alo);
#pragma unroll
      for (int np = 0; np < NJ / 2; ++np) {
        uint32_t bk[4];
        ldsm4t(bk, bkn_addr<RP>(sm.K, 16 * np, 16 * ks, lane));
        mma16816(dq[2 * np], ahi, bk[0], bk[1]);
        mma16816(dq[2 * np + 1], ahi, bk[2], bk[3]);
        mma16816(dq[2 * np], alo, bk[0], bk[1]);
        mma16816(dq[2 * np + 1], alo, bk[2], bk[3]);
      }
    }
  }
  // dQ rows of this block
  float* dqo = a.dq + base * D;
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    const int rl = r0 + g + 8 * half;
    if (rl < nt) {
      float* row = dqo + (long long)(t0 + rl) * row_stride;
#pragma unroll
      for (int j = 0; j < NJ; ++j)
        *reinterpret_cast<float2*>(row + 8 * j + 2 * tg) = make_float2(dq[j][2 * half], dq[j][2 * half + 1]);
    }
  }
  if (a.dlam) {
    __syncthreads();
    const int C = a.C;
    for (int e = tid; e < BT * C; e += NTB) {
      const int rl = e / C, x = e % C;
      if (rl < nt) a.dlam[((long long)b * a.T + t0 + rl) * a.H * C + (long long)h * C + x] = sm.dlam[rl * kMaxC + x];
    }
  }
}

template <int D>
struct DkvSmem {
  static constexpr int RP = D + 8;
  __nv_bfloat16 K[BT * RP], V[BT * RP], Q[BT * RP], Ghi[BT * RP], Glo[BT * RP];
  float lam[BT * kMaxC];
  int firsts[BT * kMaxC];
  int slot0[BT];   // per token t of the block: slot of token s0 after t
  int uni[BT];     // and whether every token of the s block shares it
};

// dK and dV of one 64-token block of s of one stream: warps 0-3 dV, warps 4-7 dK
// (16 rows of s each).
template <int D>
__global__ void __launch_bounds__(NTK) dkv_kernel(BackwardArgs a) {
  constexpr int RP = D + 8, NJ = D / 8;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  DkvSmem<D>& sm = *reinterpret_cast<DkvSmem<D>*>(smem_raw);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = lane >> 2, tg = lane & 3;
  const int nb = (a.T + BT - 1) / BT;
  const int sb = blockIdx.x;  // the longest blocks (early s) first
  const int bh = blockIdx.y, b = bh / a.H, h = bh % a.H;
  const int s0 = sb * BT, ns = min(BT, a.T - s0);
  const int row_stride = a.H * D;
  const long long base = ((long long)b * a.T) * a.H + h;
  const __nv_bfloat16* q = reinterpret_cast<const __nv_bfloat16*>(a.q) + base * D;
  const __nv_bfloat16* k = reinterpret_cast<const __nv_bfloat16*>(a.k) + base * D;
  const __nv_bfloat16* v = reinterpret_cast<const __nv_bfloat16*>(a.v) + base * D;
  const float* gsrc = a.g + base * D;
  const bool is_dv = warp < 4;     // warp-uniform role
  const int r0 = 16 * (warp & 3);  // this warp's 16 rows of s

  load_bf16_rows<D>(sm.K, k + (long long)s0 * row_stride, row_stride, ns, tid, NTK);
  load_bf16_rows<D>(sm.V, v + (long long)s0 * row_stride, row_stride, ns, tid, NTK);
  float acc[NJ][4];
#pragma unroll
  for (int j = 0; j < NJ; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;

  for (int tb = sb; tb < nb; ++tb) {
    const int t0 = tb * BT, nt = min(BT, a.T - t0);
    __syncthreads();  // the previous block's Q, G, weights are no longer read
    load_bf16_rows<D>(sm.Q, q + (long long)t0 * row_stride, row_stride, nt, tid, NTK);
    load_split_rows<D>(sm.Ghi, sm.Glo, gsrc + (long long)t0 * row_stride, row_stride, nt, tid, NTK);
    load_weights(sm.lam, sm.firsts, a, b, h, bh, t0, nt, tid, NTK);
    __syncthreads();
    if (tid < BT) {
      bool u = false;
      sm.slot0[tid] = (tid < nt) ? block_slot(sm.firsts + tid * kMaxC, s0, u) : 0;
      sm.uni[tid] = u;
    }
    __syncthreads();
    // X^T[s, t] (16 rows of s x 64 t): P^T = K Q^T (dV warps) or dP^T = V G^T (dK warps)
    float x[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) x[i][0] = x[i][1] = x[i][2] = x[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      uint32_t as[4];
      ldsm4(as, a_addr<RP>(is_dv ? sm.K : sm.V, r0, 16 * kk, lane));
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        if (is_dv) {
          uint32_t bq[4];
          ldsm4(bq, bnk_addr<RP>(sm.Q, 16 * np, 16 * kk, lane));
          mma16816(x[2 * np], as, bq[0], bq[1]);
          mma16816(x[2 * np + 1], as, bq[2], bq[3]);
        } else {
          uint32_t bh4[4], bl4[4];
          ldsm4(bh4, bnk_addr<RP>(sm.Ghi, 16 * np, 16 * kk, lane));
          ldsm4(bl4, bnk_addr<RP>(sm.Glo, 16 * np, 16 * kk, lane));
          mma16816(x[2 * np], as, bh4[0], bh4[1]);
          mma16816(x[2 * np + 1], as, bh4[2], bh4[3]);
          mma16816(x[2 * np], as, bl4[0], bl4[1]);
          mma16816(x[2 * np + 1], as, bl4[2], bl4[3]);
        }
      }
    }
    // weight W[t, s] (0 for t < s or past the sequence)
#pragma unroll
    for (int nt8 = 0; nt8 < 8; ++nt8) {
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const int tl = 8 * nt8 + 2 * tg + c, t = t0 + tl;
        const int* f = sm.firsts + tl * kMaxC;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          const int s = s0 + r0 + g + 8 * half;
          float w = 0.f;
          if (s <= t && tl < nt && s < a.T) w = sm.lam[tl * kMaxC + (sm.uni[tl] ? sm.slot0[tl] : slot_of(f, s))];
          x[nt8][2 * half + c] *= w;
        }
      }
    }
    // dV += (P o W)^T G  or  dK += (dP o W)^T Q: k runs over the block's 64 tokens t
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) {
      uint32_t ahi[4], alo[4];
      acc_to_a(x[2 * ks], x[2 * ks + 1], ahi, alo);
#pragma unroll
      for (int np = 0; np < NJ / 2; ++np) {
        if (is_dv) {
          uint32_t gh[4], gl[4];
          ldsm4t(gh, bkn_addr<RP>(sm.Ghi, 16 * np, 16 * ks, lane));
          ldsm4t(gl, bkn_addr<RP>(sm.Glo, 16 * np, 16 * ks, lane));
          mma16816(acc[2 * np], ahi, gh[0], gh[1]);
          mma16816(acc[2 * np + 1], ahi, gh[2], gh[3]);
          mma16816(acc[2 * np], ahi, gl[0], gl[1]);
          mma16816(acc[2 * np + 1], ahi, gl[2], gl[3]);
          mma16816(acc[2 * np], alo, gh[0], gh[1]);
          mma16816(acc[2 * np + 1], alo, gh[2], gh[3]);
        } else {
          uint32_t bq[4];
          ldsm4t(bq, bkn_addr<RP>(sm.Q, 16 * np, 16 * ks, lane));
          mma16816(acc[2 * np], ahi, bq[0], bq[1]);
          mma16816(acc[2 * np + 1], ahi, bq[2], bq[3]);
          mma16816(acc[2 * np], alo, bq[0], bq[1]);
          mma16816(acc[2 * np + 1], alo, bq[2], bq[3]);
        }
      }
    }
  }
  float* out = (is_dv ? a.dv : a.dk) + base * D;
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    const int rl = r0 + g + 8 * half;
    if (rl < ns) {
      float* row = out + (long long)(s0 + rl) * row_stride;
#pragma unroll
      for (int j = 0; j < NJ; ++j)
        *reinterpret_cast<float2*>(row + 8 * j + 2 * tg) = make_float2(acc[j][2 * half], acc[j][2 * half + 1]);
    }
  }
}

template <int D>
cudaError_t launch_dkv_d(const BackwardArgs& a, cudaStream_t s) {
  const size_t sk = sizeof(DkvSmem<D>);
  cudaError_t e = cudaFuncSetAttribute(dkv_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sk);
  if (e != cudaSuccess) return e;
  dkv_kernel<D><<<dim3((a.T + BT - 1) / BT, a.B * a.H), NTK, sk, s>>>(a);
  return cudaGetLastError();
}
template <int D>
cudaError_t launch_dq_d(const BackwardArgs& a, cudaStream_t s) {
  const size_t sq = sizeof(DqSmem<D>);
  cudaError_t e = cudaFuncSetAttribute(dq_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sq);
  if (e != cudaSuccess) return e;
  dq_kernel<D><<<dim3((a.T + BT - 1) / BT, a.B * a.H), NTB, sq, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_backward_slots(const BackwardArgs& a, cudaStream_t s) {
  if (a.B * a.H > 65535 || a.C > kMaxC) return cudaErrorInvalidConfiguration;
  slots_kernel<<<a.B * a.H, 32, 0, s>>>(a);
  return cudaGetLastError();
}
cudaError_t launch_backward_dkv(const BackwardArgs& a, int d, cudaStream_t s) {
  return d == 64 ? launch_dkv_d<64>(a, s) : launch_dkv_d<128>(a, s);
}
cudaError_t launch_backward_dq(const BackwardArgs& a, int d, cudaStream_t s) {
  return d == 64 ? launch_dq_d<64>(a, s) : launch_dq_d<128>(a, s);
}

size_t backward_slot_bytes(int BH, int T) {
  return (size_t)BH * T * sizeof(int32_t) + (size_t)BH * (T + 1) * kMaxC * sizeof(int32_t);
}

}  // namespace dla

// dla_decode.cu -- K3: one recurrent DLA step for every (batch, head) stream
// against its persistent fp32 cache (Sec. 3.1 inference rule, Algorithm 2,
// Eq. capacity_bounded_output).  Bandwidth-bound: the step reads every live
// state once and writes one state (plus one more when a merge happens).
//
// One CTA (512 threads) per stream.  Thread (row j, part p) owns row j of a
// state and a contiguous quarter (d = 128) of its columns, so every access is
// a coalesced 16-byte load / store and per-row reductions stay inside a quad.
//   pass A: stream the open state into shared memory while forming
//           beta = v^T S k, gam = |S|^2 and u = S q;
//   decide: score, boundary, and (full cache) the adjacent-pair argmin;
//   pass B: stream the other states once, accumulating lambda' (S q) with the
//           post-step logical slot of each state, write the merged state, then
//           the updated open state (S + v k^T) or the new state v k^T.
#include "dla_common.cuh"

namespace dla {

namespace {

constexpr int NT = 512;

template <int D>
struct DecSmem {
  float S[D * D];  // open state
  float q[D], k[D], v[D];
  float u[D];      // S_open q
  double ibar[kMaxC];
  int n[kMaxC];
  int slot[kMaxC];
  int newidx[kMaxC];  // post-step logical slot of every pre-step entry
  double red[NT / 32][2];
  float qk;
  double a_norm;
  double Ival;
  int m, bflag, jmerge, m_new;
};

}  // namespace

template <int D, typename Tin, typename Tout>
__global__ void __launch_bounds__(NT, 2) decode_kernel(DecodeArgs a) {
  constexpr int TPR = NT / D;   // threads per row
  constexpr int KPT = D / TPR;  // columns per thread
  extern __shared__ __align__(16) unsigned char smem_raw[];
  DecSmem<D>& sm = *reinterpret_cast<DecSmem<D>*>(smem_raw);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int bh = blockIdx.x;
  const int C = a.C;
  const int row = tid / TPR, part = tid % TPR;
  const int col0 = part * KPT;
  float* states = a.states + (long long)bh * C * D * D;

  if (tid == 0) sm.m = min(max(a.m[bh], 0), C);  // a corrupted cache cannot index out of bounds
  for (int i = tid; i < C; i += NT) {
    const int sl = a.slot[(long long)bh * C + i];
    sm.slot[i] = (sl >= 0 && sl < C) ? sl : i;
    sm.n[i] = a.n[(long long)bh * C + i];
    sm.ibar[i] = a.ibar[(long long)bh * C + i];
  }
  const Tin* qin = reinterpret_cast<const Tin*>(a.q) + (long long)bh * D;
  const Tin* kin = reinterpret_cast<const Tin*>(a.k) + (long long)bh * D;
  const Tin* vin = reinterpret_cast<const Tin*>(a.v) + (long long)bh * D;
  for (int i = tid; i < D; i += NT) {
    sm.q[i] = to_f32(qin[i]);
    sm.k[i] = to_f32(kin[i]);
    sm.v[i] = to_f32(vin[i]);
  }
  __syncthreads();
  if (warp == 0) {  // |k|^2 |v|^2 and q.k
    float kk = 0.f, vv = 0.f, qk = 0.f;
    for (int i = lane; i < D; i += 32) {
      kk += sm.k[i] * sm.k[i];
      vv += sm.v[i] * sm.v[i];
      qk += sm.q[i] * sm.k[i];
    }
    kk = warp_sum(kk);
    vv = warp_sum(vv);
    qk = warp_sum(qk);
    if (lane == 0) {
      sm.a_norm = (double)kk * (double)vv;
      sm.qk = qk;
    }
  }
  const int m = sm.m;
  // ---------------------------------------------------------------- pass A
  double beta_p = 0.0, gam_p = 0.0;
  if (m > 0) {
    const float* src = states + (long long)sm.slot[m - 1] * D * D + row * D + col0;
    float4 r4[KPT / 4];
#pragma unroll
    for (int c = 0; c < KPT / 4; ++c) r4[c] = load4(src + 4 * c);
    float dk = 0.f, dq = 0.f;
#pragma unroll
    for (int c = 0; c < KPT / 4; ++c) {
      const int cc = col0 + 4 * c;
      store4(sm.S + row * D + cc, r4[c]);
      dk += r4[c].x * sm.k[cc] + r4[c].y * sm.k[cc + 1] + r4[c].z * sm.k[cc + 2] + r4[c].w * sm.k[cc + 3];
      dq += r4[c].x * sm.q[cc] + r4[c].y * sm.q[cc + 1] + r4[c].z * sm.q[cc + 2] + r4[c].w * sm.q[cc + 3];
      gam_p += (double)r4[c].x * r4[c].x + (double)r4[c].y * r4[c].y + (double)r4[c].z * r4[c].z +
               (double)r4[c].w * r4[c].w;
    }
#pragma unroll
    for (int o = 1; o < TPR; o <<= 1) {
      dk += __shfl_xor_sync(0xffffffffu, dk, o);
      dq += __shfl_xor_sync(0xffffffffu, dq, o);
    }
    if (part == 0) {
      sm.u[row] = dq;
      beta_p = (double)sm.v[row] * (double)dk;
    }
  }
  beta_p = warp_sum(beta_p);
  gam_p = warp_sum(gam_p);
  if (lane == 0) {
    sm.red[warp][0] = beta_p;
    sm.red[warp][1] = gam_p;
  }
  __syncthreads();
  // ---------------------------------------------------------------- decide
  if (warp == 0) {
    double beta = 0.0, gam = 0.0;
    for (int w = 0; w < NT / 32; ++w) {
      beta += sm.red[w][0];
      gam += sm.red[w][1];
    }
    int bflag = 1, j = -1;
    double I = 0.0;
    if (m > 0) {
      I = info_score(sm.a_norm, beta, gam, (double)D * (double)D, a.sp);
      bflag = (I >= a.sp.tau) ? 1 : 0;
      if (bflag && m == C) j = pair_argmin_warp(sm.n, sm.ibar, m);
    }
    // post-step logical slot of each pre-step entry
    for (int i = lane; i < m; i += 32) sm.newidx[i] = (j >= 0 && i > j) ? i - 1 : i;
    __syncwarp();
    if (lane == 0) {
      sm.Ival = I;
      sm.bflag = bflag;
      sm.jmerge = j;
    }
    __syncwarp();
  }
  __syncthreads();
  const int bflag = sm.bflag, jm = sm.jmerge;
  const int m_new = bflag ? (jm >= 0 ? m : m + 1) : m;
  const float* lam = a.lam ? a.lam + (long long)bh * C : nullptr;
  // ---------------------------------------------------------------- pass B
  float acc = 0.f;  // this thread's share of (sum lambda' S q)_row over its columns
  const int open = m - 1;
  for (int i = 0; i < m; ++i) {
    if (i == open) continue;
    if (jm >= 0 && i == jm + 1) continue;  // consumed with its merge partner
    const float w = lam ? lam[sm.newidx[i]] : 1.f;
    const float* src = states + (long long)sm.slot[i] * D * D + row * D + col0;
    float4 r4[KPT / 4];
#pragma unroll
    for (int c = 0; c < KPT / 4; ++c) r4[c] = load4(src + 4 * c);
    if (jm >= 0 && i == jm) {
      // merge partner: global state, or the open state in shared memory; the
      // partner is streamed one 16-byte piece at a time to keep registers low
      const float* psrc = (jm + 1 == open) ? sm.S + row * D + col0
                                           : states + (long long)sm.slot[jm + 1] * D * D + row * D + col0;
      float* dst = states + (long long)sm.slot[jm] * D * D + row * D + col0;
      float d = 0.f, dp = 0.f;
#pragma unroll
      for (int c = 0; c < KPT / 4; ++c) {
        const int cc = col0 + 4 * c;
        const float4 p4 = load4(psrc + 4 * c);
        d += r4[c].x * sm.q[cc] + r4[c].y * sm.q[cc + 1] + r4[c].z * sm.q[cc + 2] + r4[c].w * sm.q[cc + 3];
        dp += p4.x * sm.q[cc] + p4.y * sm.q[cc + 1] + p4.z * sm.q[cc + 2] + p4.w * sm.q[cc + 3];
        store4(dst + 4 * c, make_float4(r4[c].x + p4.x, r4[c].y + p4.y, r4[c].z + p4.z, r4[c].w + p4.w));
      }
      acc += w * d;
      if (jm + 1 != open) acc += w * dp;  // the open state's share is added below from u
      continue;
    }
    float d = 0.f;
#pragma unroll
    for (int c = 0; c < KPT / 4; ++c) {
      const int cc = col0 + 4 * c;
      d += r4[c].x * sm.q[cc] + r4[c].y * sm.q[cc + 1] + r4[c].z * sm.q[cc + 2] + r4[c].w * sm.q[cc + 3];
    }
    acc += w * d;
  }
#pragma unroll
  for (int o = 1; o < TPR; o <<= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  // open state's read-out (S_open q from pass A) and the token's own term
  float orow = acc;
  const float vj = sm.v[row];
  if (m > 0) {
    const float wopen = lam ? lam[sm.newidx[open]] : 1.f;
    orow += wopen * sm.u[row];
  }
  {
    // the token state v k^T is read out with the slot it lands in
    const int slot_tok = bflag ? (m_new - 1) : (m - 1);
    const float wt = lam ? lam[slot_tok] : 1.f;
    orow += wt * sm.qk * vj;
  }
  // ---------------------------------------------------------------- write states
  if (!bflag) {  // S_open += v k^T
    float* dst = states + (long long)sm.slot[open] * D * D + row * D + col0;
#pragma unroll
    for (int c = 0; c < KPT / 4; ++c) {
      const int cc = col0 + 4 * c;
      float4 s4 = load4(sm.S + row * D + cc);
      store4(dst + 4 * c, make_float4(s4.x + vj * sm.k[cc], s4.y + vj * sm.k[cc + 1],
                                      s4.z + vj * sm.k[cc + 2], s4.w + vj * sm.k[cc + 3]));
    }
  } else {  // new state v k^T in the freed slot (after a merge) or slot m
    const int phys = (jm >= 0) ? sm.slot[jm + 1] : m;
    float* dst = states + (long long)phys * D * D + row * D + col0;
#pragma unroll
    for (int c = 0; c < KPT / 4; ++c) {
      const int cc = col0 + 4 * c;
      store4(dst + 4 * c, make_float4(vj * sm.k[cc], vj * sm.k[cc + 1], vj * sm.k[cc + 2], vj * sm.k[cc + 3]));
    }
  }
  if (part == 0) {
    Tout* o = reinterpret_cast<Tout*>(a.o) + (long long)bh * D;
    o[row] = from_f32<Tout>(orow);
  }
  __syncthreads();
  // ---------------------------------------------------------------- metadata
  if (warp == 0) {
    const double I = sm.Ival;
    if (!bflag) {
      if (lane == 0) {
        sm.n[open] += 1;
        sm.ibar[open] += I;
      }
    } else {
      int phys_new = m;
      if (jm >= 0) {
        const int freed = sm.slot[jm + 1];
        if (lane == 0) {
          sm.n[jm] += sm.n[jm + 1];
          sm.ibar[jm] += sm.ibar[jm + 1];
        }
        __syncwarp();
        for (int base = jm + 1; base < m - 1; base += 32) {
          int i = base + lane;
          int nv = 0, sv = 0;
          double iv = 0.0;
          if (i < m - 1) {
            nv = sm.n[i + 1];
            sv = sm.slot[i + 1];
            iv = sm.ibar[i + 1];
          }
          __syncwarp();
          if (i < m - 1) {
            sm.n[i] = nv;
            sm.slot[i] = sv;
            sm.ibar[i] = iv;
          }
          __syncwarp();
        }
        phys_new = freed;
      }
      if (lane == 0) {
        sm.slot[m_new - 1] = phys_new;
        sm.n[m_new - 1] = 1;
        sm.ibar[m_new - 1] = I;
      }
    }
    __syncwarp();
    for (int i = lane; i < C; i += 32) {
      a.slot[(long long)bh * C + i] = sm.slot[i];
      a.n[(long long)bh * C + i] = (i < m_new) ? sm.n[i] : 0;
      a.ibar[(long long)bh * C + i] = (i < m_new) ? sm.ibar[i] : 0.0;
    }
    if (lane == 0) {
      a.m[bh] = m_new;
      if (a.boundary) a.boundary[bh] = (uint8_t)bflag;
      if (a.merge_idx) a.merge_idx[bh] = jm;
    }
  }
}

template <int D, typename Tin, typename Tout>
static cudaError_t launch_dec_t(const DecodeArgs& a, cudaStream_t st) {
  const size_t smem = sizeof(DecSmem<D>);
  auto kern = decode_kernel<D, Tin, Tout>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  kern<<<a.B * a.H, NT, smem, st>>>(a);
  return cudaGetLastError();
}

template <int D>
static cudaError_t launch_dec_d(const DecodeArgs& a, bool in_bf16, cudaStream_t st) {
  if (in_bf16) return a.out_bf16 ? launch_dec_t<D, __nv_bfloat16, __nv_bfloat16>(a, st)
                                 : launch_dec_t<D, __nv_bfloat16, float>(a, st);
  return a.out_bf16 ? launch_dec_t<D, float, __nv_bfloat16>(a, st) : launch_dec_t<D, float, float>(a, st);
}

cudaError_t launch_decode(const DecodeArgs& a, int d, bool in_bf16, cudaStream_t st) {
  return d == 128 ? launch_dec_d<128>(a, in_bf16, st) : launch_dec_d<64>(a, in_bf16, st);
}

// ---------------------------------------------------------------- init cache
__global__ void init_cache_kernel(int32_t* slot, int32_t* n, double* ibar, int32_t* m, int BH, int C) {
  const long long total = (long long)BH * C;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    slot[e] = (int32_t)(e % C);
    n[e] = 0;
    ibar[e] = 0.0;
    if (e % C == 0) m[e / C] = 0;
  }
}

cudaError_t launch_init_cache(int32_t* slot, int32_t* n, double* ibar, int32_t* m, int BH, int C,
                              cudaStream_t s) {
  long long total = (long long)BH * C;
  int blocks = (int)((total + 255) / 256);
  if (blocks > 4096) blocks = 4096;
  if (blocks < 1) blocks = 1;
  init_cache_kernel<<<blocks, 256, 0, s>>>(slot, n, ibar, m, BH, C);
  return cudaGetLastError();
}

}  // namespace dla

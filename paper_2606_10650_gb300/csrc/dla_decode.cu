// dla_decode.cu -- K3: one recurrent DLA step for every (batch, head) stream
// against its persistent fp32 cache (Sec. 3.1 inference rule, Algorithm 2,
// Eq. capacity_bounded_output).  Bandwidth-bound: the step reads every live
// state once and writes one state (plus the merged one when a merge happens).
//
// One CTA (512 threads) per stream.  A state row (d_k floats) is read by
// LPR = d/4 consecutive lanes, one 16-byte load each, so a warp reads whole
// rows contiguously; thread (row group rg, lane-in-row li) owns columns
// 4li..4li+3 of rows rg, rg + NT/LPR, ...  The thread keeps its four q and k
// values in registers and accumulates a partial o for each of its rows over all
// states; the lanes of a row are reduced once at the end.
//   pass A: stream the open state into shared memory while forming
//           beta = v^T S k and gam = |S|^2;
//   decide: score, boundary, and (full cache) the adjacent-pair argmin;
//   pass B: stream every other state once, weighting S q with the post-step
//           logical slot's lambda; write the merged state, then the updated
//           open state (S + v k^T) or the new state v k^T.
#include "dla_common.cuh"

namespace dla {

namespace {

constexpr int NT = 512;

template <int D>
struct DecSmem {
  float S[D * D];  // open state
  float v[D];
  float red[NT / 32][5];
  double ibar[kMaxC];
  int n[kMaxC];
  int slot[kMaxC];
  int newidx[kMaxC];  // post-step logical slot of every pre-step entry
  float qk, Ival;
  int m, bflag, jmerge;
};

}  // namespace

template <int D, typename Tin, typename Tout>
__global__ void __launch_bounds__(NT, 2) decode_kernel(DecodeArgs a) {
  constexpr int LPR = D / 4;    // lanes per row
  constexpr int RG = NT / LPR;  // row groups
  constexpr int RPT = D / RG;   // rows per thread
  extern __shared__ __align__(16) unsigned char smem_raw[];
  DecSmem<D>& sm = *reinterpret_cast<DecSmem<D>*>(smem_raw);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int bh = blockIdx.x;
  const int C = a.C;
  const int li = tid % LPR, rg = tid / LPR;
  const int col = 4 * li;
  float* states = a.states + (long long)bh * C * D * D;

  // a corrupted cache is reported (device check) and clamped, so that it
  // cannot index out of bounds
  if (tid == 0) {
    const int m0 = a.m[bh];
    if ((m0 < 0 || m0 > C) && a.status) atomicCAS(a.status, 0, 6);
    sm.m = min(max(m0, 0), C);
  }
  for (int i = tid; i < C; i += NT) {
    const int sl = a.slot[(long long)bh * C + i];
    if ((sl < 0 || sl >= C) && a.status) atomicCAS(a.status, 0, 6);
    sm.slot[i] = (sl >= 0 && sl < C) ? sl : i;
    sm.n[i] = a.n[(long long)bh * C + i];
    sm.ibar[i] = a.ibar[(long long)bh * C + i];
  }
  const Tin* qin = reinterpret_cast<const Tin*>(a.q) + (long long)bh * D;
  const Tin* kin = reinterpret_cast<const Tin*>(a.k) + (long long)bh * D;
  const Tin* vin = reinterpret_cast<const Tin*>(a.v) + (long long)bh * D;
  const float4 q4 = make_float4(to_f32(qin[col]), to_f32(qin[col + 1]), to_f32(qin[col + 2]), to_f32(qin[col + 3]));
  const float4 k4 = make_float4(to_f32(kin[col]), to_f32(kin[col + 1]), to_f32(kin[col + 2]), to_f32(kin[col + 3]));
  for (int i = tid; i < D; i += NT) sm.v[i] = to_f32(vin[i]);
  __syncthreads();
  const int m = sm.m;
  // ---------------------------------------------------------------- pass A
  float beta_p = 0.f, gam_p = 0.f, kk_p = 0.f, vv_p = 0.f, qk_p = 0.f;
  if (rg == 0) {  // |k|^2 and q.k: each column block counted once
    kk_p = k4.x * k4.x + k4.y * k4.y + k4.z * k4.z + k4.w * k4.w;
    qk_p = q4.x * k4.x + q4.y * k4.y + q4.z * k4.z + q4.w * k4.w;
  }
  if (tid < D) vv_p = sm.v[tid] * sm.v[tid];
  if (m > 0) {
    const float* src = states + (long long)sm.slot[m - 1] * D * D;
    float4 s4[RPT];
#pragma unroll
    for (int r = 0; r < RPT; ++r) s4[r] = load4(src + (rg + r * RG) * D + col);
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
      const int row = rg + r * RG;
      store4(sm.S + row * D + col, s4[r]);
      const float dk = s4[r].x * k4.x + s4[r].y * k4.y + s4[r].z * k4.z + s4[r].w * k4.w;
      beta_p += sm.v[row] * dk;
      gam_p += s4[r].x * s4[r].x + s4[r].y * s4[r].y + s4[r].z * s4[r].z + s4[r].w * s4[r].w;
    }
  }
  beta_p = warp_sum(beta_p);
  gam_p = warp_sum(gam_p);
  kk_p = warp_sum(kk_p);
  vv_p = warp_sum(vv_p);
  qk_p = warp_sum(qk_p);
  if (lane == 0) {
    sm.red[warp][0] = beta_p;
    sm.red[warp][1] = gam_p;
    sm.red[warp][2] = kk_p;
    sm.red[warp][3] = vv_p;
    sm.red[warp][4] = qk_p;
  }
  __syncthreads();
  // ---------------------------------------------------------------- decide
  if (warp == 0) {
    float beta = 0.f, gam = 0.f, kk = 0.f, vv = 0.f, qk = 0.f;
    for (int w = 0; w < NT / 32; ++w) {
      beta += sm.red[w][0];
      gam += sm.red[w][1];
      kk += sm.red[w][2];
      vv += sm.red[w][3];
      qk += sm.red[w][4];
    }
    int bflag = 1, j = -1;
    float I = 0.f;
    if (m > 0) {
      I = info_score(kk * vv, beta, gam, (float)(D * D), a.sp);
      bflag = ((double)I >= a.sp.tau) ? 1 : 0;
      if (bflag && m == C) j = pair_argmin_warp(sm.n, sm.ibar, m);
    }
    for (int i = lane; i < m; i += 32) sm.newidx[i] = (j >= 0 && i > j) ? i - 1 : i;
    __syncwarp();
    if (lane == 0) {
      sm.Ival = I;
      sm.qk = qk;
      sm.bflag = bflag;
      sm.jmerge = j;
    }
    __syncwarp();
  }
  __syncthreads();
  const int bflag = sm.bflag, jm = sm.jmerge;
  const int m_new = bflag ? (jm >= 0 ? m : m + 1) : m;
  const float* lam = a.lam ? a.lam + (long long)bh * C : nullptr;
  const int open = m - 1;
  // ---------------------------------------------------------------- pass B
  float acc[RPT];
#pragma unroll
  for (int r = 0; r < RPT; ++r) acc[r] = 0.f;
  for (int i = 0; i < m; ++i) {
    if (i == open) continue;
    if (jm >= 0 && i == jm + 1) continue;  // consumed with its merge partner
    const float w = lam ? lam[sm.newidx[i]] : 1.f;
    const float* src = states + (long long)sm.slot[i] * D * D;
    float4 s4[RPT];
#pragma unroll
    for (int r = 0; r < RPT; ++r) s4[r] = load4(src + (rg + r * RG) * D + col);
    if (jm >= 0 && i == jm) {
      // merge partner: a global state, or the open state in shared memory
      const bool part_open = (jm + 1 == open);
      const float* psrc = part_open ? sm.S : states + (long long)sm.slot[jm + 1] * D * D;
      float* dst = states + (long long)sm.slot[jm] * D * D;
#pragma unroll
      for (int r = 0; r < RPT; ++r) {
        const int off = (rg + r * RG) * D + col;
        const float4 p4 = load4(psrc + off);
        float d = s4[r].x * q4.x + s4[r].y * q4.y + s4[r].z * q4.z + s4[r].w * q4.w;
        if (!part_open) d += p4.x * q4.x + p4.y * q4.y + p4.z * q4.z + p4.w * q4.w;
        acc[r] += w * d;  // an open partner's share is added below from shared memory
        store4(dst + off, make_float4(s4[r].x + p4.x, s4[r].y + p4.y, s4[r].z + p4.z, s4[r].w + p4.w));
      }
      continue;
    }
#pragma unroll
    for (int r = 0; r < RPT; ++r)
      acc[r] += w * (s4[r].x * q4.x + s4[r].y * q4.y + s4[r].z * q4.z + s4[r].w * q4.w);
  }
  // the open state's read-out, from its copy in shared memory
  if (m > 0) {
    const float wopen = lam ? lam[sm.newidx[open]] : 1.f;
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
      const float4 s4 = load4(sm.S + (rg + r * RG) * D + col);
      acc[r] += wopen * (s4.x * q4.x + s4.y * q4.y + s4.z * q4.z + s4.w * q4.w);
    }
  }
  // reduce the lanes of each row
#pragma unroll
  for (int r = 0; r < RPT; ++r)
#pragma unroll
    for (int o = 1; o < LPR; o <<= 1) acc[r] += __shfl_xor_sync(0xffffffffu, acc[r], o);
  // the token state v k^T is read out with the slot it lands in
  const int slot_tok = bflag ? (m_new - 1) : (m - 1);
  const float wt = lam ? lam[slot_tok] : 1.f;
  const float qk = sm.qk;
  // ---------------------------------------------------------------- write states
  if (!bflag) {  // S_open += v k^T
    float* dst = states + (long long)sm.slot[open] * D * D;
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
      const int row = rg + r * RG;
      const float vj = sm.v[row];
      const float4 s4 = load4(sm.S + row * D + col);
      store4(dst + row * D + col,
             make_float4(s4.x + vj * k4.x, s4.y + vj * k4.y, s4.z + vj * k4.z, s4.w + vj * k4.w));
    }
  } else {  // the new state v k^T goes to the freed slot (after a merge) or slot m
    const int phys = (jm >= 0) ? sm.slot[jm + 1] : m;
    float* dst = states + (long long)phys * D * D;
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
      const int row = rg + r * RG;
      const float vj = sm.v[row];
      store4(dst + row * D + col, make_float4(vj * k4.x, vj * k4.y, vj * k4.z, vj * k4.w));
    }
  }
  if (li == 0) {
    Tout* o = reinterpret_cast<Tout*>(a.o) + (long long)bh * D;
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
      const int row = rg + r * RG;
      o[row] = from_f32<Tout>(acc[r] + wt * qk * sm.v[row]);
    }
  }
  __syncthreads();
  // ---------------------------------------------------------------- metadata
  if (warp == 0) {
    const double I = (double)sm.Ival;
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
  e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
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

// ---------------------------------------------------------------- cache norm bounds
__global__ void __launch_bounds__(256) cache_bounds_kernel(const float* states, const int32_t* slot, const int32_t* m,
                                                           int C, int d, float* out) {
  const int i = blockIdx.x, bh = blockIdx.y;
  const int mm = m[bh];
  if (i >= mm || i >= C) return;
  int sl = slot[(long long)bh * C + i];
  if (sl < 0 || sl >= C) sl = i;  // an invalid slot map is reported by the kernels that use it
  const float* S = states + ((long long)bh * C + sl) * d * d;
  float acc = 0.f;
  for (int e = threadIdx.x; e < d * d / 4; e += blockDim.x) {
    const float4 x = reinterpret_cast<const float4*>(S)[e];
    acc += x.x * x.x + x.y * x.y + x.z * x.z + x.w * x.w;
  }
  __shared__ float red[8];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int w = 0; w < 8; ++w) t += red[w];
    out[(long long)bh * C + i] = sqrtf(t) * 1.001f;  // fp32 summation error: a bound, not the norm
  }
}

cudaError_t launch_cache_bounds(const float* states, const int32_t* slot, const int32_t* m, int BH, int C, int d,
                                float* out, cudaStream_t s) {
  if (BH > 65535) return cudaErrorInvalidConfiguration;
  cache_bounds_kernel<<<dim3(C, BH), 256, 0, s>>>(states, slot, m, C, d, out);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- packed rows
// Row lengths and first token rows of a packed batch from its cumulative
// offsets (see launch_varlen_rows).
__global__ void varlen_rows_kernel(const int32_t* cu, int B, int T, long long total, int32_t* lens, int32_t* start,
                                   int32_t* status) {
  for (int b = blockIdx.x * blockDim.x + threadIdx.x; b < B; b += gridDim.x * blockDim.x) {
    long long s0 = cu[b], s1 = cu[b + 1];
    const bool bad = s0 < 0 || s1 < s0 || s1 > total || s1 - s0 > T;
    if (bad) {
      atomicCAS(status, 0, 6);
      s0 = s0 < 0 ? 0 : (s0 > total ? total : s0);
      s1 = s1 < s0 ? s0 : (s1 > total ? total : s1);
      if (s1 - s0 > T) s1 = s0 + T;
    }
    start[b] = (int32_t)s0;
    lens[b] = (int32_t)(s1 - s0);
  }
}

cudaError_t launch_varlen_rows(const int32_t* cu, int B, int T, long long total, int32_t* lens, int32_t* start,
                               int32_t* status, cudaStream_t s) {
  int blocks = (B + 255) / 256;
  if (blocks > 1024) blocks = 1024;
  varlen_rows_kernel<<<blocks, 256, 0, s>>>(cu, B, T, total, lens, start, status);
  return cudaGetLastError();
}

}  // namespace dla

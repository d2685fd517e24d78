// Query proxies from proxy hidden states (Section 3.2.1, the paper's own
// construction): per (layer, request) N proxy hidden states
// H~_i = mu_pre + gamma * sigma_pre * z_i are drawn in the model's hidden
// space (d_model features; statistics over the prefill hidden states),
// rounded to bf16 and projected by the query projection,
// q~_i = W_Q H~_i (+ b_Q), then rotated to the proxies' position (RoPE,
// rotate-half pairs within each head) and rounded to bf16.
//
//  - hidden_sample_kernel: one thread per (proxy, quad of dimensions): one
//    Philox4x64-10 draw (key (seed, 1), counter (i * d_model/8 + q, 0, b,
//    layer)) gives the eight normals of dims [4q, 4q+4) and
//    [d_model/2 + 4q, +4); writes H~ [L][B][Npad][d_model] bf16 (rows past N
//    zero) into the workspace. Block (0, b, 0) also writes the RoPE table of
//    request b (cos, sin per rotation pair).
//  - hidden_proj_kernel: persistent tcgen05 GEMM, one 192-thread CTA per SM:
//    D[128 proxies x NT features] = H~ tile . W_Q tile^T over d_model in
//    64-wide K blocks (TMA, 128-byte swizzle, 4-stage ring), accumulators in
//    tensor memory (two buffers of NT columns), warp 0 loads, warp 1 issues
//    the MMAs, warps 2-5 drain: thread = proxy row, 16-column tensor-memory
//    loads of each rotation pair's two halves, + bias, rotation, bf16 round,
//    stores into the caller layout [L][B][Hq][N][d].
// Tiles are ordered (layer, request) > feature tile > proxy tile, so the
// CTAs running the proxy tiles of one feature tile read its W_Q rows at the
// same time (DRAM once, then L2).
#include <algorithm>
#include <cstring>

#include "common.cuh"
#include "rng.cuh"
#include "umma.cuh"

namespace mmshift {
namespace {

using namespace umma;

constexpr int HM = 128;          // proxy rows per tile (MMA M)
constexpr int HK = 64;           // hidden features per K block: 128 bytes of bf16
constexpr int HSTAGE = 4;        // ring depth
constexpr int HTHREADS = 192;    // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr int HNEPI = 128;
constexpr int HACC = 256;        // tensor-memory columns per accumulator buffer

__host__ __device__ constexpr int stage_bytes(int nt) { return HM * 128 + nt * 128; }

__device__ __forceinline__ void decode_tile(const HiddenJob& J, int t, int& lb, int& nt, int& mt) {
  mt = t % J.MT;
  const int r = t / J.MT;
  nt = r % J.NTL;
  lb = r / J.NTL;
}

__device__ __forceinline__ void store4_bf16(__nv_bfloat16* dst, float a, float b, float c, float d) {
  __nv_bfloat162 lo = __floats2bfloat162_rn(a, b), hi = __floats2bfloat162_rn(c, d);
  uint2 u;
  u.x = *reinterpret_cast<uint32_t*>(&lo);
  u.y = *reinterpret_cast<uint32_t*>(&hi);
  *reinterpret_cast<uint2*>(dst) = u;
}

__global__ void __launch_bounds__(256) hidden_sample_kernel(HiddenJob J) {
  const int b = blockIdx.y, l = blockIdx.z;
  const int nq = J.DM / 8;
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (blockIdx.x == 0 && l == 0 && J.rope && threadIdx.x < J.d / 2) {
    // angle = pos * theta^(-2k/d), reduced modulo 2*pi in double
    const int k = threadIdx.x;
    const double ang = (double)J.pos[b] * pow((double)J.rope_theta, -2.0 * k / (double)J.d);
    const double red = ang - 6.283185307179586 * rint(ang / 6.283185307179586);
    float sv, cv;
    sincosf((float)red, &sv, &cv);
    J.rope[((size_t)b * (J.d / 2) + k) * 2] = cv;
    J.rope[((size_t)b * (J.d / 2) + k) * 2 + 1] = sv;
  }
  if (e >= J.Npad * nq) return;
  const int i = e / nq, q = e - i * nq;
  __nv_bfloat16* row = J.hs + (((size_t)l * J.B + b) * J.Npad + i) * J.DM;
  if (i >= J.N) {
    store4_bf16(row + 4 * q, 0.f, 0.f, 0.f, 0.f);
    store4_bf16(row + J.DM / 2 + 4 * q, 0.f, 0.f, 0.f, 0.f);
    return;
  }
  const float* mu = J.hstats + ((size_t)l * J.B + b) * 2 * J.DM;
  const float* sg = mu + J.DM;
  float z[8];
  normals8_at((uint64_t)i * (uint64_t)nq + (uint64_t)q, 0ull, b, J.layer_id0 + l, J.seed, 1ull, z);
  float v[8];
  const int j0 = 4 * q, j1 = J.DM / 2 + 4 * q;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    v[k] = fmaf(J.gamma * __ldg(sg + j0 + k), z[k], __ldg(mu + j0 + k));
    v[4 + k] = fmaf(J.gamma * __ldg(sg + j1 + k), z[4 + k], __ldg(mu + j1 + k));
  }
  store4_bf16(row + j0, v[0], v[1], v[2], v[3]);
  store4_bf16(row + j1, v[4], v[5], v[6], v[7]);
}

template <int D>
__global__ void __launch_bounds__(HTHREADS, 1)
    hidden_proj_kernel(const __grid_constant__ CUtensorMap amap,
                       const __grid_constant__ CUtensorMap wmap, const __grid_constant__ HiddenJob J) {
  extern __shared__ unsigned char smraw[];
  unsigned char* sm =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
  __shared__ uint64_t full[HSTAGE], empty[HSTAGE], tfull[2], tempty[2], drain;
  __shared__ uint32_t tbase;
  __shared__ int abort_flag;
  volatile int* abort_ = &abort_flag;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int SB = stage_bytes(J.NT);
  const int nkb = J.DM / HK;

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < HSTAGE; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], HNEPI);
    }
    mbar_init(&drain, 1);
    fence_barrier_init();
    prefetch_tmap(&amap);
    prefetch_tmap(&wmap);
  }
  if (warp == 1) {
    tmem_alloc(&tbase, 2 * HACC);
    tmem_relinquish();
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = tbase;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      ArmedStages armed;
      bool ok = true;
      for (int t = blockIdx.x; t < J.tiles && ok; t += gridDim.x) {
        int lb, nt, mt;
        decode_tile(J, t, lb, nt, mt);
        const int l = lb / J.B;
        for (int kb = 0; kb < nkb; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_)) { ok = false; break; }
          unsigned char* a = sm + stage * SB;
          mbar_expect_tx(&full[stage], (uint32_t)SB);
          armed.arm(stage, phase);
          tma_load_3d(a, &amap, &full[stage], kb * HK, mt * HM, lb);
          tma_load_3d(a + HM * 128, &wmap, &full[stage], kb * HK, nt * J.NT, l);
          if (++stage == HSTAGE) { stage = 0; phase ^= 1u; }
        }
      }
      // every load issued has landed before the CTA's shared memory goes
      if (!armed.drain(full)) *abort_ = 1;
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, bphase = 0;
      const uint32_t idesc = idesc_bf16_f32(HM, J.NT);
      bool ok = true, issued = false;
      for (int t = blockIdx.x, j = 0; t < J.tiles && ok; t += gridDim.x, ++j) {
        const int buf = j & 1;
        if (!mbar_wait(&tempty[buf], ((bphase >> buf) & 1u) ^ 1u, abort_)) break;
        bphase ^= 1u << buf;
        fence_after();
        const uint32_t dcol = tmem + (uint32_t)(buf * HACC);
        for (int kb = 0; kb < nkb; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_)) { ok = false; break; }
          fence_after();
          const uint32_t a = smem_u32(sm + stage * SB);
#pragma unroll
          for (int w = 0; w < HK / 16; ++w)
            mma_bf16(dcol, sdesc_k_sw128(a + w * 32), sdesc_k_sw128(a + HM * 128 + w * 32), idesc,
                     (kb | w) ? 1u : 0u);
          mma_commit(&empty[stage]);
          issued = true;
          if (++stage == HSTAGE) { stage = 0; phase ^= 1u; }
        }
        if (ok) mma_commit(&tfull[buf]);
      }
      // every MMA issued has finished before the CTA's tensor memory goes
      if (issued) {
        mma_commit(&drain);
        if (!mbar_wait_drain(&drain, 0)) *abort_ = 1;
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp % 4;                 // tensor-memory lane quarter of this warp
    const int row = q * 32 + lane;          // proxy row of the tile
    uint32_t bphase = 0;
    for (int t = blockIdx.x, j = 0; t < J.tiles; t += gridDim.x, ++j) {
      const int buf = j & 1;
      if (!mbar_wait(&tfull[buf], (bphase >> buf) & 1u, abort_)) break;
      bphase ^= 1u << buf;
      fence_after();
      int lb, nt, mt;
      decode_tile(J, t, lb, nt, mt);
      const int l = lb / J.B, b = lb - l * J.B;
      const int m = mt * HM + row;
      const bool valid = m < J.N;
      const uint32_t tacc = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * HACC);
      const __nv_bfloat16* bias = J.bias ? J.bias + (size_t)l * J.F + (size_t)nt * J.NT : nullptr;
      const float* rope = J.rope ? J.rope + (size_t)b * D : nullptr;   // [d/2][2]
      for (int hh = 0; hh < J.NT / D; ++hh) {
        const int hq = nt * (J.NT / D) + hh;
        __nv_bfloat16* dst = J.out + ((((size_t)l * J.B + b) * J.Hq + hq) * J.N + m) * D;
#pragma unroll 1
        for (int c = 0; c < D / 2; c += 16) {
          float x[16], y[16];
          tmem_ld16(tacc + (uint32_t)(hh * D + c), x);
          tmem_ld16(tacc + (uint32_t)(hh * D + D / 2 + c), y);
          tmem_wait_ld();
          if (bias) {
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              x[k] += __bfloat162float(bias[hh * D + c + k]);
              y[k] += __bfloat162float(bias[hh * D + D / 2 + c + k]);
            }
          }
          if (rope) {
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              const float cs = __ldg(rope + (c + k) * 2), sn = __ldg(rope + (c + k) * 2 + 1);
              const float a = x[k], e = y[k];
              x[k] = a * cs - e * sn;
              y[k] = e * cs + a * sn;
            }
          }
          if (valid) {
#pragma unroll
            for (int k = 0; k < 16; k += 4) {
              store4_bf16(dst + c + k, x[k], x[k + 1], x[k + 2], x[k + 3]);
              store4_bf16(dst + D / 2 + c + k, y[k], y[k + 1], y[k + 2], y[k + 3]);
            }
          }
        }
      }
      fence_before();
      mbar_arrive(&tempty[buf]);
    }
  }

  fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, 2 * HACC);
  if (threadIdx.x == 0 && abort_flag) set_status(J.status, kStatusTimeout);
}

int device_sms() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return n;
}

}  // namespace

size_t hidden_scratch_bytes(const HiddenJob& J) {
  const size_t hs = (size_t)J.L * J.B * J.Npad * J.DM * 2;
  const size_t rope = (size_t)J.B * (J.d / 2) * 2 * sizeof(float);
  return ((hs + 255) & ~size_t(255)) + ((rope + 255) & ~size_t(255));
}

cudaError_t launch_hidden_proxies(HiddenJob J, void* scratch, const void* W, int64_t w_layer_stride,
                                  cudaStream_t st) {
  if (reinterpret_cast<uintptr_t>(W) & 15) return cudaErrorMisalignedAddress;
  const size_t hs = (size_t)J.L * J.B * J.Npad * J.DM * 2;
  J.hs = static_cast<__nv_bfloat16*>(scratch);
  J.rope = J.rope_theta > 0.f
               ? reinterpret_cast<float*>(static_cast<unsigned char*>(scratch) + ((hs + 255) & ~size_t(255)))
               : nullptr;
  const int nq = J.DM / 8;
  dim3 g1((J.Npad * nq + 255) / 256, J.B, J.L);
  hidden_sample_kernel<<<g1, 256, 0, st>>>(J);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;

  CUtensorMap amap, wmap;
  if (!make_tmap_bf16_3d(&amap, J.hs, (uint64_t)J.DM, (uint64_t)J.Npad, (uint64_t)J.L * J.B,
                         (uint64_t)J.DM * 2, (uint64_t)J.Npad * J.DM * 2, HM))
    return cudaErrorInvalidValue;
  const uint64_t wls = w_layer_stride ? (uint64_t)w_layer_stride : (uint64_t)J.F * J.DM;
  if (!make_tmap_bf16_3d(&wmap, W, (uint64_t)J.DM, (uint64_t)J.F, (uint64_t)J.L,
                         (uint64_t)J.DM * 2, wls * 2, (uint32_t)J.NT))
    return cudaErrorInvalidValue;
  const int dyn = HSTAGE * stage_bytes(J.NT) + 1024;
  const int nsm = device_sms();
  if (nsm <= 0) return cudaErrorInvalidDevice;
  const int grid = std::max(1, std::min(nsm, J.tiles));
  if (J.d == 128) {
    if ((e = cudaFuncSetAttribute(hidden_proj_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  dyn)) != cudaSuccess) return e;
    hidden_proj_kernel<128><<<grid, HTHREADS, dyn, st>>>(amap, wmap, J);
  } else {
    if ((e = cudaFuncSetAttribute(hidden_proj_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  dyn)) != cudaSuccess) return e;
    hidden_proj_kernel<64><<<grid, HTHREADS, dyn, st>>>(amap, wmap, J);
  }
  return cudaGetLastError();
}

}  // namespace mmshift

// Tensor-core linear layer for many rows (batched decode, prefill): y = epi(norm?(x) . W^T) with
// tcgen05 (5th-generation tensor cores) on sm_103a.
//
// One CTA computes a 128-row x 64-column tile of y. Per 64-wide K block:
//   * the weight tile W[n0:n0+64, k:k+64] (bf16, K-major) arrives by a TMA tensor copy with the
//     128-byte swizzle, completing on an mbarrier;
//   * each of the 128 threads converts its own activation row x[m0+tid, k:k+64] (fp32, times the
//     RMSNorm gain) to bf16 and writes it into shared memory in the same swizzled K-major layout,
//     while accumulating the row's sum of squares;
//   * one thread issues four tcgen05.mma (M=128, N=64, K=16, bf16 -> fp32) into a TMEM
//     accumulator and commits them to a second mbarrier that frees the stage.
// The epilogue reads the accumulator with tcgen05.ld (thread = row), applies the row's inverse
// RMS and the layer's epilogue. TMEM is allocated only after the grid-dependency wait, so a kernel
// launched early never holds tensor memory its predecessor needs. Every wait is bounded.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstdio>

#include "common.cuh"
#include "epilogue.cuh"

namespace lca {

namespace {

constexpr int kUM = 128;     // rows per tile (UMMA M)
constexpr int kUN = 64;      // columns per tile (UMMA N)
constexpr int kUK = 64;      // K per stage (one 128-byte swizzle row of bf16)
constexpr int kUStages = 4;
constexpr int kUThreads = 128;
constexpr int kUSpins = 1 << 22;
constexpr uint32_t kATileBytes = kUM * kUK * 2;  // 16 KB
constexpr uint32_t kBTileBytes = kUN * kUK * 2;  // 8 KB

__device__ __forceinline__ uint32_t su32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void ubar_init(uint64_t* b, uint32_t n) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(b)), "r"(n) : "memory");
}
__device__ __forceinline__ void ubar_expect(uint64_t* b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(su32(b)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool ubar_try(uint64_t* b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(su32(b)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool ubar_wait(uint64_t* b, uint32_t parity) {
  for (int i = 0; i < kUSpins; ++i)
    if (ubar_try(b, parity)) return true;
  return false;
}

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFF) >> 4);  // start address
  d |= (uint64_t)1 << 16;                   // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)(1024 >> 4) << 32;         // stride byte offset between 8-row groups
  d |= (uint64_t)1 << 46;                   // descriptor version
  d |= (uint64_t)2 << 61;                   // 128-byte swizzle
  return d;
}

// Instruction descriptor: D fp32, A and B bf16, both K-major, M = 128, N = kUN.
constexpr uint32_t kIDesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kUN >> 3) << 17) |
                            ((uint32_t)(kUM >> 4) << 24);

__device__ __forceinline__ void umma(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(kIDesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(su32(bar))
               : "memory");
}
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(
          su32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(su32(bar)), "r"(x), "r"(y)
      : "memory");
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&h);
}

template <bool NORM>
__global__ void __launch_bounds__(kUThreads, 1)
k_umma(LinearArgs a, const __grid_constant__ CUtensorMap tmW, int num_mtiles) {
  TraceScope _trace(TT_GEMM);
  extern __shared__ __align__(1024) unsigned char usm_raw[];
  // 1024-byte aligned stages (128-byte swizzle atoms need it)
  unsigned char* usm =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(usm_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* As = usm;                                    // [stages][16 KB]
  unsigned char* Bs = usm + kUStages * kATileBytes;           // [stages][8 KB]
  uint64_t* full = reinterpret_cast<uint64_t*>(Bs + kUStages * kBTileBytes);  // [stages]
  uint64_t* done = full + kUStages;                                         // [stages]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + kUStages);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n0 = blockIdx.x * kUN;
  const int grp = blockIdx.z;
  const int rbase = grp * a.Mg_stride;
  const int nkb = a.Kd / kUK;

  if (tid == 0) {
    for (int s = 0; s < kUStages; ++s) {
      ubar_init(&full[s], 1);
      ubar_init(&done[s], 1);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmW)) : "memory");
  }
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)),
                 "r"(kUN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;

  int M = *a.M;
  M = M < a.M_cap ? M : a.M_cap;
  const int ntm = (M + kUM - 1) / kUM;
  bool failed = false;
  uint32_t it = 0;  // stage uses so far (mbarrier phases)

  for (int mt = blockIdx.y; mt < ntm && !failed; mt += num_mtiles) {
    const int m0 = mt * kUM;
    const int row = m0 + tid;
    const bool live = row < M;
    const float* xr = a.x + (size_t)(rbase + (live ? row : 0)) * a.ldx;
    float ss = 0.f;
    uint32_t last = 0;
    for (int kb = 0; kb < nkb; ++kb, ++it) {
      const int s = it % kUStages;
      if (it >= (uint32_t)kUStages && !failed) {  // the MMAs that last read this stage must be done
        if (!ubar_wait(&done[s], ((it / kUStages) - 1) & 1)) failed = true;
      }
      // activation row -> bf16, swizzled K-major
      unsigned char* at = As + (size_t)s * kATileBytes;
      const int k0 = kb * kUK;
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        float4 v0 = make_float4(0.f, 0.f, 0.f, 0.f), v1 = v0;
        if (live) {
          v0 = *reinterpret_cast<const float4*>(xr + k0 + c * 8);
          v1 = *reinterpret_cast<const float4*>(xr + k0 + c * 8 + 4);
        }
        if (NORM) {
          ss += v0.x * v0.x + v0.y * v0.y + v0.z * v0.z + v0.w * v0.w;
          ss += v1.x * v1.x + v1.y * v1.y + v1.z * v1.z + v1.w * v1.w;
          const float4 g0 = *reinterpret_cast<const float4*>(a.norm + k0 + c * 8);
          const float4 g1 = *reinterpret_cast<const float4*>(a.norm + k0 + c * 8 + 4);
          v0.x *= g0.x; v0.y *= g0.y; v0.z *= g0.z; v0.w *= g0.w;
          v1.x *= g1.x; v1.y *= g1.y; v1.z *= g1.z; v1.w *= g1.w;
        }
        uint4 u;
        u.x = pack_bf16(v0.x, v0.y);
        u.y = pack_bf16(v0.z, v0.w);
        u.z = pack_bf16(v1.x, v1.y);
        u.w = pack_bf16(v1.z, v1.w);
        const int r = tid;
        *reinterpret_cast<uint4*>(at + (r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) * 16)) = u;
      }
      if (tid == 0) {
        ubar_expect(&full[s], kBTileBytes);
        tma_load_2d(Bs + (size_t)s * kBTileBytes, &tmW, k0, grp * a.N + n0, &full[s]);
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncthreads();
      if (tid == 0 && !failed) {
        if (!ubar_wait(&full[s], (it / kUStages) & 1)) failed = true;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t abase = su32(As + (size_t)s * kATileBytes);
        const uint32_t bbase = su32(Bs + (size_t)s * kBTileBytes);
#pragma unroll
        for (int k = 0; k < kUK / 16; ++k)
          umma(tmem, sdesc(abase + k * 32), sdesc(bbase + k * 32), (kb > 0 || k > 0) ? 1u : 0u);
        umma_commit(&done[s]);
      }
      last = it;
    }
    // accumulator complete when the last commit has arrived
    if (!failed && !ubar_wait(&done[last % kUStages], (last / kUStages) & 1)) failed = true;
    if (__syncthreads_or(failed)) {
      failed = true;
      break;
    }
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const float inv = NORM ? rsqrtf(ss / (float)a.Kd + a.eps) : 1.f;
#pragma unroll
    for (int cb = 0; cb < kUN; cb += 32) {
      uint32_t v[32];
      const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)cb;
      asm volatile(
          "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
          "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
          : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
            "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]),
            "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]),
            "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]),
            "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
          : "r"(taddr));
      asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
      if (live) {
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
          const int col = n0 + cb + j;
          if (col < a.N) {
            const EpiPre p = epi_load(a.epi, rbase + row, col);
            epi_store<__nv_bfloat16>(a.epi, p, rbase + row, col, __uint_as_float(v[j]) * inv,
                                     __uint_as_float(v[j + 1]) * inv);
          }
        }
      }
    }
    // all threads finished reading TMEM before the next tile overwrites it
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  }
  if (failed && tid == 0) atomicOr(a.epi.err, kErrTimeout);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kUN) : "memory");
}

size_t umma_smem_bytes() { return (size_t)kUStages * (kATileBytes + kBTileBytes) + 2 * kUStages * 8 + 16 + 1024; }

}  // namespace

// Tensor map of a bf16 weight [rows][K] (K innermost) with 64 x 64 boxes and the 128-byte swizzle.
int make_weight_tmap(void* out, const void* W, long long rows, long long K) {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  if (!encode) {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return LCA_E_CUDA;
    encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  if (K % kUK || rows % kUN) return LCA_E_ARG;
  const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)K * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kUK, (cuuint32_t)kUN};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = encode(reinterpret_cast<CUtensorMap*>(out), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                            const_cast<void*>(W), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? LCA_OK : LCA_E_CUDA;
}

void kernel_attrs_umma() {
  cudaFuncSetAttribute(k_umma<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)umma_smem_bytes());
  cudaFuncSetAttribute(k_umma<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)umma_smem_bytes());
}

// Launch on the tensor cores when the layer fits the tile shapes; false otherwise.
bool linear_umma(const Dev& D, const LinearArgs& a, cudaStream_t s) {
  if (!a.tmap || D.dtype != LCA_BF16 || a.N % kUN || a.Kd % kUK) return false;
  const int mt_cap = (a.M_cap + kUM - 1) / kUM;
  const int rows_typ = a.rows_typ > 0 ? a.rows_typ : a.M_cap;
  int mtiles = (rows_typ + kUM - 1) / kUM;
  mtiles = mtiles < 1 ? 1 : (mtiles > mt_cap ? mt_cap : mtiles);
  // keep the grid within a few waves; extra row tiles are walked by the CTAs
  const int ncol = a.N / kUN;
  while (mtiles > 1 && (long long)mtiles * ncol * a.groups > 4LL * D.num_sms) mtiles = (mtiles + 1) / 2;
  CUtensorMap tm;
  memcpy(&tm, a.tmap, sizeof(tm));
  ++g_launches;
  if (a.norm)
    launch_pdl(k_umma<true>, dim3(ncol, mtiles, a.groups), dim3(kUThreads), umma_smem_bytes(), s, a, tm, mtiles);
  else
    launch_pdl(k_umma<false>, dim3(ncol, mtiles, a.groups), dim3(kUThreads), umma_smem_bytes(), s, a, tm, mtiles);
  return true;
}

LCA_TRACE_SETTER(trace_set_umma)

}  // namespace lca

using namespace lca;

extern "C" int lca_debug_gemm(const float* x, const void* W, float* y, int32_t M, int32_t N, int32_t K,
                              const int32_t* M_dev, int32_t* err_dev, void* stream) {
  if (!x || !W || !y || !M_dev || !err_dev || M < 1 || N < 1 || K < 1) return LCA_E_ARG;
  CUtensorMap tm;
  int st = make_weight_tmap(&tm, W, N, K);
  if (st != LCA_OK) return st;
  Dev D{};
  D.dtype = LCA_BF16;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  D.num_sms = sms;
  D.use_umma = 1;
  kernel_attrs_umma();
  int* err = err_dev;
  LinearArgs a{};
  a.x = x;
  a.ldx = K;
  a.W = W;
  a.N = N;
  a.Kd = K;
  a.groups = 1;
  a.M = M_dev;
  a.M_cap = M;
  a.rows_typ = M;
  a.tmap = &tm;
  a.epi.mode = EPI_STORE;
  a.epi.y = y;
  a.epi.ldy = N;
  a.epi.err = err;
  if (!linear_umma(D, a, reinterpret_cast<cudaStream_t>(stream))) return LCA_E_ARG;
  return cudaGetLastError() == cudaSuccess ? LCA_OK : LCA_E_CUDA;
}

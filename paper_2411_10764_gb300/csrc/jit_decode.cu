// Compiled feature program for decoded screening.
//
// ML^2Tuner's explorer (Sec. 2) enumerates the knob space; each candidate's
// features come from its knob values through the feature program (derived
// features after Table 5).  Inside the walk kernels the program is data,
// interpreted one operation at a time (about 67 instructions each).  For a
// large batch the library instead turns the program into CUDA C -- one
// straight-line statement per feature, the same rounded intrinsic per
// operation as the interpreter, constants as exact bit patterns -- compiles
// it once per program and device with NVRTC, and runs the result as a
// decode kernel that writes the batch's rows to a device buffer; the
// screening then stages those rows like caller-supplied features.  Every
// feature is bit-identical to the interpreter's.
//
// NVRTC and the driver entry points are resolved with dlopen at first use,
// so the library loads where neither exists; the decoded path then keeps the
// interpreter.  Host code only.
#include <dlfcn.h>

#include <cstdio>
#include <cstring>
#include <map>
#include <string>
#include <vector>

#include <cuda.h>
#include <nvrtc.h>

#include "mlt_internal.cuh"

namespace mlt {
namespace {

struct JitApi {
  bool tried = false;
  bool ok = false;
  std::string why;
  nvrtcResult (*create)(nvrtcProgram*, const char*, const char*, int, const char* const*, const char* const*);
  nvrtcResult (*compile)(nvrtcProgram, int, const char* const*);
  nvrtcResult (*log_size)(nvrtcProgram, size_t*);
  nvrtcResult (*log)(nvrtcProgram, char*);
  nvrtcResult (*cubin_size)(nvrtcProgram, size_t*);
  nvrtcResult (*cubin)(nvrtcProgram, char*);
  nvrtcResult (*destroy)(nvrtcProgram*);
  CUresult (*load)(CUmodule*, const void*);
  CUresult (*get_fn)(CUfunction*, CUmodule, const char*);
  CUresult (*set_attr)(CUfunction, CUfunction_attribute, int);
  CUresult (*launch)(CUfunction, unsigned, unsigned, unsigned, unsigned, unsigned, unsigned, unsigned, CUstream,
                     void**, void**);
};

JitApi g_api;

template <typename F>
bool sym(void* lib, const char* name, F* out) {
  *out = reinterpret_cast<F>(dlsym(lib, name));
  return *out != nullptr;
}

const JitApi& api() {
  if (g_api.tried) return g_api;
  g_api.tried = true;
  void* rtc = nullptr;
  for (const char* n : {"libnvrtc.so.13", "libnvrtc.so", "/usr/local/cuda/lib64/libnvrtc.so.13"})
    if ((rtc = dlopen(n, RTLD_NOW | RTLD_LOCAL)) != nullptr) break;
  void* drv = nullptr;
  for (const char* n : {"libcuda.so.1", "libcuda.so"})
    if ((drv = dlopen(n, RTLD_NOW | RTLD_LOCAL)) != nullptr) break;
  if (rtc == nullptr || drv == nullptr) {
    g_api.why = rtc == nullptr ? "NVRTC library not found" : "CUDA driver library not found";
    return g_api;
  }
  const bool ok = sym(rtc, "nvrtcCreateProgram", &g_api.create) && sym(rtc, "nvrtcCompileProgram", &g_api.compile) &&
                  sym(rtc, "nvrtcGetProgramLogSize", &g_api.log_size) && sym(rtc, "nvrtcGetProgramLog", &g_api.log) &&
                  sym(rtc, "nvrtcGetCUBINSize", &g_api.cubin_size) && sym(rtc, "nvrtcGetCUBIN", &g_api.cubin) &&
                  sym(rtc, "nvrtcDestroyProgram", &g_api.destroy) && sym(drv, "cuModuleLoadData", &g_api.load) &&
                  sym(drv, "cuModuleGetFunction", &g_api.get_fn) && sym(drv, "cuFuncSetAttribute", &g_api.set_attr) &&
                  sym(drv, "cuLaunchKernel", &g_api.launch);
  if (!ok) {
    g_api.why = "an NVRTC or driver entry point is missing";
    return g_api;
  }
  g_api.ok = true;
  return g_api;
}

std::string flt(float v) {
  uint32_t u;
  std::memcpy(&u, &v, 4);
  char b[48];
  std::snprintf(b, sizeof(b), "__uint_as_float(0x%08xu)", u);
  return b;
}

// Candidates per CTA of the decode kernel: its rows are transposed through
// shared memory (F x (TC + 1) floats) so that the row writes coalesce.
int decode_tile(int F) {
  for (int tc : {256, 128, 64, 32})
    if (static_cast<size_t>(F) * (tc + 1) * 4 <= 100 * 1024) return tc;
  return 32;
}

// CUDA C of the decode kernel for program d (digits and knob values as in
// knob_digits / decode_column; feature f as operation d.op[f] on its
// operands, with the same intrinsic).
std::string decode_source(const DecodeParams& d, int TC) {
  std::string s;
  s += "__device__ __forceinline__ float ilog2_exact(float a) {\n"
       "  const unsigned u = __float_as_uint(a);\n"
       "  const unsigned e = (u >> 23) & 0xFFu;\n"
       "  if ((u & 0x80000000u) || e == 0u || e == 0xFFu) return 0.0f;\n"
       "  return static_cast<float>(static_cast<int>(e) - 127);\n"
       "}\n";
  // the option values as bit patterns (a __device__ initializer must be a
  // constant expression)
  const int n_opts = d.opt_off[d.n_knobs - 1] + d.radix[d.n_knobs - 1];
  s += "__device__ const unsigned k_opts[" + std::to_string(std::max(1, n_opts)) + "] = {";
  for (int i = 0; i < n_opts; ++i) {
    uint32_t u;
    std::memcpy(&u, &d.opts[i], 4);
    char b[16];
    std::snprintf(b, sizeof(b), "0x%08xu", u);
    s += (i ? ", " : "") + std::string(b);
  }
  s += "};\n";
  const int F = d.F;
  s += "extern \"C\" __global__ void __launch_bounds__(" + std::to_string(TC) +
       ") mlt_jit_decode(long long first, const long long* __restrict__ list, long long n, float* __restrict__ out) {\n";
  s += "  extern __shared__ float col[];  // [F][TC + 1]\n";
  s += "  const int c = threadIdx.x;\n";
  s += "  const long long tile0 = static_cast<long long>(blockIdx.x) * " + std::to_string(TC) + ";\n";
  s += "  const long long i = tile0 + c;\n";
  s += "  if (i < n) {\n";
  s += "    unsigned long long r = static_cast<unsigned long long>(list ? list[i] : first + i);\n";
  for (int j = 0; j < d.n_knobs; ++j) {
    const std::string rj = std::to_string(d.radix[j]) + "ull";
    s += "    const float k" + std::to_string(j) + " = __uint_as_float(__ldg(&k_opts[" + std::to_string(d.opt_off[j]) +
         " + static_cast<int>(r % " + rj + ")]));\n";
    if (j + 1 < d.n_knobs) s += "    r /= " + rj + ";\n";
  }
  auto operand = [&](int src, float cf) -> std::string {
    if (src < 0) return flt(cf);
    if (src < d.n_knobs) return "k" + std::to_string(src);
    return "f" + std::to_string(src - d.n_knobs);
  };
  for (int f = 0; f < F; ++f) {
    const std::string A = operand(d.a[f], d.c[f]), B = operand(d.b[f], d.c[f]);
    std::string e;
    switch (d.op[f]) {
      case 0: e = A; break;
      case 1: e = "ilog2_exact(" + A + ")"; break;
      case 2: e = "__fadd_rn(" + A + ", " + B + ")"; break;
      case 3: e = "__fsub_rn(" + A + ", " + B + ")"; break;
      case 4: e = "__fmul_rn(" + A + ", " + B + ")"; break;
      case 5: e = "__fdiv_rn(" + A + ", " + B + ")"; break;
      case 6: e = "ceilf(__fdiv_rn(" + A + ", " + B + "))"; break;
      case 7: e = "__fsub_rn(" + A + ", __fmul_rn(" + B + ", floorf(__fdiv_rn(" + A + ", " + B + "))))"; break;
      case 8: e = "((" + B + ") < (" + A + ") ? (" + B + ") : (" + A + "))"; break;
      case 9: e = "((" + B + ") > (" + A + ") ? (" + B + ") : (" + A + "))"; break;
      case 10: e = "((" + A + ") > (" + B + ") ? 1.0f : 0.0f)"; break;
      default: e = "((" + A + ") == (" + B + ") ? 1.0f : 0.0f)"; break;
    }
    const std::string fs = std::to_string(f);
    s += "    const float f" + fs + " = " + e + ";\n";
    s += "    col[" + fs + " * " + std::to_string(TC + 1) + " + c] = f" + fs + ";\n";
  }
  s += "  }\n";
  s += "  __syncthreads();\n";
  s += "  const long long rows = n - tile0 < " + std::to_string(TC) + " ? n - tile0 : " + std::to_string(TC) + ";\n";
  s += "  float* dst = out + tile0 * " + std::to_string(F) + ";\n";
  s += "  for (int e = c; e < static_cast<int>(rows) * " + std::to_string(F) + "; e += " + std::to_string(TC) +
       ") {\n";
  s += "    const int row = e / " + std::to_string(F) + ", f = e - row * " + std::to_string(F) + ";\n";
  s += "    dst[e] = col[f * " + std::to_string(TC + 1) + " + row];\n";
  s += "  }\n";
  s += "}\n";
  return s;
}

uint64_t fnv(const void* p, size_t n, uint64_t h) {
  const unsigned char* b = static_cast<const unsigned char*>(p);
  for (size_t i = 0; i < n; ++i) h = (h ^ b[i]) * 1099511628211ull;
  return h;
}

// The program's identity: everything decode_source reads.
uint64_t program_key(const DecodeParams& d, int dev) {
  uint64_t h = 1469598103934665603ull;
  h = fnv(&dev, sizeof(dev), h);
  h = fnv(&d.n_knobs, sizeof(d.n_knobs), h);
  h = fnv(&d.F, sizeof(d.F), h);
  h = fnv(d.radix, sizeof(int) * d.n_knobs, h);
  h = fnv(d.opt_off, sizeof(int) * d.n_knobs, h);
  h = fnv(d.opts, sizeof(float) * (d.opt_off[d.n_knobs - 1] + d.radix[d.n_knobs - 1]), h);
  h = fnv(d.op, sizeof(int) * d.F, h);
  h = fnv(d.a, sizeof(int) * d.F, h);
  h = fnv(d.b, sizeof(int) * d.F, h);
  h = fnv(d.c, sizeof(float) * d.F, h);
  return h;
}

struct Entry {
  CUfunction fn = nullptr;
  int tc = 0;
  size_t smem = 0;
  std::string why;  // empty when fn is usable
};
std::map<uint64_t, Entry> g_cache;

}  // namespace

// Compiled decoder for program d on device dev (compiled on first use and
// cached; a failure is cached too, with its reason).
JitDecoder jit_decoder_for(const DecodeParams& d, int dev) {
  JitDecoder out{};
  const uint64_t key = program_key(d, dev);
  auto it = g_cache.find(key);
  if (it == g_cache.end()) {
    Entry e;
    const JitApi& a = api();
    if (!a.ok) {
      e.why = a.why;
    } else {
      e.tc = decode_tile(d.F);
      e.smem = static_cast<size_t>(d.F) * (e.tc + 1) * 4;
      const std::string src = decode_source(d, e.tc);
      int major = 0, minor = 0;
      cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
      const std::string arch = "-arch=sm_" + std::to_string(major * 10 + minor) + "a";
      const char* opts[] = {arch.c_str(), "-default-device", "--fmad=false", "-std=c++17"};
      nvrtcProgram prog = nullptr;
      nvrtcResult r = a.create(&prog, src.c_str(), "mlt_jit_decode.cu", 0, nullptr, nullptr);
      if (r == NVRTC_SUCCESS) r = a.compile(prog, 4, opts);
      if (r != NVRTC_SUCCESS) {
        size_t ls = 0;
        if (prog) a.log_size(prog, &ls);
        std::string log(ls, '\0');
        if (ls) a.log(prog, &log[0]);
        e.why = "NVRTC compile failed: " + log.substr(0, 400);
      } else {
        size_t cs = 0;
        a.cubin_size(prog, &cs);
        std::vector<char> cubin(cs);
        a.cubin(prog, cubin.data());
        CUmodule mod = nullptr;
        CUfunction fn = nullptr;
        if (a.load(&mod, cubin.data()) != CUDA_SUCCESS || a.get_fn(&fn, mod, "mlt_jit_decode") != CUDA_SUCCESS ||
            a.set_attr(fn, CU_FUNC_ATTRIBUTE_MAX_DYNAMIC_SHARED_SIZE_BYTES, static_cast<int>(e.smem)) != CUDA_SUCCESS)
          e.why = "loading the compiled decoder failed";
        else
          e.fn = fn;
      }
      if (prog) a.destroy(&prog);
    }
    it = g_cache.emplace(key, e).first;
  }
  out.fn = it->second.fn;
  out.tc = it->second.tc;
  out.smem = it->second.smem;
  out.why = it->second.why.c_str();
  return out;
}

bool jit_available() { return api().ok; }

cudaError_t launch_jit_decode(const JitDecoder& jd, const DecodeParams& d, long long n, float* out,
                              cudaStream_t st) {
  if (jd.fn == nullptr) return cudaErrorInvalidValue;
  if (n <= 0) return cudaSuccess;
  long long first = d.first_index;
  const long long* list = d.index_list;
  void* args[] = {&first, &list, &n, &out};
  const unsigned grid = static_cast<unsigned>((n + jd.tc - 1) / jd.tc);
  const CUresult r = api().launch(static_cast<CUfunction>(jd.fn), grid, 1, 1, static_cast<unsigned>(jd.tc), 1, 1,
                                  static_cast<unsigned>(jd.smem), reinterpret_cast<CUstream>(st), args, nullptr);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorLaunchFailure;
}

}  // namespace mlt

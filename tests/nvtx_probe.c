/*
 * tests/nvtx_probe.c -- a minimal NVTX injection library for the tests.
 *
 * NVTX (header-only, compiled into libtreepo) looks for a tool library named
 * by the environment variable NVTX_INJECTION64_PATH at its first call and,
 * if one is there, hands it the table of NVTX entry points. This library
 * takes over nvtxRangePushA and nvtxRangePop and records them as text lines
 * ("push <name>" / "pop") that the test reads back through probe_log().
 */
#include <nvtx3/nvToolsExt.h>
#include <string.h>

static char g_log[1 << 16];
static size_t g_len = 0;
static int g_depth = 0;

static void record(const char* a, const char* b) {
    size_t la = strlen(a), lb = b ? strlen(b) : 0;
    if (g_len + la + lb + 3 >= sizeof g_log) return;
    memcpy(g_log + g_len, a, la);
    g_len += la;
    if (b) {
        g_log[g_len++] = ' ';
        memcpy(g_log + g_len, b, lb);
        g_len += lb;
    }
    g_log[g_len++] = '\n';
    g_log[g_len] = 0;
}

static int probe_push(const char* message) {
    record("push", message);
    return g_depth++;
}

static int probe_pop(void) {
    record("pop", 0);
    return --g_depth;
}

const char* probe_log(void) { return g_log; }

int InitializeInjectionNvtx2(NvtxGetExportTableFunc_t get_table) {
    const NvtxExportTableCallbacks* cb = (const NvtxExportTableCallbacks*)get_table(NVTX_ETID_CALLBACKS);
    NvtxFunctionTable table = 0;
    unsigned int size = 0;
    if (!cb || !cb->GetModuleFunctionTable(NVTX_CB_MODULE_CORE, &table, &size)) return 0;
    if (size <= NVTX_CBID_CORE_RangePop) return 0;
    *table[NVTX_CBID_CORE_RangePushA] = (NvtxFunctionPointer)probe_push;
    *table[NVTX_CBID_CORE_RangePop] = (NvtxFunctionPointer)probe_pop;
    return 1;
}

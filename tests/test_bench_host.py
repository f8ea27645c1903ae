"""bench.py host logic that needs no GPU."""
import bench


def test_traffic_record_key_covers_the_lut_kernel():
    """The DRAM-traffic record is keyed to gemv_lut_kernel's own source: its section of gemv.cu,
    its launcher and the device helpers (bench.lut_kernel_source)."""
    src = bench.lut_kernel_source()
    assert "gemv_lut_kernel(const __grid_constant__ LutLayers L" in src
    assert "aq_status run_lut_layers(const Dims* ds" in src
    assert "// ---- device helpers" in src
    assert "gemv_lut4_kernel" not in src and "gemv_direct_kernel" not in src
